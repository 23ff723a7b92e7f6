"""The first-use timeline (WT_OPEN_TIMELINE, wt_trace) on the GPU: contract C3 as data.

Checked on a small decoder: one record per ingest batch and per GEMV group; each record's end
is not before its begin; batches run in order on the ingest stream; every GEMV group begins
only after the batch it waited on has landed (the event order the contract requires) and
ends with correct results.  Also: the REGISTER route reports which registration it holds."""
import numpy as np
import pytest

import oracle
from paper_2608_12114_gb300 import build, pipeline, synth, wt

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch():
    import torch
    assert torch.cuda.is_available()
    build.build()
    wt.lib()
    return torch


def test_timeline_orders_each_group_after_its_batch(torch, tmp_path):
    ck = synth.build("mid", str(tmp_path), layers=2, vocab=8192, workers=4)
    ingest_s, consume_s = torch.cuda.Stream(), torch.cuda.Stream()
    with wt.Handle(ck.paths, wt.WT_OPEN_TIMELINE) as h:
        dev = pipeline.DeviceCheckpoint.allocate(h, pipeline.matrices(h))
        xs, ys = dev.inputs(), dev.outputs()
        for y in ys.values():
            y.fill_(float("nan"))
        torch.cuda.synchronize()
        origin = torch.cuda.Event(enable_timing=True)
        origin.record(ingest_s)
        ev = dev.adopt(h, wt.WT_ADOPT_GATHER, ingest_s.cuda_stream)
        descs = dev.descs(xs, ys, ev)
        h.pass_(descs, consume_s.cuda_stream)
        consume_s.synchronize()
        recs = h.trace(origin.cuda_event)
        assert h.trace(origin.cuda_event) == []  # records are consumed
        ing = [r for r in recs if r["kind"] == "ingest"]
        gem = [r for r in recs if r["kind"] == "gemv"]
        waits = [int(w) for w in descs["wait_event"]]
        groups = [w for n, w in enumerate(waits) if n == 0 or waits[n - 1] != w]
        assert len(gem) == len(groups)
        assert [g["event"] for g in gem] == groups
        assert set(ev.values()) <= {r["event"] for r in ing}  # every ready event is a batch's
        assert [r["index"] for r in ing] == list(range(len(ing)))
        assert sum(r["bytes"] for r in ing) == ck.data_bytes
        assert sum(r["bytes"] for r in gem) == dev.weight_bytes
        for r in recs:
            assert 0.0 <= r["begin_ms"] <= r["end_ms"], r
        for a, b in zip(ing, ing[1:]):
            assert b["begin_ms"] >= a["end_ms"] - 1e-3  # one stream: batches in order
        landed = {r["event"]: r["end_ms"] for r in ing}
        for g in gem:
            assert g["begin_ms"] >= landed[g["event"]] - 1e-3, g
        co = oracle.CheckpointOracle(ck.paths)
        try:
            for k in dev.gemv_mats():
                m = dev.mats[k]
                t = h.tensors[m.parts[0]]
                yhat, a = oracle.gemv(co.blob_of(t.file, t.name), m.dtype, m.shape[0], m.shape[1],
                                      synth.make_x(m.shape[1], m.dtype))
                assert oracle.gemv_error(ys[k].cpu().numpy(), yhat, a) <= 2e-3
        finally:
            co.close()


def test_register_route_reports_its_registration(torch, tmp_path):
    ck = synth.build("tiny", str(tmp_path))
    with wt.Handle(ck.paths, wt.WT_ROUTE_REGISTER) as h:
        flags = h.registration(0)
        assert flags & 0x02  # cudaHostRegisterMapped
        assert flags & ~0x0A == 0  # and at most cudaHostRegisterReadOnly besides
    with wt.Handle(ck.paths, wt.WT_ROUTE_DIRECT) as h:
        assert h.registration(0) == 0


def test_interleaved_wait_events_make_one_group_each(torch):
    """Descriptors whose wait events interleave (A, B, none, A, B, none, ...) form one group per
    distinct event, in order of first appearance: three GEMV records in the timeline, and the
    same results, bit for bit, as one pass with no events; a later call with fresh events in
    the same pattern reuses the plan."""
    rng = np.random.default_rng(5)
    K = 1024
    Ws, ys, descs = [], [], []
    x = torch.from_numpy(synth.make_x(K, wt.WT_BF16)).cuda()
    for i in range(12):
        M = 64 + 37 * i
        W = torch.from_numpy(synth.f32_to_bf16_bits((0.02 * rng.standard_normal(M * K)).astype(np.float32))
                             .view(np.uint8)).cuda()
        y = torch.full((M,), float("nan"), dtype=torch.float32, device="cuda")
        Ws.append(W)
        ys.append(y)
        descs.append(wt.gemv_desc(W.data_ptr(), wt.WT_BF16, M, K, x.data_ptr(), y.data_ptr()))
    s = torch.cuda.Stream()
    with wt.Handle([]) as h0:
        h0.pass_(descs, s.cuda_stream)
        s.synchronize()
    ref = [y.clone() for y in ys]
    other = torch.cuda.Stream()
    with wt.Handle([], wt.WT_OPEN_TIMELINE) as h:
        for rep in range(2):
            a, b = torch.cuda.Event(), torch.cuda.Event()
            a.record(other)
            b.record(other)
            pattern = [a.cuda_event, b.cuda_event, 0]
            d = [wt.gemv_desc(q.W, q.dtype, q.M, q.K, q.x, q.y, wait_event=pattern[i % 3])
                 for i, q in enumerate(descs)]
            for y in ys:
                y.fill_(float("nan"))
            origin = torch.cuda.Event(enable_timing=True)
            origin.record(s)
            n0 = h.kernel_launches()
            h.pass_(d, s.cuda_stream)
            s.synchronize()
            recs = [r for r in h.trace(origin.cuda_event) if r["kind"] == "gemv"]
            assert len(recs) == 3
            assert [r["event"] for r in recs] == pattern[:2] + [0]
            assert h.kernel_launches() - n0 == 3
            for y, r in zip(ys, ref):
                assert torch.equal(y, r)
        assert h.device_status() == 0
