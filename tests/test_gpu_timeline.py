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
