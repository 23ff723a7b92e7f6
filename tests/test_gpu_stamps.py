"""WT_OPEN_STAMPS: the stamping instantiation of the one-column resident kernel gives the same
results as the plain one (bit for bit, and within tolerance of the oracle), and its per-CTA
record is complete and ordered: entry <= prologue <= operands <= exit, and prologue <= first
copy <= first stage <= last stage <= exit for every CTA with rows, on one launch issued from the host and on the
latest replay of a captured graph of programmatically launched passes."""
import numpy as np
import pytest

import oracle
from paper_2608_12114_gb300 import build, synth, wt

pytestmark = pytest.mark.gpu
TOL = 2e-3
F = {f: i for i, f in enumerate(wt.STAMP_FIELDS)}


@pytest.fixture(scope="module")
def torch():
    import torch
    assert torch.cuda.is_available()
    build.build()
    wt.lib()
    return torch


def mats(torch, rng, specs):
    """[(W, x, y, s, dtype, M, K)] on the device, with host copies for the oracle."""
    out = []
    for dtype, M, K in specs:
        if dtype == wt.WT_I8:
            Wh = rng.integers(-128, 128, M * K).astype(np.int8).view(np.uint8)
            sh = rng.uniform(0.001, 0.02, M).astype(np.float16).view(np.uint8)
            xh = rng.standard_normal(K).astype(np.float16).view(np.uint8)
        else:
            w = (0.02 * rng.standard_normal(M * K)).astype(np.float32)
            Wh = (synth.f32_to_bf16_bits(w) if dtype == wt.WT_BF16 else w).view(np.uint8).reshape(-1).copy()
            sh = None
            xh = synth.make_x(K, dtype).view(np.uint8)
        W = torch.from_numpy(Wh).cuda()
        x = torch.from_numpy(xh.copy()).cuda()
        s = torch.from_numpy(sh.copy()).cuda() if sh is not None else None
        y = torch.full((M,), float("nan"), dtype=torch.float32, device="cuda")
        out.append(dict(W=W, x=x, y=y, s=s, dtype=dtype, M=M, K=K, Wh=Wh, xh=xh, sh=sh))
    return out


def descs(ms):
    return [wt.gemv_desc(m["W"].data_ptr(), m["dtype"], m["M"], m["K"], m["x"].data_ptr(), m["y"].data_ptr(),
                         scale=m["s"].data_ptr() if m["s"] is not None else 0) for m in ms]


def check_oracle(ms):
    for m in ms:
        y = m["y"].cpu().numpy()
        if m["dtype"] == wt.WT_I8:
            yhat, a = oracle.gemv_q8(m["Wh"], m["sh"], m["M"], m["K"], m["xh"])
        else:
            yhat, a = oracle.gemv(m["Wh"], m["dtype"], m["M"], m["K"], m["xh"])
        assert oracle.gemv_error(y, yhat, a) <= TOL, (m["dtype"], m["M"], m["K"])


def check_record(st, num_sms):
    assert st.ndim == 2 and st.shape[1] == len(wt.STAMP_FIELDS) and st.shape[0] >= 1
    t = st.astype(np.int64)
    assert np.all(t[:, F["entry"]] > 0) and np.all(t[:, F["exit"]] > 0)
    assert np.all(t[:, F["sm"]] < num_sms)
    busy = t[:, F["first_copy"]] > 0
    assert busy.any()
    # a CTA with no rows issues no copy and sees no stage
    assert np.all(t[~busy, F["first_full"]] == 0) and np.all(t[~busy, F["last_full"]] == 0)
    order = ["entry", "prologue", "operands"]
    for a, b in zip(order, order[1:] + ["exit"]):
        assert np.all(t[:, F[a]] <= t[:, F[b]]), (a, b)
    # the first copy is issued by another thread than the one that stamps "operands", both
    # after the same wait, so the two are not ordered against each other
    chain = ["prologue", "first_copy", "first_full", "last_full", "exit"]
    for a, b in zip(chain, chain[1:]):
        assert np.all(t[busy, F[a]] <= t[busy, F[b]]), (a, b)
    # one launch: every CTA lived within one second of the first entry
    assert t[:, F["exit"]].max() - t[:, F["entry"]].min() < 1_000_000_000


CASES = {
    "bf16_16MiB": [(wt.WT_BF16, 4096, 2048)],
    "bf16_ragged": [(wt.WT_BF16, 300, 4096), (wt.WT_BF16, 77, 1032)],
    "f32": [(wt.WT_F32, 777, 1024)],
    # int8 rows up to 8 KB go to the tensor-core kernels; longer ones are split into column
    # segments on the one-column kernel (stamped) and summed by the reduction pass
    "int8_split_k": [(wt.WT_I8, 96, 16384)],
    "many_pieces": [(wt.WT_BF16, 64, 512)] * 40,
}


@pytest.mark.parametrize("case", sorted(CASES))
def test_stamped_pass_matches_plain_and_records_every_cta(torch, case):
    rng = np.random.default_rng(11)
    ms = mats(torch, rng, CASES[case])
    d = descs(ms)
    s = torch.cuda.Stream()
    num_sms = torch.cuda.get_device_properties(0).multi_processor_count
    with wt.Handle([]) as h:
        h.pass_(d, s.cuda_stream)
        s.synchronize()
        ref = [m["y"].clone() for m in ms]
        check_oracle(ms)
        assert h.device_status() == 0
    with wt.Handle([], wt.WT_OPEN_STAMPS) as hs:
        assert hs.pass_stamps().shape[0] == 0  # nothing stamped yet
        for m in ms:
            m["y"].fill_(float("nan"))
        n0 = hs.kernel_launches()
        hs.pass_(d, s.cuda_stream)
        s.synchronize()
        assert hs.kernel_launches() > n0
        for m, r in zip(ms, ref):
            assert torch.equal(m["y"], r)
        st = hs.pass_stamps()
        check_record(st, num_sms)
        assert hs.device_status() == 0


def test_stamps_of_a_replayed_graph_of_programmatic_passes(torch):
    rng = np.random.default_rng(12)
    ms = mats(torch, rng, CASES["bf16_16MiB"])
    d = descs(ms)
    s = torch.cuda.Stream()
    num_sms = torch.cuda.get_device_properties(0).multi_processor_count
    with wt.Handle([], wt.WT_OPEN_STAMPS) as h:
        h.pass_(d, s.cuda_stream)  # outside the capture: plan resident, stamp buffer allocated
        s.synchronize()
        ref = ms[0]["y"].clone()
        before = h.pass_stamps()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            for _ in range(3):  # consecutive passes: programmatic edges between them
                h.pass_(d, torch.cuda.current_stream().cuda_stream)
        ms[0]["y"].fill_(float("nan"))
        torch.cuda.synchronize()
        for _ in range(4):
            g.replay()
        torch.cuda.synchronize()
        assert torch.equal(ms[0]["y"], ref)
        st = h.pass_stamps()
        check_record(st, num_sms)
        assert st.shape == before.shape
        # the record is the latest replay's, not the launch before the capture
        assert st[:, F["entry"]].astype(np.int64).min() > before[:, F["exit"]].astype(np.int64).max()
        assert h.device_status() == 0
        del g
