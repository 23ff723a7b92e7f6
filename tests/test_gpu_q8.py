"""int8 weights with fp16 row scales (the paper's matched-protocol kernel, Sec. 3.1):
y_i = s_i * sum_j W_ij x_j with fp16 x, through the resident (TMA) and map endpoints,
against the oracle's gemv_q8."""
import numpy as np
import pytest

import oracle
from paper_2608_12114_gb300 import build, pipeline, synth, wt

pytestmark = pytest.mark.gpu
TOL = 2e-3

# vectors per row V = K / 16: warp rows (V <= 64, lane groups of 1..16 and 32, 1..2 vectors
# per lane), block rows (64 < V <= 512, 1..2 vectors per thread), split-K (V > 512), and
# K % 16 != 0 (fallback)
SHAPES = [(9, 16), (33, 48), (100, 512), (13, 960), (40, 2048), (17, 2064), (11, 4096), (7, 7168), (5, 12288),
          (3, 16384), (6, 16400), (2, 65536), (4, 24), (0, 32), (3, 0)]


@pytest.fixture(scope="module")
def torch():
    import torch
    assert torch.cuda.is_available()
    build.build()
    wt.lib()
    return torch


@pytest.fixture(params=["default", "cuda", "q8rows"], autouse=True)
def onecol_kernel(request, monkeypatch):
    """Every test runs three times: with the default routing (rows up to K = 8192 on a
    tensor-core kernel at T = 1: the warp-MMA kernel for launches this small, longer rows on the
    CUDA-core kernel's split-K), with every int8 row on the CUDA-core kernel
    (WT_I8_ONECOL=cuda), and with the tensor-core rows on the row-owner kernel
    (WT_COLS_KERNEL=q8rows, the kernel full-size launches take), so every kernel's tile
    modes stay covered."""
    monkeypatch.delenv("WT_I8_ONECOL", raising=False)
    monkeypatch.delenv("WT_COLS_KERNEL", raising=False)
    if request.param == "cuda":
        monkeypatch.setenv("WT_I8_ONECOL", "cuda")
    elif request.param == "q8rows":
        monkeypatch.setenv("WT_COLS_KERNEL", "q8rows")
    return request.param


def check(h, dev, co, ys, ks):
    for k in ks:
        m = dev.mats[k]
        M, K = m.shape
        t, sc = h.tensors[m.parts[0]], h.tensors[m.scale]
        yhat, a = oracle.gemv_q8(co.blob_of(t.file, t.name), co.blob_of(sc.file, sc.name), M, K,
                                 synth.make_x(K, synth.DT_I8))
        err = oracle.gemv_error(ys[k].cpu().numpy(), yhat, a)
        assert err <= TOL, (m.name, m.shape, err)


def test_int8_resident_and_mapped_match_oracle(torch, tmp_path):
    ck = synth.write_files(synth.custom_q8(str(tmp_path), SHAPES))
    co = oracle.CheckpointOracle(ck.paths)
    with wt.Handle(ck.paths) as h:
        mats = pipeline.matrices(h)
        dev = pipeline.DeviceCheckpoint.allocate(h, mats)
        ks = dev.gemv_mats()
        assert len(ks) == len(SHAPES) and all(mats[k].scale is not None for k in ks)
        xs, ys = dev.inputs(), dev.outputs()
        for y in ys.values():
            y.fill_(float("nan"))
        s = torch.cuda.Stream()
        torch.cuda.synchronize()
        ev = dev.adopt(h, wt.WT_ADOPT_GATHER, s.cuda_stream)
        h.pass_(dev.descs(xs, ys, ev), s.cuda_stream)           # resident, event-gated
        s.synchronize()
        check(h, dev, co, ys, ks)
        first = {k: y.clone() for k, y in ys.items()}
        h.pass_(dev.descs(xs, ys), s.cuda_stream)               # resident, one launch
        s.synchronize()
        assert all(torch.equal(first[k], ys[k]) for k in ks)
        ym = {k: torch.full_like(ys[k], float("nan")) for k in ks}
        torch.cuda.synchronize()
        mapped = []
        for k in ks:
            m = mats[k]
            t = h.tensors[m.parts[0]]
            mapped.append(wt.gemv_desc(t.host_ptr, wt.WT_I8, m.shape[0], m.shape[1],
                                       xs[(m.shape[1], m.dtype)].data_ptr(), ym[k].data_ptr(),
                                       scale=dev.dst[m.scale]))
        h.pass_(mapped, s.cuda_stream)                          # map endpoint
        s.synchronize()
        check(h, dev, co, ym, ks)
        assert h.device_status() == 0


def test_int8_one_hot_is_the_rounded_scaled_column(torch, tmp_path):
    shapes = [(40, 48), (64, 2048), (9, 7168), (5, 20000)]
    ck = synth.write_files(synth.custom_q8(str(tmp_path), shapes, name="oh8"))
    co = oracle.CheckpointOracle(ck.paths)
    with wt.Handle(ck.paths) as h:
        mats = pipeline.matrices(h)
        dev = pipeline.DeviceCheckpoint.allocate(h, mats)
        torch.cuda.synchronize()
        dev.adopt(h, wt.WT_ADOPT_GATHER, 0)
        torch.cuda.synchronize()
        for k, (M, K) in zip(dev.gemv_mats(), shapes):
            m = mats[k]
            Wn = co.blob_of(0, m.name).view(np.int8).reshape(M, K)
            sn = co.blob_of(0, m.name + ".scale").view(np.float16)
            for j in (0, K // 2 + 5, K - 1):
                x = torch.zeros(K, dtype=torch.float16, device="cuda")
                x[j] = 1.0
                y = torch.empty(M, dtype=torch.float32, device="cuda")
                h.pass_([wt.gemv_desc(dev.bufs[k].data_ptr(), wt.WT_I8, M, K, x.data_ptr(), y.data_ptr(),
                                      scale=dev.dst[m.scale])], 0)
                want = sn.astype(np.float32) * Wn[:, j].astype(np.float32)
                assert np.array_equal(y.cpu().numpy(), want)


def test_int8_descriptor_rules(torch, tmp_path):
    ck = synth.write_files(synth.custom_q8(str(tmp_path), [(8, 64)], name="r8"))
    with wt.Handle(ck.paths) as h:
        x = torch.zeros(64, dtype=torch.float16, device="cuda")
        y = torch.zeros(8, dtype=torch.float32, device="cuda")
        W = torch.zeros(8 * 64, dtype=torch.uint8, device="cuda")
        with pytest.raises(wt.WtError) as ei:  # int8 without scales
            h.pass_([wt.gemv_desc(W.data_ptr(), wt.WT_I8, 8, 64, x.data_ptr(), y.data_ptr())], 0)
        assert ei.value.code == wt.WT_EINVAL
        with pytest.raises(wt.WtError) as ei:  # scales on a bf16 matrix
            h.pass_([wt.gemv_desc(W.data_ptr(), wt.WT_BF16, 8, 32, x.data_ptr(), y.data_ptr(),
                                  scale=x.data_ptr())], 0)
        assert ei.value.code == wt.WT_EINVAL


def test_int8_structured_rows(torch):
    """Rows that stress the int8 -> f16 decode: all zero (y must be exactly 0), sparse +-1,
    all -128, all 127, alternating extremes and uniform bytes, in every tile mode."""
    rng = np.random.default_rng(21)
    for K in (48, 2048, 7168, 20000):
        M = 30
        W = np.zeros((M, K), np.int8)
        for r in range(M):
            kind = r % 6
            if kind == 1:
                W[r, rng.choice(K, 8, replace=False)] = rng.choice([-1, 1], 8)
            elif kind == 2:
                W[r] = -128
            elif kind == 3:
                W[r] = 127
            elif kind == 4:
                W[r, 0::2], W[r, 1::2] = 127, -128
            elif kind == 5:
                W[r] = rng.integers(-128, 128, K)
        s = rng.uniform(0.001, 0.02, M).astype(np.float16)
        x = synth.make_x(K, synth.DT_I8)
        Wd = torch.from_numpy(W.view(np.uint8).reshape(-1).copy()).cuda()
        sd = torch.from_numpy(s.view(np.uint8).copy()).cuda()
        xd = torch.from_numpy(x.copy()).cuda()
        y = torch.full((M,), float("nan"), dtype=torch.float32, device="cuda")
        with wt.Handle([]) as h:  # a handle without files: W is plain device memory
            h.pass_([wt.gemv_desc(Wd.data_ptr(), wt.WT_I8, M, K, xd.data_ptr(), y.data_ptr(),
                                  scale=sd.data_ptr())], 0)
            torch.cuda.synchronize()
            assert h.device_status() == 0
        got = y.cpu().numpy()
        yhat, a = oracle.gemv_q8(W.view(np.uint8).reshape(-1), s.view(np.uint8), M, K, x)
        assert np.all(got[0::6] == 0.0), K
        assert oracle.gemv_error(got, yhat, a) <= TOL, K
