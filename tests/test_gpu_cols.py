"""Multi-column GEMV (cols = T in 1..16; the paper's multi-column packed-int8 kernel and its
T-sweep, Sec. 4.3): Y[t] = diag(s) W X[t] on the tensor cores, against the oracle's
gemv_cols on every output, max |Y - Yhat| / A <= 2e-3."""
import numpy as np
import pytest

import oracle
from paper_2608_12114_gb300 import build, synth, wt

pytestmark = pytest.mark.gpu
TOL = 2e-3
BF16, F16, I8 = wt.WT_BF16, wt.WT_F16, wt.WT_I8

# (dtype, M, K): ragged row counts around the 16-row tile and 64-row super block; K from one
# 4-vector group to many uneven chunks; K not a multiple of 16 bytes -> generic fallback
SHAPES = [(I8, 1, 16), (I8, 15, 64), (I8, 16, 1536), (I8, 17, 1552), (I8, 65, 7168), (I8, 130, 20000),
          (I8, 33, 24), (BF16, 1, 8), (BF16, 63, 768), (BF16, 64, 4096), (BF16, 100, 776), (BF16, 7, 12),
          (F16, 40, 2048), (F16, 9, 136)]
TS = [1, 2, 3, 7, 8, 9, 15, 16]


@pytest.fixture(scope="module")
def torch():
    import torch
    assert torch.cuda.is_available()
    build.build()
    wt.lib()
    return torch


@pytest.fixture(params=["default", "mma", "umma", "q8rows"], autouse=True)
def cols_kernel(request, monkeypatch):
    """Every test runs under each routing of the multi-column kernels: the default (int8 with
    T > 8 on the row-owner kernel, 2-byte weights with T > 8 on tcgen05, the rest on the
    warp-MMA kernel), everything on the warp-MMA kernel (WT_COLS_KERNEL=mma), 2-byte weights
    on tcgen05 at every T (=umma), and int8 on the row-owner kernel at every T (=q8rows)."""
    if request.param == "default":
        monkeypatch.delenv("WT_COLS_KERNEL", raising=False)
    else:
        monkeypatch.setenv("WT_COLS_KERNEL", request.param)
    return request.param


def make(torch, rng, dtype, M, K, T):
    """Host bytes and device copies of W, X (and s for int8)."""
    if dtype == I8:
        W = rng.integers(-128, 128, (M, K)).astype(np.int8).view(np.uint8)
        s = rng.uniform(0.001, 0.02, M).astype(np.float16).view(np.uint8)
        X = rng.standard_normal((T, K)).astype(np.float16).view(np.uint8)
    elif dtype == BF16:
        W = synth.f32_to_bf16_bits((0.02 * rng.standard_normal((M, K))).astype(np.float32)).view(np.uint8)
        X = synth.f32_to_bf16_bits(rng.standard_normal((T, K)).astype(np.float32)).view(np.uint8)
        s = None
    else:
        W = (0.02 * rng.standard_normal((M, K))).astype(np.float16).view(np.uint8)
        X = rng.standard_normal((T, K)).astype(np.float16).view(np.uint8)
        s = None
    dev = lambda a: None if a is None else torch.from_numpy(np.ascontiguousarray(a).reshape(-1)).cuda()  # noqa: E731
    return dict(dtype=dtype, M=M, K=K, T=T, W=W, X=X, s=s, Wd=dev(W), Xd=dev(X), sd=dev(s),
                Y=torch.full((T * max(M, 1),), float("nan"), dtype=torch.float32, device="cuda"))


def desc(c, y=None):
    return wt.gemv_desc(c["Wd"].data_ptr(), c["dtype"], c["M"], c["K"], c["Xd"].data_ptr(),
                        (y if y is not None else c["Y"]).data_ptr(),
                        scale=c["sd"].data_ptr() if c["sd"] is not None else 0, cols=c["T"])


def check(c, Y):
    Yhat, A = oracle.gemv_cols(c["W"].reshape(-1), c["dtype"], c["M"], c["K"], c["X"].reshape(-1), c["T"],
                               scale=None if c["s"] is None else c["s"])
    got = Y[:c["T"] * c["M"]].cpu().numpy().astype(np.float64).reshape(c["T"], c["M"])
    err = oracle.gemv_error(got.reshape(-1), Yhat.reshape(-1), A.reshape(-1))
    assert err <= TOL, (c["dtype"], c["M"], c["K"], c["T"], err)
    return err


@pytest.mark.parametrize("T", TS)
def test_cols_against_oracle_and_grouping(torch, T):
    rng = np.random.default_rng(100 + T)
    cases = [make(torch, rng, d, M, K, T) for d, M, K in SHAPES]
    with wt.Handle([]) as h:
        h.pass_([desc(c) for c in cases], 0)          # every matrix in one group
        torch.cuda.synchronize()
        assert h.device_status() == 0
        for c in cases:
            check(c, c["Y"])
        for c in cases:                                # one matrix per call: same bits
            y2 = torch.full_like(c["Y"], float("nan"))
            h.pass_([desc(c, y2)], 0)
            torch.cuda.synchronize()
            assert torch.equal(y2[:T * c["M"]], c["Y"][:T * c["M"]]), (c["dtype"], c["M"], c["K"])


def test_cols_one_hot_columns_are_exact(torch):
    """X[t] = e_{k_t}: Y[t] = s * W[:, k_t] rounded once (products of integers and ones are
    exact on the tensor cores)."""
    rng = np.random.default_rng(7)
    for M, K in ((70, 7168), (17, 1552), (33, 64)):
        T = 16
        W = rng.integers(-128, 128, (M, K)).astype(np.int8)
        s = rng.uniform(0.001, 0.02, M).astype(np.float16)
        ks = rng.choice(K, T, replace=False)
        X = np.zeros((T, K), np.float16)
        X[np.arange(T), ks] = 1.0
        Wd = torch.from_numpy(W.view(np.uint8).reshape(-1).copy()).cuda()
        sd = torch.from_numpy(s.view(np.uint8).copy()).cuda()
        Xd = torch.from_numpy(X.view(np.uint8).reshape(-1).copy()).cuda()
        Y = torch.empty(T * M, dtype=torch.float32, device="cuda")
        with wt.Handle([]) as h:
            h.pass_([wt.gemv_desc(Wd.data_ptr(), I8, M, K, Xd.data_ptr(), Y.data_ptr(), scale=sd.data_ptr(),
                                  cols=T)], 0)
            torch.cuda.synchronize()
        want = (s.astype(np.float32)[None, :] * W[:, ks].T.astype(np.float32))
        assert np.array_equal(Y.cpu().numpy().reshape(T, M), want)


def test_cols_zero_rows_and_zero_k(torch):
    rng = np.random.default_rng(8)
    M, K, T = 40, 3072, 5
    W = rng.integers(-128, 128, (M, K)).astype(np.int8)
    W[::3] = 0
    s = rng.uniform(0.001, 0.02, M).astype(np.float16)
    X = rng.standard_normal((T, K)).astype(np.float16)
    Wd = torch.from_numpy(W.view(np.uint8).reshape(-1).copy()).cuda()
    sd = torch.from_numpy(s.view(np.uint8).copy()).cuda()
    Xd = torch.from_numpy(X.view(np.uint8).reshape(-1).copy()).cuda()
    Y = torch.full((T * M,), float("nan"), dtype=torch.float32, device="cuda")
    Y0 = torch.full((T * M,), float("nan"), dtype=torch.float32, device="cuda")
    with wt.Handle([]) as h:
        h.pass_([wt.gemv_desc(Wd.data_ptr(), I8, M, K, Xd.data_ptr(), Y.data_ptr(), scale=sd.data_ptr(), cols=T),
                 wt.gemv_desc(Wd.data_ptr(), I8, M, 0, Xd.data_ptr(), Y0.data_ptr(), scale=sd.data_ptr(), cols=T)],
                0)
        torch.cuda.synchronize()
    got = Y.cpu().numpy().reshape(T, M)
    assert np.all(got[:, ::3] == 0.0)
    Yhat, A = oracle.gemv_cols(W.view(np.uint8), 3, M, K, X.view(np.uint8), T, scale=s.view(np.uint8))
    assert oracle.gemv_error(got.reshape(-1), Yhat.reshape(-1), A.reshape(-1)) <= TOL
    assert torch.count_nonzero(Y0) == 0


def test_cols_descriptor_rules(torch):
    x = torch.zeros(64 * 17, dtype=torch.float16, device="cuda")
    y = torch.zeros(8 * 17, dtype=torch.float32, device="cuda")
    W = torch.zeros(8 * 64 * 4, dtype=torch.uint8, device="cuda")
    with wt.Handle([]) as h:
        for bad in (-1, 17):
            with pytest.raises(wt.WtError) as ei:
                h.pass_([wt.gemv_desc(W.data_ptr(), BF16, 8, 64, x.data_ptr(), y.data_ptr(), cols=bad)], 0)
            assert ei.value.code == wt.WT_EINVAL
        with pytest.raises(wt.WtError) as ei:
            h.pass_([wt.gemv_desc(W.data_ptr(), wt.WT_F32, 8, 64, x.data_ptr(), y.data_ptr(), cols=2)], 0)
        assert ei.value.code == wt.WT_ENOTSUP


def test_cols_map_endpoint_reads_in_place(torch, tmp_path):
    """W inside the handle's mapping with cols > 0 (plain loads through the host page tables)."""
    shapes = [(33, 2048), (9, 7168)]
    ck = synth.write_files(synth.custom_q8(str(tmp_path), shapes, name="mc8"))
    co = oracle.CheckpointOracle(ck.paths)
    T = 6
    with wt.Handle(ck.paths) as h:
        for i, (M, K) in enumerate(shapes):
            t = h.tensors[h.find("w%d" % i)]
            sc = h.tensors[h.find("w%d.scale" % i)]
            s = co.blob_of(sc.file, sc.name)
            sd = torch.from_numpy(s.copy()).cuda()
            X = np.random.default_rng(M).standard_normal((T, K)).astype(np.float16)
            Xd = torch.from_numpy(X.view(np.uint8).reshape(-1).copy()).cuda()
            Y = torch.full((T * M,), float("nan"), dtype=torch.float32, device="cuda")
            h.pass_([wt.gemv_desc(t.host_ptr, I8, M, K, Xd.data_ptr(), Y.data_ptr(), scale=sd.data_ptr(),
                                  cols=T)], 0)
            torch.cuda.synchronize()
            Yhat, A = oracle.gemv_cols(co.blob_of(t.file, t.name), 3, M, K, X.view(np.uint8), T, scale=s)
            assert oracle.gemv_error(Y.cpu().numpy().astype(np.float64), Yhat.reshape(-1), A.reshape(-1)) <= TOL
        assert h.device_status() == 0


def test_cols_mixed_column_counts_and_dtypes_in_one_pass(torch):
    """One wt_pass whose matrices ask for different T (one- and two-tile MMA paths in the same
    launch) and different dtypes (separate launches of one group)."""
    rng = np.random.default_rng(9)
    spec = [(I8, 40, 1536, 3), (I8, 70, 4096, 12), (BF16, 33, 2048, 16), (I8, 17, 7168, 1), (BF16, 50, 768, 9),
            (F16, 20, 512, 8)]
    cases = [make(torch, rng, d, M, K, T) for d, M, K, T in spec]
    with wt.Handle([]) as h:
        h.pass_([desc(c) for c in cases], 0)
        torch.cuda.synchronize()
        assert h.device_status() == 0
    for c in cases:
        check(c, c["Y"])


def test_cols_full_size_matched_protocol(torch, tmp_path, cols_kernel):
    """The T-sweep's launch configuration at full size: 12 matrices of 12288 x 7168 int8 with
    fp16 row scales in one pass, T = 8 and 16; every output against the oracle (its functions
    run unchanged on blocks of rows, in threads), Y NaN-filled first."""
    from concurrent.futures import ThreadPoolExecutor
    from paper_2608_12114_gb300 import pipeline
    if cols_kernel != "default":
        pytest.skip("full size runs the default routing; the small cases cover the forced ones")
    pool = ThreadPoolExecutor(16)
    ck = synth.build("protocol_q8", str(tmp_path), workers=16)
    co = oracle.CheckpointOracle(ck.paths)
    try:
        with wt.Handle(ck.paths) as h:
            dev = pipeline.DeviceCheckpoint.allocate(h, pipeline.matrices(h))
            torch.cuda.synchronize()
            dev.adopt(h, wt.WT_ADOPT_GATHER, 0)
            torch.cuda.synchronize()
            ks = dev.gemv_mats()
            for T in (8, 16):
                X = np.random.default_rng(T).standard_normal((T, 7168)).astype(np.float16)
                Xd = torch.from_numpy(X.view(np.uint8).reshape(-1).copy()).cuda()
                ys = {k: torch.full((T * 12288,), float("nan"), dtype=torch.float32, device="cuda") for k in ks}
                d = dev.descs({(7168, wt.WT_I8): Xd}, ys)
                d["cols"] = T
                h.pass_(d, 0)
                torch.cuda.synchronize()
                assert h.device_status() == 0
                for k in ks:
                    m = dev.mats[k]
                    t, sc = h.tensors[m.parts[0]], h.tensors[m.scale]
                    W, S = co.blob_of(t.file, t.name), co.blob_of(sc.file, sc.name)
                    blocks = [(r, min(12288, r + 1024)) for r in range(0, 12288, 1024)]
                    parts = list(pool.map(lambda b: oracle.gemv_cols(W[b[0] * 7168:b[1] * 7168], 3, b[1] - b[0], 7168,
                                                                     X.view(np.uint8), T, scale=S[2 * b[0]:2 * b[1]]),
                                          blocks))
                    Yhat = np.concatenate([p[0] for p in parts], axis=1)
                    A = np.concatenate([p[1] for p in parts], axis=1)
                    got = ys[k].cpu().numpy().reshape(T, 12288)
                    assert oracle.gemv_error(got.reshape(-1), Yhat.reshape(-1), A.reshape(-1)) <= TOL, (T, m.name)
    finally:
        co.close()


def test_cols_map_endpoint_bf16_and_f16(torch, tmp_path):
    """The map endpoint with T columns for 2-byte weights (mapped multi-column kernel)."""
    for dtype, name in ((synth.DT_BF16, "mb"), (synth.DT_F16, "mh")):
        shapes = [(70, 4096), (5, 40), (33, 1032)]
        ck = synth.write_files(synth.custom(str(tmp_path / name), shapes, dtype=dtype, name=name))
        co = oracle.CheckpointOracle(ck.paths)
        T = 11
        with wt.Handle(ck.paths) as h:
            for i, (M, K) in enumerate(shapes):
                t = h.tensors[i]
                rng = np.random.default_rng(i)
                if dtype == synth.DT_BF16:
                    X = synth.f32_to_bf16_bits(rng.standard_normal((T, K)).astype(np.float32)).view(np.uint8)
                else:
                    X = rng.standard_normal((T, K)).astype(np.float16).view(np.uint8)
                Xd = torch.from_numpy(X.reshape(-1).copy()).cuda()
                Y = torch.full((T * M,), float("nan"), dtype=torch.float32, device="cuda")
                h.pass_([wt.gemv_desc(t.host_ptr, dtype, M, K, Xd.data_ptr(), Y.data_ptr(), cols=T)], 0)
                torch.cuda.synchronize()
                Yhat, A = oracle.gemv_cols(co.blob_of(t.file, t.name), dtype, M, K, X.reshape(-1), T)
                assert oracle.gemv_error(Y.cpu().numpy().astype(np.float64), Yhat.reshape(-1), A.reshape(-1)) <= TOL
            assert h.device_status() == 0
        co.close()
