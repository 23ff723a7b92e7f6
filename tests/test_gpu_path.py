"""GPU parity: the CUDA path, called through the C ABI, against the CPU oracle.

Bytes must match bit for bit (full compare and both FNV digests); every GEMV row
must satisfy |y - yhat| / sum_j |W_ij x_j| <= 2e-3 (the tolerance the benchmark spec fixes
for fp32-accumulated bf16 GEMV; fp64 oracle)."""
import numpy as np
import pytest

import oracle
from paper_2608_12114_gb300 import build, pipeline, synth, wt

pytestmark = pytest.mark.gpu
TOL = 2e-3
CANARY = 64


@pytest.fixture(scope="module")
def torch():
    import torch
    assert torch.cuda.is_available()
    build.build()
    wt.lib()
    torch.cuda.init()
    return torch


def ingest(torch, ck, mode=wt.WT_ADOPT_GATHER, flags=0, stream=None, slab=True):
    h = wt.Handle(ck.paths, flags)
    mats = pipeline.matrices(h)
    dev = pipeline.DeviceCheckpoint.allocate(h, mats, canary=CANARY, slab=slab)
    for b in dev.bufs:
        b.fill_(0xA5)
    torch.cuda.synchronize()
    s = stream or torch.cuda.Stream()
    ev = dev.adopt(h, mode, s.cuda_stream)
    return h, dev, ev, s


def check_bytes(torch, h, dev, co):
    """Full compare of every tensor against the oracle's file bytes, and canaries intact."""
    for m, b in zip(dev.mats, dev.bufs):
        got = b.cpu().numpy()
        want = np.concatenate([co.files[h.tensors[i].file].blob(
            [e["name"] for e in co.files[h.tensors[i].file].entries].index(h.tensors[i].name)) for i in m.parts]) \
            if m.parts else np.zeros(0, np.uint8)
        n = want.size
        assert np.array_equal(got[:n], want), m.name
        assert np.all(got[n:n + CANARY] == 0xA5), "canary overwritten after " + m.name


def device_digests(torch, h, dev, plain=False):
    """D_tree (or D_plain) of every tensor, on the device, per tensor index."""
    idx = sorted(dev.dst)
    out = torch.zeros(len(idx), dtype=torch.int64, device="cuda")
    h.checksum([dev.dst[i] for i in idx], [h.tensors[i].nbytes for i in idx], out.data_ptr(), 0, plain=plain)
    return {i: int(v) & 0xFFFFFFFFFFFFFFFF for i, v in zip(idx, out.cpu().tolist())}


def oracle_digests(h, co):
    d = {}
    for i, t in enumerate(h.tensors):
        fo = co.files[t.file]
        e = [x["name"] for x in fo.entries].index(t.name)
        d[i] = (oracle.fnv1a64(fo.blob(e)), oracle.fnv_tree(fo.blob(e)))
    return d


def check_gemv(h, dev, co, ys, rows=None):
    worst = 0.0
    for k in dev.gemv_mats():
        m = dev.mats[k]
        M, K = m.shape
        W = co.matrix_bytes([(h.tensors[i].file, h.tensors[i].name) for i in m.parts])
        x = synth.make_x(K, m.dtype)
        y = ys[k].cpu().numpy().astype(np.float64)
        r = None if rows is None else \
            sorted(set([0, M - 1] + [int(v) for v in np.random.default_rng(k).integers(0, M, rows)]))
        if m.scale is not None:  # int8 weights with fp16 row scales
            t = h.tensors[m.scale]
            yhat, a = oracle.gemv_q8(W, co.blob_of(t.file, t.name), M, K, x, rows=r)
        elif r is None:
            yhat, a = oracle.gemv(W, m.dtype, M, K, x)
        else:
            yhat, a = oracle.gemv_rows(W, m.dtype, M, K, x, r)
        err = oracle.gemv_error(y if r is None else y[r], yhat, a)
        assert err <= TOL, (m.name, err)
        worst = max(worst, err)
    return worst


# ----------------------------------------------------------------------------- ingest

@pytest.mark.parametrize("mode", [wt.WT_ADOPT_GATHER, wt.WT_ADOPT_CE, wt.WT_ADOPT_STAGED])
def test_tiny_ingest_bit_exact_all_modes(torch, tmp_path, mode):
    ck = synth.build("tiny", str(tmp_path))
    co = oracle.CheckpointOracle(ck.paths)
    h, dev, ev, s = ingest(torch, ck, mode)
    s.synchronize()
    check_bytes(torch, h, dev, co)
    assert all(ev[i] for i in ev)
    od = oracle_digests(h, co)
    tree, plain = device_digests(torch, h, dev), device_digests(torch, h, dev, plain=True)
    for i in od:
        assert (plain[i], tree[i]) == od[i]
    h.close()


@pytest.mark.parametrize("flags", [wt.WT_ROUTE_DIRECT, wt.WT_ROUTE_REGISTER,
                                   wt.WT_ROUTE_DIRECT | wt.WT_OPEN_PREFAULT])
def test_routes_give_identical_bytes(torch, tmp_path, flags):
    ck = synth.build("mid", str(tmp_path), layers=1, vocab=500)
    co = oracle.CheckpointOracle(ck.paths)
    h, dev, ev, s = ingest(torch, ck, wt.WT_ADOPT_GATHER, flags)
    s.synchronize()
    assert h.route(0) == (flags & 3)
    check_bytes(torch, h, dev, co)
    h.close()


def test_route_none_needs_staged(torch, tmp_path):
    ck = synth.build("tiny", str(tmp_path))
    co = oracle.CheckpointOracle(ck.paths)
    with pytest.raises(wt.WtError) as ei:
        ingest(torch, ck, wt.WT_ADOPT_GATHER, wt.WT_ROUTE_NONE)
    assert ei.value.code == wt.WT_ENOTSUP
    h, dev, ev, s = ingest(torch, ck, wt.WT_ADOPT_STAGED, wt.WT_ROUTE_NONE)
    s.synchronize()
    check_bytes(torch, h, dev, co)
    h.close()


def test_many_halves_land_contiguously(torch, tmp_path):
    ck = synth.build("many", str(tmp_path), n_matrices=300, workers=4)
    co = oracle.CheckpointOracle(ck.paths)
    for mode in (wt.WT_ADOPT_GATHER, wt.WT_ADOPT_CE):
        h, dev, ev, s = ingest(torch, ck, mode, slab=False)
        s.synchronize()
        check_bytes(torch, h, dev, co)
        od = oracle_digests(h, co)
        tree = device_digests(torch, h, dev)
        assert all(tree[i] == od[i][1] for i in od)
        h.close()


def test_destination_inside_mapping_is_refused(torch, tmp_path):
    ck = synth.build("tiny", str(tmp_path))
    with wt.Handle(ck.paths) as h:
        with pytest.raises(wt.WtError) as ei:
            h.adopt([0], [h.tensors[1].host_ptr])
        assert ei.value.code == wt.WT_EINVAL


# ----------------------------------------------------------------------------- GEMV

SHAPES = [(1, 8), (3, 16), (7, 24), (33, 40), (100, 256), (65, 264), (17, 2048), (9, 2056),
          (5, 4096), (3, 16384), (10, 16392), (4, 100000), (300, 512), (2, 7), (6, 0), (0, 64)]


@pytest.mark.parametrize("dtype", [synth.DT_BF16, synth.DT_F16, synth.DT_F32])
def test_gemv_shapes_against_oracle(torch, tmp_path, dtype):
    shapes = SHAPES
    ck = synth.write_files(synth.custom(str(tmp_path), shapes, dtype=dtype, name="c%d" % dtype))
    co = oracle.CheckpointOracle(ck.paths)
    h, dev, ev, s = ingest(torch, ck)
    xs, ys = dev.inputs(), dev.outputs()
    for y in ys.values():
        y.fill_(float("nan"))
    torch.cuda.synchronize()
    h.pass_(dev.descs(xs, ys, ev), s.cuda_stream)
    s.synchronize()
    check_gemv(h, dev, co, ys)
    assert h.device_status() == 0
    h.close()


def test_one_hot_x_returns_exact_columns(torch, tmp_path):
    shapes = [(40, 24), (64, 1024), (9, 2056), (5, 20000)]
    ck = synth.write_files(synth.custom(str(tmp_path), shapes, dtype=synth.DT_BF16, name="oh"))
    co = oracle.CheckpointOracle(ck.paths)
    h, dev, ev, s = ingest(torch, ck)
    s.synchronize()
    for k, (M, K) in zip(dev.gemv_mats(), shapes):
        for j in (0, K // 2 + 3, K - 1):
            x = torch.zeros(K, dtype=torch.bfloat16, device="cuda")
            x[j] = 1.0
            y = torch.empty(M, dtype=torch.float32, device="cuda")
            h.pass_([wt.gemv_desc(dev.bufs[k].data_ptr(), wt.WT_BF16, M, K, x.data_ptr(), y.data_ptr())], 0)
            W = co.files[0].blob(k).view("<u2").reshape(M, K)[:, j].astype(np.uint32) << 16
            assert np.array_equal(y.cpu().numpy().view(np.uint32), W.astype(np.uint32))
    h.close()


def test_grouping_does_not_change_results(torch, tmp_path):
    ck = synth.build("mid", str(tmp_path), layers=2, vocab=3000)
    h, dev, ev, s = ingest(torch, ck)
    xs = dev.inputs()
    ya, yb = dev.outputs(), dev.outputs()
    torch.cuda.synchronize()
    h.pass_(dev.descs(xs, ya, ev), s.cuda_stream)               # grouped by ingest batch
    for k in dev.gemv_mats():                                     # one matrix per call
        h.pass_(dev.descs(xs, yb, None, only=[k]), s.cuda_stream)
    yc = dev.outputs()
    torch.cuda.synchronize()
    h.pass_(dev.descs(xs, yc), s.cuda_stream)                     # all in one resident launch
    s.synchronize()
    for k in dev.gemv_mats():
        assert torch.equal(ya[k], yb[k]) and torch.equal(ya[k], yc[k])
    h.close()


def test_first_use_pipeline_mid(torch, tmp_path):
    """Ingest on one stream, consume on another gated only by per-batch events."""
    ck = synth.build("mid", str(tmp_path), layers=3, workers=4)
    co = oracle.CheckpointOracle(ck.paths)
    ingest_s, consume_s = torch.cuda.Stream(), torch.cuda.Stream()
    h = wt.Handle(ck.paths)
    dev = pipeline.DeviceCheckpoint.allocate(h, pipeline.matrices(h))
    xs, ys = dev.inputs(), dev.outputs()
    torch.cuda.synchronize()
    ev = dev.adopt(h, wt.WT_ADOPT_GATHER, ingest_s.cuda_stream)
    h.pass_(dev.descs(xs, ys, ev), consume_s.cuda_stream)  # no host wait between the two
    consume_s.synchronize()
    check_gemv(h, dev, co, ys)
    yr = dev.outputs()
    torch.cuda.synchronize()
    h.pass_(dev.descs(xs, yr), consume_s.cuda_stream)
    consume_s.synchronize()
    for k in dev.gemv_mats():
        assert torch.equal(ys[k], yr[k])
    h.close()


@pytest.mark.parametrize("workload", ["tiny", "many", "protocol_q8"])
def test_first_use_with_io_region(torch, tmp_path, workload):
    """The timed first use: slabs allocated segment by segment with the step's inputs and
    outputs in the first one (x copied from a pinned host buffer, y NaN-filled first), every
    GEMV gated on its batch's event; every row against the oracle, the weight bytes exact."""
    kw = {"many": {"n_matrices": 40}, "protocol_q8": {"matrices": 2, "rows": 2048}}.get(workload, {})
    ck = synth.build(workload, str(tmp_path), **kw)
    co = oracle.CheckpointOracle(ck.paths)
    ingest_s, consume_s = torch.cuda.Stream(), torch.cuda.Stream()
    h = wt.Handle(ck.paths)
    mats = pipeline.matrices(h)
    x_host = pipeline.host_inputs(mats)
    dev, ev, _ = pipeline.DeviceCheckpoint.stream_in(h, mats, wt.WT_ADOPT_GATHER, ingest_s.cuda_stream, io=True)
    ys = dev.io_outputs()
    with torch.cuda.stream(consume_s):
        ys.buf.fill_(float("nan"))
        dev.io_x().copy_(x_host, non_blocking=True)
        h.pass_(dev.descs(dev.io_inputs(), ys, ev), consume_s.cuda_stream)
    consume_s.synchronize()
    _, y_off, rows, total = pipeline.io_layout(mats)
    assert dev.io.numel() >= total and ys.buf.numel() == max(1, sum(rows))
    assert dev.io.data_ptr() % 256 == 0 and all(p % 256 == 0 for p in dev.ptrs)
    check_gemv(h, dev, co, ys)
    check_bytes(torch, h, dev, co)
    h.close()


# ----------------------------------------------------------------------------- checksums

def test_checksum_edges(torch):
    rng = np.random.default_rng(7)
    data = rng.integers(0, 256, 40 * 4096 + 100, dtype=np.uint8)
    buf = torch.from_numpy(data).cuda()
    # empty, sub-vector, unaligned starts (bytewise staging), ragged last leaves, and
    # buffers of more leaves than the combine kernel loads ahead (16)
    cases = [(0, 0), (0, 1), (1, 15), (3, 4095), (0, 4096), (0, 4097), (5, 8192 + 17), (16, 3 * 4096 + 84),
             (0, 37 * 4096 + 5), (7, 20 * 4096), (32, 17 * 4096)]
    base = buf.data_ptr()
    for plain in (False, True):
        with wt.Handle([]) as h:
            out = torch.zeros(len(cases), dtype=torch.int64, device="cuda")
            h.checksum([base + o for o, n in cases], [n for o, n in cases], out.data_ptr(), 0, plain=plain)
            got = [int(v) & (2 ** 64 - 1) for v in out.cpu().tolist()]
        fn = oracle.fnv1a64 if plain else oracle.fnv_tree
        assert got == [fn(data[o:o + n]) for o, n in cases]


def test_checksum_many_buffers(torch):
    """More buffers than one launch carries (the host splits them into batches)."""
    n = 600
    rng = np.random.default_rng(8)
    sizes = rng.integers(0, 9000, n)
    data = rng.integers(0, 256, int(sizes.sum()) + 64, dtype=np.uint8)
    buf = torch.from_numpy(data).cuda()
    offs = np.concatenate([[0], np.cumsum(sizes)[:-1]])
    with wt.Handle([]) as h:
        out = torch.zeros(n, dtype=torch.int64, device="cuda")
        h.checksum([buf.data_ptr() + int(o) for o in offs], [int(s) for s in sizes], out.data_ptr(), 0)
        got = [int(v) & (2 ** 64 - 1) for v in out.cpu().tolist()]
    assert got == [oracle.fnv_tree(data[o:o + s]) for o, s in zip(offs, sizes)]


def test_checksum_chunked_second_level(torch):
    """Buffers above 4096 leaves combine their leaf digests in parallel chunks of 512; the
    digest must equal the oracle's serial chain: 4096 leaves (serial), 4097 (eight full
    chunks and one of one digest), a ragged unaligned 40 MiB buffer, and zero-chunk buffers
    between chunked ones in one batch; through wt_checksum and wt_checksum_noalloc."""
    rng = np.random.default_rng(9)
    data = rng.integers(0, 256, 100 << 20, dtype=np.uint8)
    buf = torch.from_numpy(data).cuda()
    cases = [(0, 4096 * 4096), (64, 4096 * 4096 + 1), (3, (40 << 20) + 777), (5, 100),
             (4096, 4096 * (4096 + 512) - 5), (0, 0), (17, 9000), (1 << 20, 4096 * 8192)]
    want = [oracle.fnv_tree(data[o:o + n]) for o, n in cases]
    base = buf.data_ptr()
    for noalloc in (False, True):
        out = torch.zeros(len(cases), dtype=torch.int64, device="cuda")
        if noalloc:
            wt.checksum_noalloc([base + o for o, n in cases], [n for o, n in cases], out.data_ptr(), 0)
        else:
            with wt.Handle([]) as h:
                h.checksum([base + o for o, n in cases], [n for o, n in cases], out.data_ptr(), 0)
        torch.cuda.synchronize()
        got = [int(v) & (2 ** 64 - 1) for v in out.cpu().tolist()]
        assert got == want, noalloc


def test_unaligned_operands_take_the_generic_kernel(torch):
    """W and x 2 bytes past a 16-byte boundary (element-aligned only): the scalar fallback,
    checked against the oracle; one and several columns."""
    rng = np.random.default_rng(13)
    M, K, T = 37, 1000, 3
    Wb = synth.f32_to_bf16_bits((0.02 * rng.standard_normal(M * K)).astype(np.float32)).view(np.uint8)
    X = synth.f32_to_bf16_bits(rng.standard_normal(T * K).astype(np.float32)).view(np.uint8)
    Wd = torch.zeros(Wb.size + 16, dtype=torch.uint8, device="cuda")
    Wd[2:2 + Wb.size] = torch.from_numpy(Wb.copy()).cuda()
    Xd = torch.zeros(X.size + 16, dtype=torch.uint8, device="cuda")
    Xd[2:2 + X.size] = torch.from_numpy(X.copy()).cuda()
    y1 = torch.full((M,), float("nan"), dtype=torch.float32, device="cuda")
    yT = torch.full((T * M,), float("nan"), dtype=torch.float32, device="cuda")
    with wt.Handle([]) as h:
        h.pass_([wt.gemv_desc(Wd.data_ptr() + 2, wt.WT_BF16, M, K, Xd.data_ptr() + 2, y1.data_ptr()),
                 wt.gemv_desc(Wd.data_ptr() + 2, wt.WT_BF16, M, K, Xd.data_ptr() + 2, yT.data_ptr(), cols=T)], 0)
        torch.cuda.synchronize()
        assert h.device_status() == 0
    Y, A = oracle.gemv_cols(Wb, wt.WT_BF16, M, K, X, T)
    assert oracle.gemv_error(y1.cpu().numpy(), Y[0], A[0]) <= 2e-3
    assert oracle.gemv_error(yT.cpu().numpy(), Y.reshape(-1), A.reshape(-1)) <= 2e-3


def test_descriptor_bounds_are_refused_before_any_launch(torch):
    x = torch.zeros(64, dtype=torch.bfloat16, device="cuda")
    y = torch.zeros(64, dtype=torch.float32, device="cuda")
    with wt.Handle([]) as h:
        n0 = h.kernel_launches()
        for M, K in ((2 ** 31, 16), (16, 2 ** 31)):
            with pytest.raises(wt.WtError) as ei:
                h.pass_([wt.gemv_desc(x.data_ptr(), wt.WT_BF16, M, K, x.data_ptr(), y.data_ptr())], 0)
            assert ei.value.code == wt.WT_EINVAL
        with pytest.raises(wt.WtError) as ei:                       # u8 weights have no GEMV
            h.pass_([wt.gemv_desc(x.data_ptr(), wt.WT_U8, 4, 16, x.data_ptr(), y.data_ptr())], 0)
        assert ei.value.code == wt.WT_ENOTSUP
        with pytest.raises(wt.WtError) as ei:                       # null y with rows
            h.pass_([wt.gemv_desc(x.data_ptr(), wt.WT_BF16, 4, 16, x.data_ptr(), 0)], 0)
        assert ei.value.code == wt.WT_EINVAL
        assert h.kernel_launches() == n0 and h.device_status() == 0


def test_device_overruns_are_refused_on_the_host(torch, tmp_path):
    """A destination or operand that starts in a device allocation and runs past its end is
    refused before anything is enqueued (no out-of-bounds GPU access is ever attempted)."""
    ck = synth.write_files(synth.custom(str(tmp_path), [(1024, 8192)], name="big"))   # 16 MiB bf16
    small = torch.empty(1 << 20, dtype=torch.uint8, device="cuda")   # a 1 MiB block of a small segment
    with wt.Handle(ck.paths) as h:
        n0 = h.kernel_launches()
        with pytest.raises(wt.WtError) as ei:
            h.adopt([0], [small.data_ptr()], wt.WT_ADOPT_GATHER, 0)
        assert ei.value.code == wt.WT_EINVAL and "past the end" in str(ei.value)
        x = torch.zeros(8192, dtype=torch.bfloat16, device="cuda")
        y = torch.zeros(16, dtype=torch.float32, device="cuda")
        W = torch.zeros(1024 * 8192, dtype=torch.bfloat16, device="cuda")
        for M, K, Wp, yp in ((1 << 20, 8192, W.data_ptr(), y.data_ptr()),     # y far too short
                             (65536, 8192, small.data_ptr(), W.data_ptr())):  # W far too short
            with pytest.raises(wt.WtError) as ei:
                h.pass_([wt.gemv_desc(Wp, wt.WT_BF16, M, K, x.data_ptr(), yp)], 0)
            assert ei.value.code == wt.WT_EINVAL and "past the end" in str(ei.value)
        assert h.kernel_launches() == n0 and h.device_status() == 0
        big = torch.empty(16 << 20, dtype=torch.uint8, device="cuda")     # right size: accepted
        torch.cuda.synchronize()
        h.adopt([0], [big.data_ptr()], wt.WT_ADOPT_GATHER, 0)
        torch.cuda.synchronize()
        assert h.device_status() == 0


# ----------------------------------------------------------------------------- unmapped (pread) route

@pytest.mark.parametrize("workload,kw", [("many", dict(n_matrices=300)), ("mid", dict(layers=1, vocab=40000))],
                         ids=["many-300", "mid-1-layer"])
def test_nomap_staged_ingest_matches_oracle(torch, tmp_path, workload, kw):
    """WT_OPEN_NOMAP + STAGED: no file is mapped; host threads pread into the pinned ring and the
    gather kernel moves each slot.  Row blocks land contiguously, tensors larger than a 64 MiB
    slot (the 40000 x 2560 embedding, 205 MB) span slots; bytes and canaries bit-exact, digests
    and every GEMV row against the oracle, with the event-gated pass."""
    ck = synth.build(workload, str(tmp_path), workers=4, **kw)
    co = oracle.CheckpointOracle(ck.paths)
    h, dev, ev, s = ingest(torch, ck, wt.WT_ADOPT_STAGED, wt.WT_OPEN_NOMAP)
    assert not [l for l in open("/proc/self/maps") if str(tmp_path) in l]
    xs, ys = dev.inputs(), dev.outputs()
    for y in ys.values():
        y.fill_(float("nan"))
    c = torch.cuda.Stream()
    h.pass_(dev.descs(xs, ys, ev), c.cuda_stream)
    c.synchronize()
    s.synchronize()
    check_bytes(torch, h, dev, co)
    od = oracle_digests(h, co)
    tree = device_digests(torch, h, dev)
    assert all(tree[i] == od[i][1] for i in od)
    check_gemv(h, dev, co, ys)
    assert h.device_status() == 0
    h.close()


def test_nomap_refuses_device_routes_and_changed_files(torch, tmp_path):
    ck = synth.build("tiny", str(tmp_path))
    with pytest.raises(wt.WtError) as ei:  # no mapping, so no gather or copy-engine route
        ingest(torch, ck, wt.WT_ADOPT_GATHER, wt.WT_OPEN_NOMAP)
    assert ei.value.code == wt.WT_ENOTSUP
    h = wt.Handle(ck.paths, wt.WT_OPEN_NOMAP)
    dev = pipeline.DeviceCheckpoint.allocate(h, pipeline.matrices(h))
    # the path now names another file of the same size: the staged adopt refuses it
    p = ck.paths[0]
    data = open(p, "rb").read()
    open(p + ".new", "wb").write(data)
    import os
    os.replace(p + ".new", p)
    with pytest.raises(wt.WtError) as ei:
        dev.adopt(h, wt.WT_ADOPT_STAGED, 0)
    assert ei.value.code == wt.WT_EIO and "changed" in str(ei.value)
    h.close()
    # a fresh handle on the new file adopts it
    co = oracle.CheckpointOracle(ck.paths)
    h, dev, ev, s = ingest(torch, ck, wt.WT_ADOPT_STAGED, wt.WT_OPEN_NOMAP)
    s.synchronize()
    check_bytes(torch, h, dev, co)
    h.close()


# ----------------------------------------------------------------------------- mixed (WT_OPEN_MAP_LARGE)

@pytest.mark.parametrize("mode", [wt.WT_ADOPT_GATHER, wt.WT_ADOPT_CE, wt.WT_ADOPT_STAGED], ids=["gather", "ce", "staged"])
def test_map_large_mixed_ingest_matches_oracle(torch, tmp_path, monkeypatch, mode):
    """WT_OPEN_MAP_LARGE maps only the files at or above the threshold (here the median file
    size).  A GATHER or CE adopt moves the small files through the pinned ring on the library's
    own stream, concurrently with the mapped files; the caller's stream is ordered after both
    (digests taken on it with no host wait see every byte); bytes, canaries, digests and every
    GEMV row match the oracle with the event-gated pass on another stream."""
    ck = synth.build("many", str(tmp_path), workers=4, n_matrices=300)
    import os
    sizes = [os.path.getsize(p) for p in ck.paths]
    thr = sorted(sizes)[len(sizes) // 2]
    monkeypatch.setenv("WT_MAP_MIN_BYTES", str(thr))
    co = oracle.CheckpointOracle(ck.paths)
    h, dev, ev, s = ingest(torch, ck, mode, wt.WT_OPEN_MAP_LARGE)
    mapped = {l.split()[-1] for l in open("/proc/self/maps") if str(tmp_path) in l}
    assert len(mapped) == sum(n >= thr for n in sizes)
    assert all((h.route(f) == wt.WT_ROUTE_NONE) == (sizes[f] < thr) for f in range(len(sizes)))
    idx = sorted(dev.dst)
    out = torch.zeros(len(idx), dtype=torch.int64, device="cuda")
    h.checksum([dev.dst[i] for i in idx], [h.tensors[i].nbytes for i in idx], out.data_ptr(), s.cuda_stream)
    xs, ys = dev.inputs(), dev.outputs()
    for y in ys.values():
        y.fill_(float("nan"))
    c = torch.cuda.Stream()
    h.pass_(dev.descs(xs, ys, ev), c.cuda_stream)
    c.synchronize()
    s.synchronize()
    od = oracle_digests(h, co)
    got = {i: int(v) & 0xFFFFFFFFFFFFFFFF for i, v in zip(idx, out.cpu().tolist())}
    assert all(got[i] == od[i][1] for i in idx)
    check_bytes(torch, h, dev, co)
    check_gemv(h, dev, co, ys)
    assert h.device_status() == 0
    h.close()


def test_map_large_matrix_across_both_ways(torch, tmp_path, monkeypatch):
    """Matrices whose row blocks lie in a small (unmapped) and a large (mapped) file: the two
    blocks cross two streams, so the pipeline gives the matrix one event recorded after the
    wt_adopt call; every GEMV row matches the oracle with y NaN-filled first, for adopts issued
    at once and segment by segment (stream_in)."""
    T = []
    mats = []
    paths = []
    K = 512
    for m in range(12):
        small_rows, large_rows = 1 + 3 * m, 200 + 17 * m  # 1 KB .. 34 KB and 200 KB .. 391 KB blocks
        parts = []
        for b, rows in enumerate((small_rows, large_rows) if m % 2 == 0 else (large_rows, small_rows)):
            f = len(paths)
            parts.append(len(T))
            T.append(synth.TensorSpec(f"m{m}#r{b}", synth.DT_BF16, (rows, K), f, key=(5, 700 + f)))
            paths.append(str(tmp_path / f"x{f:03d}.wt"))
        mats.append(synth.Matrix(f"m{m}", synth.DT_BF16, small_rows + large_rows, K, parts))
    ck = synth.write_files(synth.Checkpoint("split", paths, T, mats))
    monkeypatch.setenv("WT_MAP_MIN_BYTES", str(100 << 10))
    co = oracle.CheckpointOracle(ck.paths)
    for how in ("adopt", "stream_in"):
        h = wt.Handle(ck.paths, wt.WT_OPEN_MAP_LARGE)
        hm = pipeline.matrices(h)
        assert all(len({h.tensors.host_ptrs[i] == 0 for i in m.parts}) == 2 for m in hm)
        s = torch.cuda.Stream()
        if how == "adopt":
            dev = pipeline.DeviceCheckpoint.allocate(h, hm)
            ev = dev.adopt(h, wt.WT_ADOPT_GATHER, s.cuda_stream)
        else:
            dev, ev, _ = pipeline.DeviceCheckpoint.stream_in(h, hm, wt.WT_ADOPT_GATHER, s.cuda_stream,
                                                             first_bytes=1 << 20, growth=1.0)
        assert dev._joined  # one joint event per adopt call that held such matrices
        for m in hm:
            assert len({ev[i] for i in m.parts}) == 1
        xs, ys = dev.inputs(), dev.outputs()
        for y in ys.values():
            y.fill_(float("nan"))
        c = torch.cuda.Stream()
        h.pass_(dev.descs(xs, ys, ev), c.cuda_stream)
        c.synchronize()
        s.synchronize()
        check_gemv(h, dev, co, ys)
        assert h.device_status() == 0
        h.close()


def test_map_large_staged_failure_is_reported_and_the_handle_recovers(torch, tmp_path, monkeypatch):
    """The fifth pread of the staged half fails (WT_FAULT, made on the host) while the mapped
    half is being enqueued: wt_adopt returns WT_EIO with the file named, the caller's stream is
    still ordered after every copy the call issued, the pinned ring is free again, and the next
    adopt on the same handle moves every byte (and leaves every canary) correctly."""
    ck = synth.build("many", str(tmp_path), workers=4, n_matrices=120)
    import os
    sizes = [os.path.getsize(p) for p in ck.paths]
    monkeypatch.setenv("WT_MAP_MIN_BYTES", str(sorted(sizes)[len(sizes) // 2]))
    co = oracle.CheckpointOracle(ck.paths)
    h = wt.Handle(ck.paths, wt.WT_OPEN_MAP_LARGE)
    dev = pipeline.DeviceCheckpoint.allocate(h, pipeline.matrices(h), canary=CANARY)
    for b in dev.bufs:
        b.fill_(0xA5)
    torch.cuda.synchronize()
    s = torch.cuda.Stream()
    monkeypatch.setenv("WT_FAULT", "pread:5")
    with pytest.raises(wt.WtError) as ei:
        dev.adopt(h, wt.WT_ADOPT_GATHER, s.cuda_stream)
    monkeypatch.delenv("WT_FAULT")
    assert ei.value.code == wt.WT_EIO and "injected" in str(ei.value)
    s.synchronize()
    for b in dev.bufs:
        b.fill_(0xA5)
    torch.cuda.synchronize()
    ev = dev.adopt(h, wt.WT_ADOPT_GATHER, s.cuda_stream)
    s.synchronize()
    assert all(ev.values())
    check_bytes(torch, h, dev, co)
    assert h.device_status() == 0
    h.close()
