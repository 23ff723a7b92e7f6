"""Lifetime and cold-cache checks on the GPU.

Sec. 5.1 asks that a file-backed tensor's lifetime leave nothing behind (its producer
runs 200 consumed and 200 unconsumed cycles with a flat footprint); here the same holds for
the whole device path: 200 x (wt_open -> wt_adopt -> wt_pass -> wt_close) on the REGISTER
and the DIRECT routes keep device memory, RSS, open descriptors, the files' mappings and the
library's own live objects (wt_live) flat.

Sec. 6.4 (RQ3) checks that digests after complete eviction still reproduce the file's values:
here the test's own file is dropped from the page cache (posix_fadvise DONTNEED on that file
only), ingested cold on each route, and its tree and plain digests compared with the oracle's.
"""
import os
import shutil

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


def rss_bytes():
    for line in open("/proc/self/status"):
        if line.startswith("VmRSS:"):
            return int(line.split()[1]) * 1024
    return 0


def footprint(torch, tag):
    free, _ = torch.cuda.mem_get_info()
    return {"free": free, "rss": rss_bytes(), "fds": len(os.listdir("/proc/self/fd")),
            "maps": sum(1 for l in open("/proc/self/maps") if tag in l), "live": wt.live()}


@pytest.mark.parametrize("route", [wt.WT_ROUTE_REGISTER, wt.WT_ROUTE_DIRECT], ids=["register", "direct"])
def test_200_device_cycles_are_flat(torch, tmp_path, route):
    d = str(tmp_path / ("cyc%d" % route))
    ck = synth.build("many", d, n_matrices=6)  # 12 files, row blocks joined on the device
    s = torch.cuda.Stream()

    def cycle(dev, xs, ys):
        with wt.Handle(ck.paths, route) as h:
            assert all(h.route(f) == route for f in range(h.n_files))
            ev = dev.adopt(h, wt.WT_ADOPT_GATHER, s.cuda_stream)
            h.pass_(dev.descs(xs, ys, ev), s.cuda_stream)
            s.synchronize()
            assert h.device_status() == 0

    with wt.Handle(ck.paths, route) as h0:
        dev = pipeline.DeviceCheckpoint.allocate(h0, pipeline.matrices(h0))
        xs, ys = dev.inputs(), dev.outputs()
    for _ in range(5):  # warm-up: the library's pools, torch's allocator, the driver's caches
        cycle(dev, xs, ys)
    torch.cuda.synchronize()
    before = footprint(torch, d)
    first = {k: y.clone() for k, y in ys.items()}
    for _ in range(200):
        cycle(dev, xs, ys)
    torch.cuda.synchronize()
    after = footprint(torch, d)
    assert all(torch.equal(first[k], ys[k]) for k in ys)  # every cycle computed the same y
    assert after["live"] == before["live"], (before["live"], after["live"])
    assert after["live"]["handles"] == 0
    assert after["fds"] == before["fds"]
    assert after["maps"] == before["maps"] == 0
    assert abs(after["free"] - before["free"]) <= (2 << 20), (before["free"], after["free"])
    assert after["rss"] - before["rss"] <= (16 << 20), (before["rss"], after["rss"])
    # the results are right, not only repeatable
    co = oracle.CheckpointOracle(ck.paths)
    try:
        with wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY) as h:
            for k in dev.gemv_mats():
                m = dev.mats[k]
                W = co.matrix_bytes([(h.tensors[i].file, h.tensors[i].name) for i in m.parts])
                yhat, a = oracle.gemv(W, m.dtype, m.shape[0], m.shape[1], synth.make_x(m.shape[1], m.dtype))
                assert oracle.gemv_error(ys[k].cpu().numpy(), yhat, a) <= 2e-3
    finally:
        co.close()
    shutil.rmtree(d, ignore_errors=True)


def evict(paths):
    """Drop the files' pages (and only theirs) from the page cache."""
    for p in paths:
        fd = os.open(p, os.O_RDONLY)
        try:
            os.fdatasync(fd)
            os.posix_fadvise(fd, 0, 0, os.POSIX_FADV_DONTNEED)
        finally:
            os.close(fd)


@pytest.mark.parametrize("route,mode", [(wt.WT_ROUTE_DIRECT, wt.WT_ADOPT_GATHER),
                                        (wt.WT_ROUTE_REGISTER, wt.WT_ADOPT_GATHER),
                                        (wt.WT_ROUTE_DIRECT, wt.WT_ADOPT_STAGED)],
                         ids=["direct-gather", "register-gather", "staged"])
def test_bytes_after_eviction_match_the_oracle(torch, tmp_path, route, mode):
    d = str(tmp_path / "ev")
    ck = synth.build("mid", d, layers=1, vocab=4096, workers=4)  # ~118 MB, 3 files
    evict(ck.paths)
    s = torch.cuda.Stream()
    with wt.Handle(ck.paths, route | wt.WT_OPEN_HOST_ONLY) as hq:
        resident, total = hq.residency()
    # the page cache may keep a few pages (the index read by the open above), never the bulk
    if resident > total // 2:
        pytest.skip("this file system keeps the pages after DONTNEED (%d of %d bytes)" % (resident, total))
    with wt.Handle(ck.paths, route) as h:
        dev = pipeline.DeviceCheckpoint.allocate(h, pipeline.matrices(h))
        for b in dev.bufs:
            b.fill_(0xA5)
        torch.cuda.synchronize()
        dev.adopt(h, mode, s.cuda_stream)
        s.synchronize()
        idx = list(range(len(h.tensors)))
        ptrs = [dev.dst[i] for i in idx]
        nb = [h.tensors[i].nbytes for i in idx]
        out = torch.zeros(len(idx), dtype=torch.int64, device="cuda")
        outp = torch.zeros(len(idx), dtype=torch.int64, device="cuda")
        h.checksum(ptrs, nb, out.data_ptr(), s.cuda_stream)
        h.checksum(ptrs, nb, outp.data_ptr(), s.cuda_stream, plain=True)
        s.synchronize()
        tree = [int(v) & (2 ** 64 - 1) for v in out.cpu().tolist()]
        plain = [int(v) & (2 ** 64 - 1) for v in outp.cpu().tolist()]
        names = [(t.file, t.name) for t in h.tensors]
    co = oracle.CheckpointOracle(ck.paths)  # read after the GPU path, which found the cache cold
    try:
        for i, (f, nm) in enumerate(names):
            blob = co.blob_of(f, nm)
            assert tree[i] == oracle.fnv_tree(blob), nm
            assert plain[i] == oracle.fnv1a64(blob), nm
    finally:
        co.close()
    shutil.rmtree(d, ignore_errors=True)


def test_block_cache_serves_later_handles(torch):
    """A closed handle's status word, plan tables (pinned and device) and split-K workspace go
    back to the library's block cache and later handles take them from there: the bytes the
    cache holds stay constant over the cycles, the bytes handed out return to their earlier
    value, and every cycle computes the same y, within the bound of the oracle."""
    rng = np.random.default_rng(11)
    shapes = [(64, 4096), (8, 40000)]  # the second is cut into column segments: a workspace
    cases, descs = [], []
    for M, K in shapes:
        W = synth.f32_to_bf16_bits((0.02 * rng.standard_normal((M, K))).astype(np.float32)).view(np.uint8).reshape(-1)
        x = synth.make_x(K, wt.WT_BF16)
        Wd, xd = torch.from_numpy(W.copy()).cuda(), torch.from_numpy(x.copy()).cuda()
        y = torch.full((M,), float("nan"), dtype=torch.float32, device="cuda")
        cases.append((W, x, Wd, xd, y))
        descs.append(wt.gemv_desc(Wd.data_ptr(), wt.WT_BF16, M, K, xd.data_ptr(), y.data_ptr()))
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    torch.cuda.synchronize()
    with wt.Handle([]) as h:  # warm-up: the cache takes this handle's blocks at close
        h.pass_(descs, s1.cuda_stream)
    base = wt.live()
    counts, first = [], None
    for _ in range(20):
        with wt.Handle([]) as h:
            h.pass_(descs, s1.cuda_stream)
            s2.wait_stream(s1)
            h.pass_(descs, s2.cuda_stream)  # the same plan on a second stream; close waits for both
            assert wt.live()["device_bytes"] > base["device_bytes"]
        counts.append(wt.live())
        s2.synchronize()
        ys = [c[4].clone() for c in cases]
        if first is None:
            first = ys
        assert all(torch.equal(a, b) for a, b in zip(first, ys))
    assert all(c == base for c in counts), (base, counts[-1])
    assert base["cached_device_bytes"] > 0 and base["cached_pinned_bytes"] > 0
    for (W, x, _, _, _), (M, K), y in zip(cases, shapes, first):
        yhat, a = oracle.gemv(W, wt.WT_BF16, M, K, x)
        assert oracle.gemv_error(y.cpu().numpy(), yhat, a) <= 2e-3


def test_plan_run_on_many_streams_holds_few_events(torch):
    """A plan keeps one completion event per stream it ran on, at most eight: a caller that
    runs one pass on ever-new streams holds a bounded number of events, and closing the handle
    releases them."""
    rng = np.random.default_rng(12)
    M, K = 96, 2048
    W = synth.f32_to_bf16_bits((0.02 * rng.standard_normal((M, K))).astype(np.float32)).view(np.uint8).reshape(-1)
    x = synth.make_x(K, wt.WT_BF16)
    Wd, xd = torch.from_numpy(W.copy()).cuda(), torch.from_numpy(x.copy()).cuda()
    y = torch.full((M,), float("nan"), dtype=torch.float32, device="cuda")
    d = [wt.gemv_desc(Wd.data_ptr(), wt.WT_BF16, M, K, xd.data_ptr(), y.data_ptr())]
    with wt.Handle([]) as h:  # warm-up: the block cache takes this plan's blocks at close
        h.pass_(d, 0)
    torch.cuda.synchronize()
    base = wt.live()
    streams = [torch.cuda.Stream() for _ in range(12)]
    with wt.Handle([]) as h:
        prev = None
        for s in streams:
            if prev is not None:
                s.wait_stream(prev)  # one run at a time: they all write the same y
            h.pass_(d, s.cuda_stream)
            prev = s
        live = wt.live()
        assert live["plans"] == base["plans"] + 1
        assert live["events"] <= base["events"] + 1 + 8, (base, live)  # the upload event and 8 streams
    torch.cuda.synchronize()
    assert wt.live() == base
    yhat, a = oracle.gemv(W, wt.WT_BF16, M, K, x)
    assert oracle.gemv_error(y.cpu().numpy(), yhat, a) <= 2e-3
