"""The file-backed tensor producer (Algorithm 1, Sec. 7.1) through torch.from_dlpack, on the
host (WT_DLPACK_HOST capsules: no GPU needed): content identity, file-write aliasing,
the size and page guards, lifetime after every producer reference is gone, deleter on
another thread, and 200 consumed plus 200 unconsumed capsule cycles leaving the process
flat (live capsules, descriptors, mappings, resident memory)."""
import gc
import os
import threading

import numpy as np
import pytest

import oracle
from paper_2608_12114_gb300 import build, synth, wt

PAGE = os.sysconf("SC_PAGE_SIZE")


@pytest.fixture(scope="module")
def torch():
    import torch
    build.build()
    wt.lib()
    return torch


def write(path, arr):
    with open(path, "wb") as f:
        f.write(np.ascontiguousarray(arr).tobytes())
    return path


def mapped(path):
    return [l for l in open("/proc/self/maps") if path in l]


def rss_kib():
    for l in open("/proc/self/status"):
        if l.startswith("VmRSS:"):
            return int(l.split()[1])
    return 0


@pytest.mark.parametrize("dtype,npdt,K", [(wt.WT_F32, np.float32, PAGE // 4), (wt.WT_F16, np.float16, PAGE // 2),
                                          (wt.WT_I8, np.int8, PAGE), (wt.WT_U8, np.uint8, PAGE),
                                          (wt.WT_BF16, np.uint16, PAGE // 2)])
def test_content_shape_strides_flags(torch, tmp_path, dtype, npdt, K):
    M = 3
    rng = np.random.default_rng(dtype)
    a = rng.integers(-100, 100, (M, K)).astype(npdt)
    p = write(str(tmp_path / "t.bin"), a)
    ft = wt.FileTensor.from_file(p, dtype, M, K, wt.WT_DLPACK_HOST)
    assert ft.shape == (M, K) and ft.strides == (K, 1)
    assert ft.version == (1, 0) and ft.flags & wt.DLPACK_FLAG_BITMASK_READ_ONLY
    assert ft.__dlpack_device__() == (wt.kDLCPU, 0)
    t = torch.from_dlpack(ft)
    want = {wt.WT_F32: torch.float32, wt.WT_F16: torch.float16, wt.WT_I8: torch.int8, wt.WT_U8: torch.uint8,
            wt.WT_BF16: torch.bfloat16}[dtype]
    assert t.dtype == want and tuple(t.shape) == (M, K) and t.stride() == (K, 1)
    assert t.view(torch.uint8).numpy().tobytes() == open(p, "rb").read()   # the file's bytes, unchanged
    del t


def test_tensor_aliases_the_file(torch, tmp_path):
    """MAP_SHARED: a write to the file through another descriptor shows in the adopted tensor."""
    M, K = 2, PAGE // 4
    p = write(str(tmp_path / "a.bin"), np.zeros((M, K), np.float32))
    t = torch.from_dlpack(wt.FileTensor.from_file(p, wt.WT_F32, M, K, wt.WT_DLPACK_HOST))
    assert float(t.sum()) == 0.0
    fd = os.open(p, os.O_WRONLY)
    os.pwrite(fd, np.array([7.5], np.float32).tobytes(), 4 * (K + 3))
    os.close(fd)
    assert float(t[1, 3]) == 7.5 and float(t.sum()) == 7.5


def test_guards_reject(torch, tmp_path):
    p = write(str(tmp_path / "odd.bin"), np.zeros(PAGE + 64, np.uint8))   # partial last page
    with pytest.raises(wt.WtError) as ei:
        wt.FileTensor.from_file(p, wt.WT_U8, 1, PAGE + 64, wt.WT_DLPACK_HOST)
    assert ei.value.code == wt.WT_EINVAL and "page" in str(ei.value)
    q = write(str(tmp_path / "ok.bin"), np.zeros(2 * PAGE, np.uint8))
    for M, K, dt in ((1, PAGE, wt.WT_U8), (2, PAGE, wt.WT_F16), (2, PAGE // 2, wt.WT_F32)):  # size mismatch
        with pytest.raises(wt.WtError) as ei:
            wt.FileTensor.from_file(q, dt, M, K, wt.WT_DLPACK_HOST)
        assert ei.value.code == wt.WT_EINVAL
    with pytest.raises(wt.WtError) as ei:
        wt.FileTensor.from_file(q, 9, 2, PAGE, wt.WT_DLPACK_HOST)
    assert ei.value.code == wt.WT_EINVAL
    with pytest.raises(wt.WtError) as ei:
        wt.FileTensor.from_file(str(tmp_path / "missing.bin"), wt.WT_U8, 1, PAGE, wt.WT_DLPACK_HOST)
    assert ei.value.code == wt.WT_EIO
    z = write(str(tmp_path / "empty.bin"), np.zeros(0, np.uint8))
    with pytest.raises(wt.WtError):
        wt.FileTensor.from_file(z, wt.WT_U8, 0, 0, wt.WT_DLPACK_HOST)
    assert wt.dlpack_live() == 0 and not mapped(str(tmp_path))


def test_lifetime_follows_the_consumer(torch, tmp_path):
    M, K = 4, PAGE // 4
    a = np.arange(M * K, dtype=np.float32).reshape(M, K)
    p = write(str(tmp_path / "l.bin"), a)
    base = wt.dlpack_live()
    ft = wt.FileTensor.from_file(p, wt.WT_F32, M, K, wt.WT_DLPACK_HOST)
    t = torch.from_dlpack(ft)
    del ft
    gc.collect()
    assert wt.dlpack_live() == base + 1 and mapped(p)     # the tensor holds the mapping
    assert np.array_equal(t.numpy(), a)
    v = t[2:]                                                # views share the storage
    del t
    gc.collect()
    assert wt.dlpack_live() == base + 1 and float(v[0, 0]) == float(a[2, 0])
    del v
    gc.collect()
    assert wt.dlpack_live() == base and not mapped(p)       # last reference gone: unmapped


def test_unconsumed_paths_release(torch, tmp_path):
    p = write(str(tmp_path / "u.bin"), np.ones(PAGE, np.uint8))
    base = wt.dlpack_live()
    ft = wt.FileTensor.from_file(p, wt.WT_U8, 1, PAGE, wt.WT_DLPACK_HOST)
    del ft                                                   # never exported
    cap = wt.FileTensor.from_file(p, wt.WT_U8, 1, PAGE, wt.WT_DLPACK_HOST).__dlpack__(max_version=(1, 0))
    assert wt.dlpack_live() == base + 1
    del cap                                                  # exported, never adopted
    gc.collect()
    assert wt.dlpack_live() == base and not mapped(p)
    ft = wt.FileTensor.from_file(p, wt.WT_U8, 1, PAGE, wt.WT_DLPACK_HOST)
    with pytest.raises(BufferError):
        ft.__dlpack__()                                      # unversioned request: refused
    ft.__dlpack__(max_version=(1, 0))
    with pytest.raises(BufferError):
        ft.__dlpack__(max_version=(1, 0))                    # exports once
    gc.collect()
    assert wt.dlpack_live() == base


def test_deleter_runs_on_another_thread(torch, tmp_path):
    p = write(str(tmp_path / "th.bin"), np.ones(PAGE, np.uint8))
    base = wt.dlpack_live()
    fts = [wt.FileTensor.from_file(p, wt.WT_U8, 1, PAGE, wt.WT_DLPACK_HOST) for _ in range(8)]
    ptrs = [ft._p for ft in fts]
    for ft in fts:
        ft._p = None                                         # hand the raw structs to a thread
    th = threading.Thread(target=lambda: [wt.lib().wt_dlpack_release(q) for q in ptrs])
    th.start()
    th.join()
    assert wt.dlpack_live() == base and not mapped(p)


def test_200_consumed_and_200_unconsumed_cycles_stay_flat(torch, tmp_path):
    M, K = 16, PAGE  # 16 pages of uint8
    p = write(str(tmp_path / "c.bin"), np.arange(M * K, dtype=np.uint8))
    for _ in range(5):   # warm the allocators before taking the baseline
        torch.from_dlpack(wt.FileTensor.from_file(p, wt.WT_U8, M, K, wt.WT_DLPACK_HOST)).sum()
    gc.collect()
    base_live, base_fds, base_rss = wt.dlpack_live(), len(os.listdir("/proc/self/fd")), rss_kib()
    for _ in range(200):
        t = torch.from_dlpack(wt.FileTensor.from_file(p, wt.WT_U8, M, K, wt.WT_DLPACK_HOST))
        assert int(t[3, 5]) == (3 * K + 5) % 256
        del t
    for i in range(200):
        ft = wt.FileTensor.from_file(p, wt.WT_U8, M, K, wt.WT_DLPACK_HOST)
        if i % 2:
            ft.__dlpack__(max_version=(1, 0))                # capsule dropped unadopted
        del ft
    gc.collect()
    assert wt.dlpack_live() == base_live
    assert len(os.listdir("/proc/self/fd")) == base_fds
    assert not mapped(p)
    assert rss_kib() - base_rss < 8 * 1024                   # no growth beyond noise (KiB)


def test_handle_tensor_export_outlives_the_handle(torch, tmp_path):
    ck = synth.build("mid", str(tmp_path / "mid"), layers=1, vocab=64)
    co = oracle.CheckpointOracle(ck.paths)
    h = wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY)
    picks = [i for i, t in enumerate(h.tensors) if t.nbytes > 0][:6]
    ts = []
    for i in picks:
        info = h.tensors[i]
        t = torch.from_dlpack(wt.FileTensor.from_handle(h, i, wt.WT_DLPACK_HOST))
        assert tuple(t.shape) == info.shape
        ts.append((info, t))
    h.close()
    for info, t in ts:   # the capsules own their own mappings
        assert t.contiguous().view(torch.uint8).numpy().tobytes() == co.blob_of(info.file, info.name).tobytes()
    co.close()
    del ts, t   # the loop variable holds the last tensor too
    gc.collect()
    assert wt.dlpack_live() == 0
    with pytest.raises(wt.WtError):
        wt.FileTensor.from_handle(wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY), 0, wt.WT_DLPACK_DEVICE)
