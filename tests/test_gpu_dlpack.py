"""The file-backed producer on the GPU (Algorithm 1 with a CUDA device capsule): the adopted
torch tensor is a cuda tensor whose storage is the file's pages, read in place by the GPU
(torch kernels, the checksum kernel, and the GEMV's plain-load path).  Reads only: the
pages are PROT_READ, and a device store into them would fault the context."""
import gc
import inspect
import os

import numpy as np
import pytest

import oracle
from paper_2608_12114_gb300 import build, synth, wt

pytestmark = pytest.mark.gpu
PAGE = os.sysconf("SC_PAGE_SIZE")


@pytest.fixture(scope="module")
def torch():
    import torch
    assert torch.cuda.is_available()
    build.build()
    wt.lib()
    import torch.utils.dlpack as tdl
    if "max_version" not in inspect.getsource(tdl.from_dlpack):
        pytest.skip("this torch does not request versioned DLPack capsules")
    return torch


def bf16_file(path, M, K, seed):
    bits = synth.f32_to_bf16_bits((0.02 * np.random.default_rng(seed).standard_normal((M, K))).astype(np.float32))
    with open(path, "wb") as f:
        f.write(bits.astype("<u2").tobytes())
    return bits.view(np.uint8).reshape(-1)


def test_device_capsule_is_read_in_place(torch, tmp_path):
    M, K = 64, PAGE  # M*K*2 bytes: whole pages
    p = str(tmp_path / "w.bin")
    raw = bf16_file(p, M, K, 1)
    ft = wt.FileTensor.from_file(p, wt.WT_BF16, M, K)
    assert ft.__dlpack_device__() == (wt.kDLCUDA, torch.cuda.current_device())
    ptr = ft.data_ptr
    t = torch.from_dlpack(ft)
    assert t.is_cuda and t.dtype == torch.bfloat16 and tuple(t.shape) == (M, K) and t.data_ptr() == ptr
    ref = torch.from_numpy(raw.copy()).cuda().view(M, 2 * K)
    assert torch.equal(t.view(torch.uint8), ref)                     # a torch kernel reads the pages
    with wt.Handle([]) as h:
        out = torch.zeros(1, dtype=torch.int64, device="cuda")
        h.checksum([t.data_ptr()], [M * K * 2], out.data_ptr(), 0)   # the checksum kernel reads them
        assert int(out.item()) & (2 ** 64 - 1) == oracle.fnv_tree(raw)
        x = torch.from_numpy(synth.make_x(K, wt.WT_BF16)).cuda()
        y = torch.full((M,), float("nan"), dtype=torch.float32, device="cuda")
        h.pass_([wt.gemv_desc(t.data_ptr(), wt.WT_BF16, M, K, x.data_ptr(), y.data_ptr())], 0)
        torch.cuda.synchronize()                                      # host W: plain-load GEMV
        assert h.device_status() == 0
    yhat, a = oracle.gemv(raw, wt.WT_BF16, M, K, synth.make_x(K, wt.WT_BF16))
    assert oracle.gemv_error(y.cpu().numpy(), yhat, a) <= 2e-3
    T = 5                                                             # and with T columns
    X = synth.f32_to_bf16_bits(np.random.default_rng(2).standard_normal((T, K)).astype(np.float32)).view(np.uint8)
    Xd = torch.from_numpy(X.reshape(-1).copy()).cuda()
    Y = torch.full((T * M,), float("nan"), dtype=torch.float32, device="cuda")
    with wt.Handle([]) as h:
        h.pass_([wt.gemv_desc(t.data_ptr(), wt.WT_BF16, M, K, Xd.data_ptr(), Y.data_ptr(), cols=T)], 0)
        torch.cuda.synchronize()
        assert h.device_status() == 0
    Yh, A = oracle.gemv_cols(raw, wt.WT_BF16, M, K, X.reshape(-1), T)
    assert oracle.gemv_error(Y.cpu().numpy(), Yh.reshape(-1), A.reshape(-1)) <= 2e-3
    fd = os.open(p, os.O_WRONLY)                                     # the file stays the storage
    os.pwrite(fd, b"\x80\x3f", 2 * (K + 1))                          # element (1, 1) = 1.0
    os.close(fd)
    torch.cuda.synchronize()
    assert float(t[1, 1].float().item()) == 1.0
    del t
    gc.collect()
    assert wt.dlpack_live() == 0


def test_device_capsules_from_a_handle_and_cycles(torch, tmp_path):
    ck = synth.build("mid", str(tmp_path / "mid"), layers=1, vocab=64)
    co = oracle.CheckpointOracle(ck.paths)
    with wt.Handle(ck.paths) as h:
        for i, info in enumerate(h.tensors[:8]):
            t = torch.from_dlpack(wt.FileTensor.from_handle(h, i))
            ref = torch.from_numpy(co.blob_of(info.file, info.name).copy()).cuda()
            assert t.is_cuda and torch.equal(t.reshape(-1).view(torch.uint8), ref), info.name
            del t
    co.close()
    M, K = 16, PAGE
    p = str(tmp_path / "c.bin")
    bf16_file(p, M, K, 2)
    gc.collect()
    fds = len(os.listdir("/proc/self/fd"))
    for i in range(200):
        t = torch.from_dlpack(wt.FileTensor.from_file(p, wt.WT_BF16, M, K))
        assert t.is_cuda
        del t
        ft = wt.FileTensor.from_file(p, wt.WT_BF16, M, K)
        if i % 2:
            ft.__dlpack__(max_version=(1, 0))
        del ft
    gc.collect()
    assert wt.dlpack_live() == 0
    assert len(os.listdir("/proc/self/fd")) == fds
    assert not [l for l in open("/proc/self/maps") if p in l]
