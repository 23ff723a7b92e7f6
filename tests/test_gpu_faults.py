"""Failure detection on the GPU without a GPU fault.  Failures are made on the host
(WT_FAULT): a registration or allocation that "fails", and a GEMV launch whose producer
issues no copy, so every mbarrier wait of the kernel runs out (~1 s).  The kernel must then
report WT_ETIMEDOUT through the handle's status word and leave the context usable."""
import os

import numpy as np
import pytest

import oracle
from paper_2608_12114_gb300 import build, synth, wt

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch():
    import torch
    assert torch.cuda.is_available()
    build.build()
    wt.lib()
    return torch


def bf16_case(torch, M=64, K=4096, seed=5):
    W = synth.f32_to_bf16_bits((0.02 * np.random.default_rng(seed).standard_normal((M, K))).astype(np.float32))
    Wraw = W.view(np.uint8).reshape(-1)
    x = synth.make_x(K, wt.WT_BF16)
    return Wraw, x, torch.from_numpy(Wraw.copy()).cuda(), torch.from_numpy(x.copy()).cuda()


def test_stalled_launch_times_out_and_the_context_survives(torch, monkeypatch):
    M, K = 64, 4096
    Wraw, x, Wd, xd = bf16_case(torch, M, K)
    y = torch.zeros(M, dtype=torch.float32, device="cuda")
    d = [wt.gemv_desc(Wd.data_ptr(), wt.WT_BF16, M, K, xd.data_ptr(), y.data_ptr())]
    with wt.Handle([]) as h:
        monkeypatch.setenv("WT_FAULT", "stall")
        h.pass_(d, 0)
        torch.cuda.synchronize()                     # returns: the waits gave up
        assert h.device_status() == wt.WT_ETIMEDOUT
        monkeypatch.delenv("WT_FAULT")
    with wt.Handle([]) as h:                         # same process, same context: still good
        assert h.device_status() == 0                # the recycled status word was cleared
        h.pass_(d, 0)
        torch.cuda.synchronize()
        assert h.device_status() == 0
    yhat, a = oracle.gemv(Wraw, wt.WT_BF16, M, K, x)
    assert oracle.gemv_error(y.cpu().numpy(), yhat, a) <= 2e-3


def test_injected_plan_allocation_failure(torch, monkeypatch):
    M, K = 16, 1024
    Wraw, x, Wd, xd = bf16_case(torch, M, K, seed=6)
    y = torch.zeros(M, dtype=torch.float32, device="cuda")
    d = [wt.gemv_desc(Wd.data_ptr(), wt.WT_BF16, M, K, xd.data_ptr(), y.data_ptr())]
    with wt.Handle([]) as h:
        monkeypatch.setenv("WT_FAULT", "alloc")
        with pytest.raises(wt.WtError) as ei:
            h.pass_(d, 0)
        assert ei.value.code == wt.WT_ENOMEM
        monkeypatch.delenv("WT_FAULT")
        h.pass_(d, 0)                                 # the failed plan left nothing behind
        torch.cuda.synchronize()
        assert h.device_status() == 0
    yhat, a = oracle.gemv(Wraw, wt.WT_BF16, M, K, x)
    assert oracle.gemv_error(y.cpu().numpy(), yhat, a) <= 2e-3


def test_injected_registration_failure_leaks_nothing(torch, tmp_path, monkeypatch):
    ck = synth.build("many", str(tmp_path / "m"), n_matrices=6)
    wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY).close()
    fds = len(os.listdir("/proc/self/fd"))
    monkeypatch.setenv("WT_FAULT", "register:3")
    with pytest.raises(wt.WtError) as ei:
        wt.Handle(ck.paths, wt.WT_ROUTE_REGISTER)    # an explicit route that fails is an error
    assert ei.value.code == wt.WT_ECUDA
    monkeypatch.delenv("WT_FAULT")
    assert len(os.listdir("/proc/self/fd")) == fds
    assert not [l for l in open("/proc/self/maps") if str(tmp_path) in l]
