"""wt_pass inside a captured CUDA graph: the resident pass of a launch-bound loop replays
without host work.  A capture needs the same descriptors run once outside it (the plan's
tables resident); the captured plan survives the plan cache's eviction."""
import numpy as np
import pytest

from paper_2608_12114_gb300 import build, synth, wt

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch():
    import torch
    assert torch.cuda.is_available()
    build.build()
    wt.lib()
    return torch


@pytest.mark.filterwarnings("ignore:The CUDA Graph is empty")  # the refused capture records nothing
def test_pass_replays_from_a_cuda_graph(torch):
    rng = np.random.default_rng(3)
    M1, K1 = 300, 4096
    W1 = torch.from_numpy(synth.f32_to_bf16_bits((0.02 * rng.standard_normal((M1, K1))).astype(np.float32))
                          .view(np.uint8).reshape(-1).copy()).cuda()
    x1 = torch.from_numpy(synth.make_x(K1, wt.WT_BF16)).cuda()
    y1 = torch.empty(M1, dtype=torch.float32, device="cuda")
    M2, K2, T = 96, 2048, 4
    W2 = torch.from_numpy(rng.integers(-128, 128, M2 * K2).astype(np.int8).view(np.uint8)).cuda()
    s2 = torch.from_numpy(rng.uniform(0.001, 0.02, M2).astype(np.float16).view(np.uint8)).cuda()
    X2 = torch.from_numpy(rng.standard_normal((T, K2)).astype(np.float16).view(np.uint8).reshape(-1)).cuda()
    y2 = torch.empty(T * M2, dtype=torch.float32, device="cuda")
    descs = [wt.gemv_desc(W1.data_ptr(), wt.WT_BF16, M1, K1, x1.data_ptr(), y1.data_ptr()),
             wt.gemv_desc(W2.data_ptr(), wt.WT_I8, M2, K2, X2.data_ptr(), y2.data_ptr(), scale=s2.data_ptr(),
                          cols=T)]
    s = torch.cuda.Stream()
    with wt.Handle([]) as h:
        g0 = torch.cuda.CUDAGraph()
        with pytest.raises(wt.WtError) as ei:                 # no warm-up: refused before any CUDA call
            with torch.cuda.graph(g0, stream=s):
                h.pass_(descs, torch.cuda.current_stream().cuda_stream)
        assert ei.value.code == wt.WT_EINVAL and "outside the capture" in str(ei.value)
        torch.cuda.synchronize()
        h.pass_(descs, s.cuda_stream)                          # warm-up: builds and uploads the plan
        s.synchronize()
        ref1, ref2 = y1.clone(), y2.clone()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            h.pass_(descs, torch.cuda.current_stream().cuda_stream)
        y1.fill_(float("nan"))
        y2.fill_(float("nan"))
        torch.cuda.synchronize()
        g.replay()
        torch.cuda.synchronize()
        assert torch.equal(y1, ref1) and torch.equal(y2, ref2)
        # 40 other plans push the captured one past the cache limit; it stays alive
        ys = torch.empty(40, 64, dtype=torch.float32, device="cuda")
        for i in range(40):
            h.pass_([wt.gemv_desc(W1.data_ptr(), wt.WT_BF16, 1 + i, K1, x1.data_ptr(), ys[i].data_ptr())], s.cuda_stream)
        s.synchronize()
        for _ in range(10):
            y1.fill_(float("nan"))
            g.replay()
        torch.cuda.synchronize()
        assert torch.equal(y1, ref1) and torch.equal(y2, ref2)
        assert torch.equal(ys[39, :40], ref1[:40])           # row results do not depend on grouping
        assert h.device_status() == 0
        del g
