"""Cross-CTA split-K (rows longer than the segment length): few rows, very long rows, every
dtype, ragged last segments; results against the oracle and independent of grouping."""
import numpy as np
import pytest

import oracle
from paper_2608_12114_gb300 import build, synth, wt

pytestmark = pytest.mark.gpu
TOL = 2e-3
F32, BF16, F16, I8 = wt.WT_F32, wt.WT_BF16, wt.WT_F16, wt.WT_I8

# (dtype, M, K): V = K * es / 16 vectors per row, cut into ceil(V / 2048) (int8: 512)
# segments of nearly equal length
SHAPES = [(BF16, 1, 8 * 1024 * 1024),      # V = 1,048,576: 512 one-row segments
          (BF16, 5, 65544),                 # V = 8193: 5 segments, the last shorter
          (I8, 3, 600000),                  # V = 37500: 74 segments
          (F32, 2, 1048580),                # V = 262145: 129 segments
          (F16, 9, 40000),                  # V = 5000: 3 segments
          (BF16, 17, 32768),                # V = 4096: 2 segments
          (BF16, 40, 16384)]                # V = 2048: not split


@pytest.fixture(scope="module")
def torch():
    import torch
    assert torch.cuda.is_available()
    build.build()
    wt.lib()
    return torch


def make(torch, rng, dtype, M, K):
    if dtype == I8:
        W = rng.integers(-128, 128, M * K).astype(np.int8).view(np.uint8)
        s = rng.uniform(0.001, 0.02, M).astype(np.float16).view(np.uint8)
        x = synth.make_x(K, I8)
    elif dtype == BF16:
        W = synth.f32_to_bf16_bits((0.02 * rng.standard_normal(M * K)).astype(np.float32)).view(np.uint8)
        s, x = None, synth.make_x(K, BF16)
    elif dtype == F16:
        W = (0.02 * rng.standard_normal(M * K)).astype(np.float16).view(np.uint8)
        s, x = None, synth.make_x(K, F16)
    else:
        W = (0.02 * rng.standard_normal(M * K)).astype(np.float32).view(np.uint8)
        s, x = None, synth.make_x(K, F32)
    dev = lambda a: None if a is None else torch.from_numpy(np.ascontiguousarray(a)).cuda()  # noqa: E731
    return dict(dtype=dtype, M=M, K=K, W=W, s=s, x=x, Wd=dev(W), sd=dev(s), xd=dev(x),
                y=torch.full((M,), float("nan"), dtype=torch.float32, device="cuda"))


def desc(c, y):
    return wt.gemv_desc(c["Wd"].data_ptr(), c["dtype"], c["M"], c["K"], c["xd"].data_ptr(), y.data_ptr(),
                        scale=c["sd"].data_ptr() if c["sd"] is not None else 0)


def test_long_rows_against_oracle_and_grouping(torch):
    rng = np.random.default_rng(77)
    cases = [make(torch, rng, *sh) for sh in SHAPES]
    with wt.Handle([]) as h:
        h.pass_([desc(c, c["y"]) for c in cases], 0)      # all in one group
        torch.cuda.synchronize()
        assert h.device_status() == 0
        for c in cases:
            if c["dtype"] == I8:
                yhat, a = oracle.gemv_q8(c["W"], c["s"], c["M"], c["K"], c["x"])
            else:
                yhat, a = oracle.gemv(c["W"], c["dtype"], c["M"], c["K"], c["x"])
            err = oracle.gemv_error(c["y"].cpu().numpy(), yhat, a)
            assert err <= TOL, (c["dtype"], c["M"], c["K"], err)
        for c in cases:                                    # alone: the same bits
            y2 = torch.full_like(c["y"], float("nan"))
            h.pass_([desc(c, y2)], 0)
            torch.cuda.synchronize()
            assert torch.equal(y2, c["y"]), (c["dtype"], c["M"], c["K"])
