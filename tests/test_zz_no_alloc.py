"""wt_checksum_noalloc, called through the C ABI, against wt_checksum.

wt_checksum_noalloc is for callers that cannot allocate device memory at the
moment they need a digest: code running inside an allocator hook, programs that
have given all device memory to their own pool, loops that cannot take the
synchronisation cudaFree brings.  Instead of a temporary allocation it keeps its
leaf digests in a fixed array inside the library.  These tests check that its
digests equal those of the allocating entry point on two calls in a row (the
second call must not see anything left over from the first), and that input
too large for the fixed array is refused rather than overrun.  Digests are
integers, so the comparison is exact.
"""
import numpy as np
import pytest

from paper_2608_12114_gb300 import build, wt

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch():
    import torch
    assert torch.cuda.is_available()
    build.build()
    wt.lib()
    return torch


def _digests_both_ways(torch, ptrs, sizes):
    n = len(ptrs)
    ref = torch.zeros(n, dtype=torch.int64, device="cuda")
    got = torch.full((n,), -1, dtype=torch.int64, device="cuda")
    with wt.Handle([]) as h:
        h.checksum(ptrs, sizes, ref.data_ptr(), 0)
    wt.checksum_noalloc(ptrs, sizes, got.data_ptr(), 0)
    torch.cuda.synchronize()
    return ref.cpu().tolist(), got.cpu().tolist()


def test_matches_allocating_entry_point_two_calls_in_a_row(torch):
    rng = np.random.default_rng(11)
    data = torch.from_numpy(rng.integers(0, 256, 6 << 20, dtype=np.uint8)).cuda()
    base = data.data_ptr()
    # call 1: many buffers, odd sizes and offsets, more than one launch's worth of buffers
    sizes1 = [int(s) for s in rng.integers(0, 40000, 300)] + [0, 1, 4095, 4096, 4097, 1 << 20]
    offs1 = [int(o) for o in rng.integers(0, 4 << 20, len(sizes1))]
    ref1, got1 = _digests_both_ways(torch, [base + o for o in offs1], sizes1)
    assert got1 == ref1
    # call 2: different, fewer leaves; stale leaf slots from call 1 must not leak in
    sizes2 = [3, 5000, 12288, 70000]
    offs2 = [7, 100, 4096 * 9 + 1, 999]
    ref2, got2 = _digests_both_ways(torch, [base + o for o in offs2], sizes2)
    assert got2 == ref2
    assert got2 != got1[:4]


def test_refuses_input_beyond_the_fixed_array(torch):
    # 4 GiB + one byte needs 1,048,577 leaves, one more than the array holds; the
    # buffer is real so nothing could be read out of bounds even if the check were missing
    big = torch.empty((4 << 30) + 1, dtype=torch.uint8, device="cuda")
    out = torch.zeros(1, dtype=torch.int64, device="cuda")
    with pytest.raises(wt.WtError) as ei:
        wt.checksum_noalloc([big.data_ptr()], [big.numel()], out.data_ptr(), 0)
    assert ei.value.code == wt.WT_EINVAL
    assert "4 GiB" in str(ei.value)
    torch.cuda.synchronize()
    assert out.item() == 0
    # exactly at the limit is accepted and matches the allocating entry point
    ref, got = _digests_both_ways(torch, [big.data_ptr()], [4 << 30])
    assert got == ref
    del big
