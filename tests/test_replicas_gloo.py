"""The N > 1 host logic of bench.py (replicas, one per GPU, no data-path collective) on
CPU: two gloo ranks on 127.0.0.1, each with its own timings."""
import multiprocessing as mp
import socket

import pytest


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank(rank, world, port, q):
    import torch.distributed as dist

    import bench
    dist.init_process_group("gloo", init_method="tcp://127.0.0.1:%d" % port, rank=rank, world_size=world)
    local_ms, local_e2e = [(100.0, 0.5), (130.0, 0.4)][rank]
    total_ms, e2e_s = bench.combine_ranks(dist, "cpu", local_ms, local_e2e)
    value = bench.aggregate_gbs(1e9 * 10, world, total_ms / 1e3)
    dist.barrier()
    dist.destroy_process_group()
    q.put((rank, total_ms, e2e_s, value))


def test_two_replicas_take_the_max_and_sum_bytes():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    ps = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in ps:
        p.start()
    out = sorted(q.get(timeout=120) for _ in ps)
    for p in ps:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, total_ms, e2e_s, value in out:
        assert total_ms == 130.0 and e2e_s == 0.5          # the slowest replica sets the clock
        assert value == pytest.approx(2 * 10e9 / 0.130 / 1e9)  # bytes of both replicas


def test_single_process_needs_no_group():
    import bench
    assert bench.combine_ranks(None, "cpu", 12.5, 0.25) == (12.5, 0.25)
    assert bench.aggregate_gbs(16e9, 1, 2.0) == pytest.approx(8.0)
