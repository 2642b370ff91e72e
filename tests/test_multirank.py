"""The bench's N > 1 path on CPU: two gloo ranks, each a replica that
processed its own bytes in its own time.  The job's time is the slowest
rank's, and its throughput counts the bytes of every rank."""

import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def rank_main(rank, world, port, times, nbytes, results):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import sys
        sys.path.insert(0, ROOT)
        import bench
        dist.barrier()
        total_s, value = bench.aggregate(nbytes, times[rank], world, "cpu")
        results[rank] = (total_s, value)
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("times", [(0.50, 0.75), (2.0, 1.0)])
def test_two_gloo_ranks_take_the_slowest(times):
    world, nbytes = 2, 3.0e9
    ctx = mp.get_context("spawn")
    with ctx.Manager() as mgr:
        results = mgr.dict()
        mp.start_processes(rank_main, args=(world, free_port(), times, nbytes, results),
                           nprocs=world, start_method="spawn", join=True)
        got = dict(results)
    slowest = max(times)
    for rank in range(world):
        total_s, value = got[rank]
        assert total_s == pytest.approx(slowest)
        assert value == pytest.approx(world * nbytes / slowest / 1e9)


def test_single_rank_needs_no_process_group():
    import sys
    sys.path.insert(0, ROOT)
    import bench
    assert not dist.is_initialized()
    total_s, value = bench.aggregate(5e9, 2.0, 1)
    assert total_s == 2.0 and value == pytest.approx(2.5)
