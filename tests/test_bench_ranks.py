"""The benchmark's multi-rank timing on CPU (gloo, two ranks): each rank runs an
independent replica, the job's time is the slowest rank's, and the whole-job rate counts
every rank's images over that time."""
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms = 100.0 + 25.0 * rank  # rank 1 is the slower replica
        out[rank] = bench.max_over_ranks(ms)
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_time():
    world, port = 2, _free_port()
    out = mp.Manager().dict()
    mp.spawn(_rank, args=(world, port, out), nprocs=world, join=True)
    assert dict(out) == {0: 125.0, 1: 125.0}
    sys.path.insert(0, ROOT)
    import bench
    # 1920 images per step per rank, 2 ranks, 20 steps in 125 ms: weak scaling counts both ranks' images
    assert bench.whole_job_rate(1920, world, 20, 125.0) == pytest.approx(2 * 1920 * 20 / 0.125)


def test_one_process_without_a_group_is_its_own_max():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(42.5) == 42.5
