"""The N > 1 path of bench.py on CPU: two gloo ranks (replicas only, no collective on the data path) agree on
the slowest rank's time and report the whole-job rate from it."""
import os
import socket
import sys

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def free_port():
    with socket.socket(socket.AF_INET, socket.SOCK_STREAM) as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def rank_main(rank, world, port, times, out):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    try:
        ms = bench.max_over_ranks(times[rank], torch.device("cpu"), world)
        out[rank] = (ms, bench.job_rate(world, 1000, ms))
    finally:
        dist.destroy_process_group()


def test_two_ranks_take_the_slowest_time():
    times = [12.5, 20.0]
    port = free_port()
    ctx = mp.get_context("spawn")
    with ctx.Manager() as manager:
        out = manager.dict()
        mp.start_processes(rank_main, args=(2, port, times, out), nprocs=2, join=True, start_method="spawn")
        res = dict(out)
    assert res[0] == res[1] == (20.0, 2 * 1000 / 0.020)


def test_one_rank_without_a_process_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(7.0, torch.device("cpu"), 1) == 7.0
    assert bench.job_rate(1, 500, 250.0) == 2000.0
