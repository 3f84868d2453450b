"""The N > 1 path of bench.py on CPU: independent replicas whose only exchange is
the max over ranks of the timing; checked with two gloo ranks."""
import os
import socket
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    sys.path.insert(0, ROOT)
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    # rank r was slower on the first value, faster on the second
    got = bench.max_over_ranks([1.0 + rank, 10.0 - rank])
    thr = bench.job_throughput(world, 16, 100, got[0])
    dist.barrier()
    dist.destroy_process_group()
    out.put((rank, got, thr))


def test_max_over_ranks_and_job_throughput_two_gloo_ranks():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, out)) for r in range(world)]
    for p in procs:
        p.start()
    res = sorted(out.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, got, thr in res:
        assert got == [2.0, 10.0]  # every rank sees the slowest replica's times
        assert thr == pytest.approx(2 * 16 * 100 / 2.0e-3)  # units of all ranks / the slowest time


def test_single_process_values_pass_through():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks([3.5, 1.25]) == [3.5, 1.25]
    assert bench.job_throughput(1, 4096, 10, 20.0) == pytest.approx(4096 * 10 / 0.02)
