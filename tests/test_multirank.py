"""Multi-process host logic of the benchmark (replicas: no collective on the
data path, only the max-over-ranks timing reduction), run as two gloo ranks
on the CPU."""
import os
import socket

import pytest


def _free_port() -> int:
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank: int, world: int, port: int, out):
    import torch.distributed as dist
    import bench
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    ms = 10.0 + 5.0 * rank            # rank 1 is the slowest
    m = bench.max_over_ranks(ms, world, "cpu")
    out[rank] = (m, bench.job_throughput(world, 1, 100, m))
    dist.barrier()
    dist.destroy_process_group()


def test_two_rank_timing_reduction_takes_the_slowest_rank():
    mp = pytest.importorskip("torch.multiprocessing")
    ctx = mp.get_context("spawn")
    with ctx.Manager() as mgr:
        out = mgr.dict()
        port = _free_port()
        procs = [ctx.Process(target=_worker, args=(r, 2, port, out)) for r in range(2)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(120)
            assert p.exitcode == 0
        for r in range(2):
            m, v = out[r]
            assert m == 15.0
            # two replicas x 1 token x 100 steps over the slowest rank's 15 ms
            assert abs(v - 2 * 100 / 0.015) < 1e-6


def test_single_rank_needs_no_process_group():
    import bench
    assert bench.max_over_ranks(3.5, 1, "cpu") == 3.5
    assert bench.job_throughput(1, 32, 10, 1000.0) == 320.0
