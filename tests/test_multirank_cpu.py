"""Multi-rank host logic on CPU (gloo, world size 2).

The translation has no exchange step, so N GPUs run N independent replicas;
the only cross-rank logic is the timing aggregation (slowest rank, whole-job
tokens/s), checked here without a GPU.
"""
import os
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _worker(rank, world, port, q):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    local_ms = [10.0, 25.0][rank]
    ms, value = bench.aggregate(local_ms, tokens_per_step=4096, steps=100, world=world, dist=dist)
    dist.barrier()
    q.put((rank, ms, value))
    dist.destroy_process_group()


def test_two_rank_aggregation_takes_the_slowest_rank():
    world = 2
    port = 29500 + os.getpid() % 1000
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = [q.get(timeout=120) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, ms, value in out:
        assert ms == 25.0
        assert value == pytest.approx(4096 * 100 * 2 / 0.025)


def test_single_rank_aggregation_is_local():
    sys.path.insert(0, ROOT)
    import bench
    ms, value = bench.aggregate(8.0, tokens_per_step=10, steps=5, world=1)
    assert ms == 8.0 and value == pytest.approx(10 * 5 / 0.008)
