"""bench.py's multi-rank logic on CPU: two gloo ranks, as torchrun would start
them.  The job time is the slowest rank's, the barrier holds every rank, and
the whole-job value counts every rank's bytes (replicas, weak scaling)."""

import os
import sys
import time
from pathlib import Path

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = Path(__file__).resolve().parents[1]


def _rank(rank, world, port, out):
    sys.path.insert(0, str(ROOT))
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    t0 = time.time()
    if rank == 1:
        time.sleep(0.5)  # a slow rank
    bench.barrier(world)
    waited = time.time() - t0
    mx = bench.reduce_max(10.0 * (rank + 1), world)
    out.put((rank, waited, mx))
    dist.destroy_process_group()


def test_two_gloo_ranks_barrier_and_max():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = 29500 + os.getpid() % 1000
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = dict((r, (w, m)) for r, w, m in (q.get(timeout=120) for _ in procs))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert res[0][0] >= 0.45          # rank 0 waited for the slow rank at the barrier
    assert res[0][1] == res[1][1] == 20.0


def test_job_value_counts_every_rank():
    sys.path.insert(0, str(ROOT))
    import bench
    one = bench.job_gbs(1, 5e8, 1.0)
    assert one == pytest.approx(500.0)
    assert bench.job_gbs(4, 5e8, 1.0) == pytest.approx(4 * one)
    assert bench.job_gbs(2, 5e8, 2.0) == pytest.approx(one)
