"""bench.py's multi-rank host logic (replicas, no data-path collective):
the job time is the slowest rank's, the value counts every rank's rows.
Two gloo ranks on the CPU."""
import os
import sys
from pathlib import Path

import pytest
import torch.multiprocessing as mp

ROOT = Path(__file__).resolve().parents[1]


def _rank(rank, world, port, q):
    sys.path.insert(0, str(ROOT))
    import torch.distributed as dist

    import bench

    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    ms = [12.5, 20.0][rank]
    got = bench.max_over_ranks(ms)
    dist.barrier()
    q.put((rank, got, bench.whole_job_rate(1000, world, got)))
    dist.destroy_process_group()


def test_two_rank_timing_is_max_and_value_is_whole_job():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = 29500 + (os.getpid() % 1000)
    ps = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in ps:
        p.start()
    res = sorted(q.get(timeout=120) for _ in ps)
    for p in ps:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, got, rate in res:
        assert got == 20.0
        assert rate == pytest.approx(2 * 1000 / 0.020)


def test_single_process_is_identity():
    sys.path.insert(0, str(ROOT))
    import bench

    assert bench.max_over_ranks(7.0) == 7.0
    assert bench.whole_job_rate(500, 1, 10.0) == pytest.approx(50_000)
