"""The multi-rank leg of bench.py on CPU: world_size 2 over gloo.

With N GPUs bench.py runs N independent replicas of the workload (the
simulated workers share nothing across GPUs), times each, and reports the
whole-job rate over the slowest rank's time.  Here two gloo ranks on the host
exercise that aggregation; no GPU is touched."""
from __future__ import annotations

import os
import socket

import pytest

torch = pytest.importorskip("torch")


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank: int, world: int, port: int, results):
    import torch.distributed as tdist

    import bench

    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    tdist.init_process_group("gloo", rank=rank, world_size=world)
    local_ms = 100.0 + 50.0 * rank  # rank 1 is the slow one
    slowest = bench.max_over_ranks(local_ms, world)
    value = bench.whole_job_rate(units_per_rank=1000, steps=10, world=world, max_ms=slowest)
    tdist.barrier()
    tdist.destroy_process_group()
    results[rank] = (slowest, value, bench.dist_env())


def test_two_gloo_ranks_report_the_slowest_time():
    import multiprocessing as mp

    ctx = mp.get_context("spawn")
    port = _free_port()
    with ctx.Manager() as mgr:
        results = mgr.dict()
        procs = [ctx.Process(target=_rank_main, args=(r, 2, port, results)) for r in range(2)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(timeout=120)
            assert p.exitcode == 0
        res = dict(results)
    for rank in range(2):
        slowest, value, env = res[rank]
        assert slowest == 150.0
        assert value == pytest.approx(2 * 1000 * 10 / 0.150)
        assert env == (rank, 2, rank)


def test_single_rank_is_unchanged():
    import bench
    assert bench.max_over_ranks(12.5, 1) == 12.5
    assert bench.whole_job_rate(10, 4, 1, 2.0) == pytest.approx(20000.0)
