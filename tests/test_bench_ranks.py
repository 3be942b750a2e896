"""The multi-rank bookkeeping of bench.py on CPU: two gloo ranks, each with its own timing, combine into the
slowest rank's time and the whole job's throughput (replicas: every rank serves its own batches)."""
import os
import socket

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, results):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # rank r took (r + 1) * 100 ms for its steps and (r + 1) * 2 s end to end
        job = bench.combine_ranks(100.0 * (rank + 1), 2.0 * (rank + 1), world, steps=50, e2e_steps=10, batch=32)
        results[rank] = job
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world", [2])
def test_ranks_combine_to_slowest_time_and_total_queries(world):
    ctx = mp.get_context("spawn")
    with ctx.Manager() as mgr:
        results = mgr.dict()
        port = _free_port()
        procs = [ctx.Process(target=_rank, args=(r, world, port, results)) for r in range(world)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(120)
            assert p.exitcode == 0
        res = dict(results)
    for r in range(world):
        job = res[r]
        assert job["elapsed_ms"] == 100.0 * world and job["e2e_s"] == 2.0 * world
        assert job["value"] == pytest.approx(world * 50 * 32 / (0.1 * world))
        assert job["e2e_value"] == pytest.approx(world * 10 * 32 / (2.0 * world))


def test_single_rank_needs_no_process_group():
    job = bench.combine_ranks(200.0, 4.0, 1, steps=100, e2e_steps=20, batch=64)
    assert job["value"] == pytest.approx(100 * 64 / 0.2) and job["e2e_value"] == pytest.approx(20 * 64 / 4.0)
