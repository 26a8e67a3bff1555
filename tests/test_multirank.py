"""bench.py's multi-rank logic with two gloo ranks on the CPU.

Every rank condenses its own video (replicas); the job time is the slowest
rank's and the job value counts every rank's frames.
"""

import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    import bench
    import workload as wl
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms = 10.0 + 5.0 * rank                    # rank 1 is the slow one
        job_ms = bench.max_over_ranks(ms, world)
        spec = bench.replica_spec(wl.CONFIGS["video64_13x13_bf16"], rank)
        seeds = [None] * world
        dist.all_gather_object(seeds, spec.seed)
        out[rank] = (job_ms, bench.job_value(64, world, job_ms), seeds)
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks():
    world, port = 2, _free_port()
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_rank_main, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    for rank in range(world):
        job_ms, value, seeds = res[rank]
        assert job_ms == 15.0                      # max over ranks on every rank
        assert value == pytest.approx(2 * 64 / 0.015)
        assert len(set(seeds)) == world            # independent replicas


def test_single_rank_is_identity():
    import bench
    assert bench.max_over_ranks(3.5, 1) == 3.5
    assert bench.job_value(256, 1, 1.0) == pytest.approx(256000.0)
