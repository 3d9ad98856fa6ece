"""Multi-rank host logic of bench.py on CPU (gloo, world size 2): each rank
times its own replica of the round; the job reports the slowest rank's step
time and the units all ranks processed.  No GPU is used."""
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


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port),
                      RANK=str(rank), WORLD_SIZE=str(world))
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        w, r, _ = bench.dist_env()
        assert (w, r) == (world, rank)
        # rank 1 is the slow one
        ms = 2.0 if rank == 0 else 3.5
        worst = bench.reduce_max(ms, world)
        value = bench.job_value(1.0, worst / 1e3, world)
        out[rank] = (worst, value)
    finally:
        dist.destroy_process_group()


def test_two_rank_job_takes_slowest_rank_and_total_units():
    world, port = 2, _free_port()
    out = mp.Manager().dict()
    mp.spawn(_worker, args=(world, port, out), nprocs=world, join=True)
    for rank in range(world):
        worst, value = out[rank]
        assert worst == 3.5
        assert value == pytest.approx(2 / 3.5e-3)


def test_single_rank_is_identity():
    import bench
    assert bench.reduce_max(1.25, 1) == 1.25
    assert bench.job_value(1.0, 0.002, 1) == pytest.approx(500.0)
