"""Multi-GPU runs are replicas (independent requests per rank, no data-path
collective): the benchmark takes the slowest rank's step time and counts
every rank's units.  Exercised here with world_size 2 on the gloo backend."""

import os

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _rank(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms = 2.0 + rank  # rank 1 is the slow one
        slowest = bench.reduce_step_time(ms, world, torch.device("cpu"))
        out[rank] = (slowest, bench.job_throughput(112, world, slowest))
    finally:
        dist.destroy_process_group()


def test_replicas_use_the_slowest_rank():
    world = 2
    port = 29500 + (os.getpid() % 2000)
    # the result dict's server process is spawned too: nothing is forked
    out = mp.get_context("spawn").Manager().dict()
    mp.spawn(_rank, args=(world, port, out), nprocs=world, join=True)
    assert out[0] == out[1]
    slowest, value = out[0]
    assert slowest == 3.0
    assert value == pytest.approx(2 * 112 / 3e-3)


def test_single_rank_is_unchanged():
    assert bench.reduce_step_time(1.5, 1, None) == 1.5
    assert bench.job_throughput(448, 1, 2.0) == pytest.approx(224000.0)
