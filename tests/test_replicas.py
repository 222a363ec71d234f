"""Multi-GPU path of the benchmark on CPU: the path shards over sequences with no exchange step,
so N GPUs run N independent replicas; the job time is the slowest rank's and the throughput is
every rank's drafted tokens over that time (weak scaling). Checked with two gloo ranks."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms_local = 10.0 * (rank + 1)          # rank 1 is the slow one
        ms, value = bench.replica_aggregate(ms_local, units_per_step=15, steps=100, dist=dist, device="cpu")
        out[rank] = (ms, value)
    finally:
        dist.destroy_process_group()


def test_two_replicas_aggregate_max_time_and_total_units():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    with ctx.Manager() as m:
        out = m.dict()
        mp.start_processes(_rank, args=(world, port, out), nprocs=world, join=True, start_method="spawn")
        res = dict(out)
    for r in range(world):
        ms, value = res[r]
        assert ms == pytest.approx(20.0)                       # max over ranks
        assert value == pytest.approx(world * 15 * 100 / 0.020)  # all ranks' units / job time


def test_single_process_aggregate_is_local():
    ms, value = bench.replica_aggregate(12.5, units_per_step=15, steps=40)
    assert ms == 12.5 and value == pytest.approx(15 * 40 / 0.0125)
