"""The multi-GPU path of bench.py on CPU: two gloo ranks check the
slowest-rank timing and the whole-job (weak-scaling) throughput."""
from __future__ import annotations

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
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        ms_local = 10.0 + 5.0 * rank                 # rank 1 is the slow one
        ms_max = bench.max_over_ranks(ms_local)
        value = bench.job_throughput(world, 7, ms_max)
        out[rank] = (ms_max, value)
    finally:
        dist.destroy_process_group()


@pytest.mark.timeout(120)
def test_two_rank_max_and_weak_scaling():
    world = 2
    port = _free_port()
    with mp.Manager() as mgr:
        out = mgr.dict()
        mp.start_processes(_worker, args=(world, port, out), nprocs=world, start_method="spawn", join=True)
        res = dict(out)
    import bench
    per_rank = 7 * bench.L * bench.B * bench.H * bench.T
    for rank in range(world):
        ms_max, value = res[rank]
        assert ms_max == 15.0                       # every rank sees the slowest rank's time
        assert value == pytest.approx(world * per_rank / 15e-3)


def test_single_process_is_identity():
    import bench
    assert bench.max_over_ranks(3.5) == 3.5
    assert bench.job_throughput(1, 2, 1000.0) == pytest.approx(2 * bench.L * bench.B * bench.H * bench.T)
