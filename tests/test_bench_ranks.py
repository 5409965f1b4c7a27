"""The benchmark's multi-rank path on CPU: two gloo ranks, each an independent
replica (chains are independent, Eq. 11, so ranks exchange nothing on the data
path); the job rate is every rank's tokens over the slowest rank's time."""
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
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    ms_local = 100.0 + 50.0 * rank          # rank 1 is the slow one
    ms, rate = bench.job_rate(ms_local, tokens_per_rank=131072, world=world)
    out[rank] = (ms, rate)
    dist.barrier()
    dist.destroy_process_group()


def test_job_rate_takes_the_slowest_rank_and_all_tokens():
    world = 2
    mgr = mp.Manager()
    out = mgr.dict()
    mp.spawn(_rank_main, args=(world, _free_port(), out), nprocs=world, join=True)
    for rank in range(world):
        ms, rate = out[rank]
        assert ms == 150.0
        assert rate == pytest.approx(world * 131072 / 0.150)


def test_job_rate_single_process():
    import bench
    ms, rate = bench.job_rate(50.0, 1000, 1)
    assert ms == 50.0 and rate == pytest.approx(20000.0)
