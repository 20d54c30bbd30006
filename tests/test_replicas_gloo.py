"""bench.py's multi-replica path (one independent replica per rank, weak
scaling) on 2 CPU ranks over gloo: whole-job tokens are summed over ranks and
divided by the slowest rank's time."""

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


def _worker(rank, world, port, results):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench

    tokens = 1000.0 * (rank + 1)     # each replica its own batch size
    ms = 250.0 + 50.0 * rank         # rank 1 is the slower one
    total, ms_max, value = bench.aggregate(tokens, ms, world, device="cpu")
    results[rank] = (total, ms_max, value)
    dist.barrier()
    dist.destroy_process_group()


def test_two_replicas_weak_scaling_aggregate():
    world = 2
    port = _free_port()
    with mp.Manager() as m:
        results = m.dict()
        mp.spawn(_worker, args=(world, port, results), nprocs=world, join=True)
        res = dict(results)
    for rank in range(world):
        total, ms_max, value = res[rank]
        assert total == 3000.0 and ms_max == 300.0
        assert value == pytest.approx(3000.0 / 0.3)


def test_single_rank_is_identity():
    import bench

    assert bench.aggregate(128.0, 500.0, 1) == (128.0, 500.0, 256.0)
