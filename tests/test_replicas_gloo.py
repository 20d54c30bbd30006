"""bench.py's multi-rank path on 2 CPU ranks over gloo: whole-job tokens are
summed over ranks and divided by the slowest rank's time (weak scaling), and
the backward's data-parallel exchange leaves every rank with the sum of the
ranks' grad_w."""

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
    with mp.get_context("spawn").Manager() as m:  # no fork of this multi-threaded process
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


def _allreduce_worker(rank, world, port, results):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench

    g = torch.Generator().manual_seed(rank)
    gw = torch.randn(7, 5, generator=g)      # this rank's grad_w of its own batch
    mine = gw.clone()
    out = bench.dp_grad_w_allreduce(gw, world)
    assert out is gw                          # in place, as the step's buffer
    results[rank] = (mine.tolist(), gw.tolist())
    dist.barrier()
    dist.destroy_process_group()


def test_grad_w_allreduce_sums_over_ranks():
    world = 2
    port = _free_port()
    with mp.get_context("spawn").Manager() as m:  # no fork of this multi-threaded process
        results = m.dict()
        mp.spawn(_allreduce_worker, args=(world, port, results), nprocs=world, join=True)
        res = dict(results)
    want = sum(torch.tensor(res[r][0]) for r in range(world))
    for r in range(world):
        torch.testing.assert_close(torch.tensor(res[r][1]), want)


def test_grad_w_allreduce_single_rank_is_identity():
    import bench

    gw = torch.randn(3, 4)
    ref = gw.clone()
    assert torch.equal(bench.dp_grad_w_allreduce(gw, 1), ref)
