"""Host logic of the multi-GPU benchmark, on CPU with two gloo ranks.

The step partitions by task (each task owns its router, experts and tokens), so
with N GPUs every rank runs its own workload and the only exchange is the barrier
and the max over ranks of the timed region.  These tests run that logic as two
real processes over gloo (127.0.0.1) without any GPU.
"""
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


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        local = [10.0 + rank, 3.0 - rank]  # rank 1 slower on the first, faster on the second
        res = bench.max_over_ranks(local, dist)
        dist.barrier()
        out[rank] = (res, bench.rank_weight_seed(rank))
    finally:
        dist.destroy_process_group()


def test_max_over_two_gloo_ranks():
    world = 2
    port = _free_port()
    with mp.Manager() as mgr:
        out = mgr.dict()
        mp.start_processes(_rank_main, args=(world, port, out), nprocs=world, join=True,
                           start_method="spawn")
        res = dict(out)
    assert res[0][0] == [11.0, 3.0] and res[1][0] == [11.0, 3.0]
    assert res[0][1] != res[1][1]  # independent experts per rank


def test_weak_scaling_throughput_formula():
    # 17 tasks x 1576 tokens per rank, 4 ranks, 3 ms per step
    v = bench.job_tokens_per_s(17 * 1576, 4, 3.0)
    assert v == pytest.approx(17 * 1576 * 4 / 3e-3)
    assert bench.max_over_ranks([1.0, 2.0]) == [1.0, 2.0]  # no process group: identity
