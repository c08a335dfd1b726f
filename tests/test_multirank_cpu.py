"""The multi-GPU benchmark path (independent replicas, max-over-ranks timing) on CPU:
two gloo ranks exercise the cross-rank logic of bench.py without a GPU."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench
from paper_2601_01513_gb300 import configs


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        cfg = configs.V7B
        seed = bench.replica_seed(cfg, rank)
        # rank r "measured" 100 + 10 r ms for the step loop and 200 - r ms end to end
        got = bench.max_over_ranks([100.0 + 10 * rank, 200.0 - rank], torch.device("cpu"))
        ws, r, local = bench.dist_env()
        q.put((rank, seed, got, (ws, r, local)))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_rank():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    mp.start_processes(_worker, args=(world, port, q), nprocs=world, join=True, start_method="spawn")
    res = sorted(q.get(timeout=60) for _ in range(world))
    seeds = [r[1] for r in res]
    assert len(set(seeds)) == world                       # independent replicas
    for rank, _, got, env in res:
        assert got == [110.0, 200.0]                      # max over ranks, per quantity
        assert env == (world, rank, rank)
    # whole-job throughput counts every rank's tokens over the slowest rank's time
    assert bench.job_throughput(80, 100, 2, 110.0) == pytest.approx(80 * 100 * 2 / 0.110)


def test_single_process_needs_no_collective():
    assert bench.max_over_ranks([3.0, 4.0], torch.device("cpu")) == [3.0, 4.0]
