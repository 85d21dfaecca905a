"""The N > 1 bench path: independent replicas with host-side max-over-ranks
timing, run as two gloo ranks on the CPU."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2605_24793_gb300 import replicas, workload


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        w, r, lr = replicas.env_ranks()
        assert (w, r, lr) == (world, rank, rank)
        # each replica draws the identical workload from the same seeds
        inp = workload.make_round_inputs(workload.CONFIGS["tiny"], device="cpu")
        mine = inp["q"].float().sum().item() + inp["w"].float().sum().item()
        sums = [None] * world
        dist.all_gather_object(sums, mine)
        # the slowest rank bounds the job
        elapsed = 0.25 + 0.5 * rank
        m = replicas.max_over_ranks(elapsed, dist)
        out[rank] = (sums, m, replicas.job_throughput(30.0, m, world))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_gloo_replicas_share_workload_and_take_the_slowest_time():
    world = 2
    mgr = mp.get_context("spawn").Manager()
    out = mgr.dict()
    mp.start_processes(_worker, args=(world, _free_port(), out), nprocs=world, start_method="spawn")
    for rank in range(world):
        sums, m, thr = out[rank]
        assert sums[0] == sums[1]
        assert m == pytest.approx(0.75)
        assert thr == pytest.approx(2 * 30.0 / 0.75)


def test_single_process_needs_no_group():
    assert replicas.max_over_ranks(1.5) == 1.5
    assert replicas.job_throughput(6, 0.5, 1) == 12.0


def test_reference_arm_runs_on_rank_zero_only(monkeypatch):
    import bench
    monkeypatch.setenv("RANK", "1")
    called = []
    monkeypatch.setattr(bench.W, "make_round_inputs", lambda *a, **k: called.append(1))
    args = type("A", (), dict(config="tiny", steps=1, warmup=0, gpus=2))()
    assert bench.run_reference(args) is None
    assert not called
