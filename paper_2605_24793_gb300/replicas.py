"""Multi-GPU runs of the round: independent replicas, one process per GPU.

Every sequence's round is independent of every other's (the paper's rounds
share nothing across requests), so N GPUs run N copies of the workload with
no collective on the data path.  The only cross-rank steps are host-side
bookkeeping: a barrier around the timed region and the maximum of the ranks'
elapsed times, from which the whole-job throughput follows.
"""
from __future__ import annotations

import os
from typing import Optional, Tuple

import torch


def env_ranks() -> Tuple[int, int, int]:
    """(world_size, rank, local_rank) from the torchrun environment."""
    return (int(os.environ.get("WORLD_SIZE", "1")), int(os.environ.get("RANK", "0")),
            int(os.environ.get("LOCAL_RANK", "0")))


def max_over_ranks(value: float, dist=None, device: Optional[torch.device] = None) -> float:
    """Largest `value` over all ranks (the slowest rank bounds the job)."""
    if dist is None or not dist.is_initialized() or dist.get_world_size() == 1:
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device or "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(units_per_rank: float, max_seconds: float, world: int) -> float:
    """Whole-job rate: every rank processed `units_per_rank` in at most `max_seconds`."""
    return world * units_per_rank / max_seconds
