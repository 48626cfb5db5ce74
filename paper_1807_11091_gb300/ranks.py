"""Host-side logic of the multi-GPU path (one process per GPU under torchrun).

The pruned layer shards by batch: every rank runs the same per-GPU batch of its
own synthetic images through its own plan, with no collective on the data path
(weak scaling).  The only cross-rank step is the timing: each rank's total of
the timed steps is reduced with MAX, and the job's throughput counts the work of
all ranks over that time.  Rank 0 alone reports.
"""
from __future__ import annotations

import os
from typing import Tuple


def dist_env() -> Tuple[int, int, int]:
    """(world size, rank, local rank) from the torchrun environment."""
    return (int(os.environ.get("WORLD_SIZE", "1")), int(os.environ.get("RANK", "0")),
            int(os.environ.get("LOCAL_RANK", "0")))


def shard_seed(seed: int, rank: int) -> int:
    """Seed of a rank's synthetic batch: distinct images per rank, same shapes."""
    return int(seed) + 1000 * int(rank)


def max_over_ranks(value: float, device=None) -> float:
    """The largest of every rank's value (all ranks must call; returns value
    unchanged when torch.distributed is not initialised)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(work_per_step_per_rank: float, world_size: int, steps: int, max_total_ms: float) -> float:
    """Whole-job throughput in work units per second: every rank's work over the
    slowest rank's time."""
    return work_per_step_per_rank * world_size * steps / (max_total_ms * 1e-3)


def reports(rank: int) -> bool:
    """Only rank 0 prints the result line."""
    return int(rank) == 0
