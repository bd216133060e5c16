"""Host-side helpers of multi-GPU runs (one process per GPU): the launcher's
rank environment, the seed of each rank's part of the pool, and the job's
totals.

A data-parallel step (sharded.ShardedPaceStep) partitions the pool by prompt
group: rank r draws its groups with its own seed, and the whole pool is the
union of the ranks' parts.  The job's work is the sum of the ranks' rows in the
loss and its time the slowest rank's, with a barrier around the timed region.
"""
from __future__ import annotations

import os
from typing import Tuple

from . import workloads


def rank_env() -> Tuple[int, int, int]:
    """(world_size, rank, local_rank) from the torch.distributed launcher's environment."""
    return (int(os.environ.get("WORLD_SIZE", "1")), int(os.environ.get("RANK", "0")),
            int(os.environ.get("LOCAL_RANK", "0")))


def replica_seed(workload: str, rank: int) -> int:
    """Seed of rank's part of the pool: rank 0 draws the workload's default pool."""
    return workloads.SEED_BASE + workloads.SPECS[workload].index + 1000 * rank


def job_totals(local_rows: int, local_ms: float, device="cpu") -> Tuple[int, float]:
    """(rows over all ranks, slowest rank's milliseconds); identity without a process group."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return int(local_rows), float(local_ms)
    rows = torch.tensor([float(local_rows)], dtype=torch.float64, device=device)
    ms = torch.tensor([float(local_ms)], dtype=torch.float64, device=device)
    dist.all_reduce(rows, op=dist.ReduceOp.SUM)
    dist.all_reduce(ms, op=dist.ReduceOp.MAX)
    return int(rows.item()), float(ms.item())
