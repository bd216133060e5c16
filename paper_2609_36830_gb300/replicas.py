"""Host-side logic of multi-GPU runs: one process per GPU, each running an
independent replica of the PACE step on its own pool.

The path has no exchange step between replicas (each trainer replica admits
from its own pool), so a job of N ranks is N weak-scaled replicas: distinct
seeds per rank, a barrier around the timed region, the maximum of the ranks'
step times as the job's time, and the sum of the ranks' rows as the job's work.
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
    """Seed of rank's pool: rank 0 draws the workload's default pool."""
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
