"""Host logic of running the verification pass as independent replicas, one
process per GPU (the pass of one sequence does not shard across GPUs here).

Each rank runs its own steps; a step's time for the whole job is the slowest
rank's, and the job's throughput is the units all ranks processed over that
time (weak scaling: per-GPU work is fixed as ranks are added)."""
from __future__ import annotations

import os


def dist_info():
    """(world_size, rank, local_rank) from the torchrun environment."""
    return (int(os.environ.get("WORLD_SIZE", "1")), int(os.environ.get("RANK", "0")),
            int(os.environ.get("LOCAL_RANK", "0")))


def max_over_ranks(value: float, device=None) -> float:
    """The largest `value` over all ranks of the default process group (or
    `value` itself without one)."""
    import torch
    import torch.distributed as dist

    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(units_per_rank: float, slowest_seconds: float, world: int) -> float:
    """Units processed by all ranks per second of the slowest rank."""
    if slowest_seconds <= 0:
        raise ValueError("elapsed time must be positive")
    return world * units_per_rank / slowest_seconds
