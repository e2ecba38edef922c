"""Multi-process helpers (one process per GPU).

Layers and channels are independent and nothing on the quantization path exchanges data, so N GPUs
run N independent replicas of a workload (weak scaling) with no collective on the data path.  The
only collectives are for measurement: a barrier around the timed region and the maximum of the
ranks' step times, so the aggregate throughput is (units of all ranks) / (slowest rank's time).
"""
from __future__ import annotations

import os

import torch
import torch.distributed as dist


def world_from_env():
    """(world_size, rank, local_rank) from the torchrun environment (1, 0, 0 when absent)."""
    return (int(os.environ.get("WORLD_SIZE", "1")), int(os.environ.get("RANK", "0")),
            int(os.environ.get("LOCAL_RANK", "0")))


def max_over_ranks(x: float, device=None) -> float:
    """Maximum of a float over all ranks (identity without an initialised process group)."""
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device or "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def aggregate_throughput(units_per_rank: float, ms_per_step_max: float, world: int) -> float:
    """Whole-job units per second: every rank processes its own replica of the workload."""
    return units_per_rank * world / (ms_per_step_max / 1e3)


def shard(n: int, world: int, rank: int):
    """Contiguous [begin, end) share of n independent items for one rank (for callers that split
    one network's layers or channels across GPUs instead of replicating it)."""
    base, rem = divmod(n, world)
    begin = rank * base + min(rank, rem)
    return begin, begin + base + (1 if rank < rem else 0)
