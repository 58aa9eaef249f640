"""Host-side logic of multi-GPU runs: one process per GPU, launched by torchrun.

The single-matrix path does not shard: its pivot chain runs down the diagonal one
column after the other, so N GPUs run N independent replicas (weak scaling).  A
batch of independent matrices is split into contiguous shards, one per rank, with
no collective on the data path.  The only collectives are for the measurement:
the maximum over ranks of a step time and sums of counted work.
"""
from __future__ import annotations

import os


def rank_info(env=None) -> tuple[int, int, int]:
    """(rank, world_size, local_rank) from the torchrun environment (1 process by default)."""
    env = os.environ if env is None else env
    return int(env.get("RANK", "0")), int(env.get("WORLD_SIZE", "1")), int(env.get("LOCAL_RANK", "0"))


def shard_range(batch: int, rank: int, world: int) -> tuple[int, int]:
    """Contiguous shard [b0, b1) of a batch for one rank; shard sizes differ by at most one
    and the shards of all ranks partition [0, batch) in rank order."""
    if world < 1 or not 0 <= rank < world or batch < 0:
        raise ValueError("bad shard request")
    return batch * rank // world, batch * (rank + 1) // world


def _reduce(value: float, op_name: str, device=None) -> float:
    import torch
    import torch.distributed as dist

    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=getattr(dist.ReduceOp, op_name))
    return float(t.item())


def max_over_ranks(value: float, device=None) -> float:
    """Largest value over all ranks (the job's time is its slowest rank's)."""
    return _reduce(value, "MAX", device)


def sum_over_ranks(value: float, device=None) -> float:
    """Sum over all ranks (work counted on each rank)."""
    return _reduce(value, "SUM", device)


def job_throughput(total_units: float, max_time_s: float) -> float:
    """Whole-job throughput: the units all ranks processed over the slowest rank's time."""
    if max_time_s <= 0:
        raise ValueError("non-positive time")
    return total_units / max_time_s
