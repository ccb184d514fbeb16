"""Host logic for running boundary compression on several GPUs of one node.

Boundaries (images) are independent and the method has no exchange step, so
every rank runs its own replica of the path on its own GPU ("replicas only",
no collective on the data path).  The only cross-rank operations are the
benchmark's bookkeeping: a barrier around the timed region, the maximum of
the ranks' step times, and the whole-job rate.  A batch of images can also be
split over the ranks, image by image.
"""

from __future__ import annotations


def rank_info(env=None) -> tuple[int, int, int]:
    """(rank, world size, local rank) from the torchrun environment (1 process if unset)."""
    import os
    env = os.environ if env is None else env
    return int(env.get("RANK", "0")), int(env.get("WORLD_SIZE", "1")), int(env.get("LOCAL_RANK", "0"))


def max_over_ranks(value: float, device=None) -> float:
    """The largest of every rank's value (the slowest rank sets the step time)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(world: int, units_per_rank: int, step_ms: float) -> float:
    """Whole-job units per second: every rank processes units_per_rank per step."""
    if step_ms <= 0:
        raise ValueError("step time must be positive")
    return world * units_per_rank * 1000.0 / step_ms


def shard_images(B: int, rank: int, world: int) -> list[int]:
    """Images of a batch that this rank compresses: a contiguous, balanced block
    (sizes differ by at most one; every image goes to exactly one rank)."""
    if not 0 <= rank < world:
        raise ValueError("rank out of range")
    lo = rank * B // world
    hi = (rank + 1) * B // world
    return list(range(lo, hi))
