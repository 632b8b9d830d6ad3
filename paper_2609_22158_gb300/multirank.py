"""Host-side logic for running the compression pass on several GPUs (one process per GPU).

The pass partitions by trajectory: every trajectory is an independent problem (its own cache, steps and
budget), so ranks share nothing on the data path.  What the ranks do exchange is timing only: a barrier
before and after the timed region and the maximum step time over ranks.  These helpers hold that logic
so it can be exercised with the gloo backend on CPU.
"""
from __future__ import annotations

import os
from typing import List, Sequence, Tuple


def rank_env() -> Tuple[int, int, int]:
    """(world size, rank, local rank) from the torchrun environment; (1, 0, 0) when run directly."""
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", str(rank)))
    if world < 1 or not (0 <= rank < world):
        raise ValueError(f"invalid rank {rank} for world size {world}")
    return world, rank, local


def shard(n_items: int, world: int, rank: int) -> range:
    """Contiguous share of n_items independent trajectories for `rank`: sizes differ by at most one and
    the shares of all ranks cover every item exactly once, in order."""
    if world < 1 or not (0 <= rank < world):
        raise ValueError(f"invalid rank {rank} for world size {world}")
    base, extra = divmod(max(n_items, 0), world)
    lo = rank * base + min(rank, extra)
    return range(lo, lo + base + (1 if rank < extra else 0))


def rank_seed(base_seed: int, rank: int) -> int:
    """Seed of the per-rank random tensors, so ranks compress different (but equally shaped) inputs."""
    return base_seed + 7919 * rank


def max_over_ranks(value: float, dist=None, device=None) -> float:
    """The largest `value` over all ranks (the job's step time is its slowest rank's)."""
    if dist is None or not dist.is_initialized() or dist.get_world_size() == 1:
        return float(value)
    import torch
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(tokens_per_rank: Sequence[int], step_seconds: float) -> float:
    """Whole-job tokens per second: every rank's tokens over the slowest rank's time."""
    if step_seconds <= 0:
        raise ValueError("step time must be positive")
    return float(sum(tokens_per_rank)) / step_seconds


def gather_tokens(tokens: int, dist=None, device=None) -> List[int]:
    """Tokens each rank processes per step (rank order)."""
    if dist is None or not dist.is_initialized() or dist.get_world_size() == 1:
        return [int(tokens)]
    import torch
    t = torch.tensor([int(tokens)], dtype=torch.int64, device=device)
    out = [torch.zeros_like(t) for _ in range(dist.get_world_size())]
    dist.all_gather(out, t)
    return [int(x.item()) for x in out]
