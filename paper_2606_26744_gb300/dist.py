"""Host-side helpers for running the draft step on several GPUs.

The path has no exchange step: the reducer is independent per token and the
drafter, LM head and verification are independent per sequence.  N GPUs are
therefore N replicas, each drafting its own sequences (or its own slice of
tokens); the only collective is the timing reduction (max over ranks).
"""
from __future__ import annotations

from typing import List, Sequence, Tuple

import torch


def rank_seed(base: int, rank: int) -> int:
    """Seed of the synthetic inputs of one rank (distinct sequences per rank)."""
    return base + 17 * rank


def shard(n: int, rank: int, world: int) -> Tuple[int, int]:
    """Contiguous [lo, hi) share of n units for rank (sizes differ by <= 1)."""
    if world <= 0 or not 0 <= rank < world:
        raise ValueError("bad rank/world")
    lo = n * rank // world
    hi = n * (rank + 1) // world
    return lo, hi


def max_over_ranks(values: Sequence[float], device=None) -> List[float]:
    """Element-wise maximum over all ranks (identity without a process group)."""
    if not (torch.distributed.is_available() and torch.distributed.is_initialized()):
        return [float(v) for v in values]
    t = torch.tensor([float(v) for v in values], dtype=torch.float64,
                     device=device if device is not None else "cpu")
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return [float(v) for v in t.tolist()]


def whole_job_rate(units_per_rank: int, world: int, ms_per_step_max: float) -> float:
    """Whole-job throughput of N replicas in units per second: every rank
    processes units_per_rank units per step, and the job's step takes the
    slowest rank's time (ms_per_step_max, the max over ranks)."""
    if world <= 0 or ms_per_step_max <= 0:
        raise ValueError("world and step time must be positive")
    return units_per_rank * world / (ms_per_step_max / 1e3)
