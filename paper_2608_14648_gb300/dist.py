"""Data-parallel glue for running the Lloyd iteration on several GPUs.

Rows are sharded across ranks; every rank holds the same centroids.  The one
exchange per iteration is the sum of the update's partial cluster sums and
member counts (skm_update with `partial`), after which every rank finalises
the same centroids (skm_update_finalize).  Integer partials (SQ8, RBQ1) make
the merged result independent of the number of ranks.  The RBQ1 encoding
also needs the global mean and the global fixed-point exponent.

Only torch.distributed collectives are used here; the arithmetic stays in
libskm.
"""
from __future__ import annotations

import torch
import torch.distributed as dist


def shard_bounds(n: int, rank: int, world: int) -> tuple[int, int]:
    """Contiguous, balanced row range [lo, hi) of `rank` among `world` ranks."""
    base, extra = divmod(n, world)
    lo = rank * base + min(rank, extra)
    hi = lo + base + (1 if rank < extra else 0)
    return lo, hi


def allreduce_partials(partial: torch.Tensor, counts: torch.Tensor) -> None:
    """Sum the update's partial cluster sums and member counts over ranks (in place)."""
    dist.all_reduce(partial, op=dist.ReduceOp.SUM)
    dist.all_reduce(counts, op=dist.ReduceOp.SUM)


def global_mean(local_sum: torch.Tensor, local_n: int) -> torch.Tensor:
    """Dataset mean from per-rank column sums (fp64) and row counts."""
    s = local_sum.to(torch.float64).clone()
    cnt = torch.tensor([float(local_n)], dtype=torch.float64, device=s.device)
    dist.all_reduce(s, op=dist.ReduceOp.SUM)
    dist.all_reduce(cnt, op=dist.ReduceOp.SUM)
    return (s / cnt).to(torch.float32)


def global_exponent(local_e: int, device) -> int:
    """Fixed-point exponent for the global maximum F: the minimum of the ranks' exponents."""
    t = torch.tensor([int(local_e)], dtype=torch.int64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MIN)
    return int(t.item())
