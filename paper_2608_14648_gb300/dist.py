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


def global_mean_fixed(amax_local: float, n_local: int, column_sums, mean_from_sums, device):
    """The RabitQ dataset mean over all ranks' rows, the same bits as one
    process computing it over all rows: the maximum of the ranks' max |x|
    and the total row count give the fixed-point scale s (skm_mean_scale);
    each rank's exact int64 column sums at that scale (column_sums(s)) are
    summed over the ranks; mean_from_sums(S, n_total, s) finishes.  The two
    callables carry the arithmetic (libskm on the GPU)."""
    import paper_2608_14648_gb300 as skm

    mx = torch.tensor([float(amax_local)], dtype=torch.float32, device=device)
    cnt = torch.tensor([int(n_local)], dtype=torch.int64, device=device)
    dist.all_reduce(mx, op=dist.ReduceOp.MAX)
    dist.all_reduce(cnt, op=dist.ReduceOp.SUM)
    n_total = int(cnt.item())
    s = skm.skm_mean_scale(float(mx.item()), n_total)
    S = column_sums(s)
    dist.all_reduce(S, op=dist.ReduceOp.SUM)
    return mean_from_sums(S, n_total, s)


def global_rbq1_mean(X: torch.Tensor) -> torch.Tensor:
    """global_mean_fixed with libskm's kernels on this rank's rows X (device float32 [n, d])."""
    import paper_2608_14648_gb300 as skm

    def sums(s):
        S = torch.zeros(X.shape[1], dtype=torch.int64, device=X.device)
        return skm.skm_column_sums_fixed(X, s, S)

    return global_mean_fixed(skm.skm_column_absmax(X), X.shape[0], sums,
                             lambda S, n, s: skm.skm_mean_from_sums(S, n, s), X.device)


def global_exponent(local_e: int, device) -> int:
    """Fixed-point exponent for the global maximum F: the minimum of the ranks' exponents."""
    t = torch.tensor([int(local_e)], dtype=torch.int64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MIN)
    return int(t.item())
