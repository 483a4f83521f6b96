"""Seeded synthetic inputs for the k-means hot path.

This module draws random data only: Gaussian-mixture embeddings shaped like the
paper's workloads (unit-norm text/image embeddings, Table 2 of Section 4), Haar
random rotations used to build them, and Forgy initial-centroid indices
(Section 2.3, STEP 1: k points sampled at random).  It holds no step of the
clustering method itself (no projection, quantization, distance, assignment or
update), so both the CPU oracle and the CUDA path can take their inputs from it
without sharing any of the method's arithmetic.

Every function is deterministic in its seed.  Large arrays are generated on the
requested torch device in row chunks, so 10M x 1024 inputs never pass through
host memory unless the caller copies them.
"""
from __future__ import annotations

from dataclasses import dataclass

import torch

__all__ = [
    "WorkloadSpec",
    "WORKLOADS",
    "haar_rotation",
    "gmm_points",
    "forgy_indices",
    "workload_points",
]


@dataclass(frozen=True)
class WorkloadSpec:
    """Shape and recipe of one synthetic workload.

    n, d, k        points, dimensions, centroids
    n_comp         Gaussian-mixture components
    decay          True: per-dim variance (1+j)^-0.5, then a Haar rotation and
                   L2 normalisation (embedding-like); False: isotropic means
    std            within-component standard deviation (before the decay scaling)
    iters          Lloyd iterations
    """

    name: str
    n: int
    d: int
    k: int
    n_comp: int
    decay: bool
    std: float
    iters: int = 10


# The five workloads the hot path is specified on (points, dims, centroids,
# mixture components).  The 10M-point ones are generated on the GPU.
WORKLOADS = {
    "tiny_f32": WorkloadSpec("tiny_f32", 20_000, 128, 100, 100, False, 0.3),
    "emb1m_d768": WorkloadSpec("emb1m_d768", 1_000_000, 768, 1000, 2000, True, 0.3),
    "emb1m_d1024_sq8": WorkloadSpec("emb1m_d1024_sq8", 1_000_000, 1024, 1024, 2000, True, 0.3),
    "emb10m_d1024_rbq1": WorkloadSpec("emb10m_d1024_rbq1", 10_000_000, 1024, 3162, 10_000, True, 0.3),
    "emb10m_pca256": WorkloadSpec("emb10m_pca256", 10_000_000, 1024, 10_000, 10_000, True, 0.3),
}


def _generator(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def haar_rotation(d: int, seed: int) -> torch.Tensor:
    """Haar-distributed d x d orthogonal matrix (float64, CPU).

    QR of a seeded standard-Gaussian matrix with the signs of R's diagonal
    folded into Q (Mezzadri's construction), so the draw is uniform on O(d).
    """
    g = _generator(seed, "cpu")
    a = torch.randn(d, d, generator=g, dtype=torch.float64)
    q, r = torch.linalg.qr(a)
    sgn = torch.sign(torch.diagonal(r))
    sgn[sgn == 0] = 1.0
    return q * sgn.unsqueeze(0)


def gmm_points(
    n: int,
    d: int,
    n_comp: int,
    seed: int = 0,
    *,
    decay: bool = True,
    std: float = 0.3,
    device="cpu",
    chunk: int = 1 << 18,
    out: torch.Tensor | None = None,
) -> torch.Tensor:
    """Gaussian-mixture points, float32 [n, d], row-major.

    Component means mu_c ~ N(0, I_d); component of each point uniform over
    n_comp; point = mu_c + std * eps with eps ~ N(0, I_d).
    decay=True (embedding-like): the point is additionally scaled per dimension
    by sqrt(v_j), v_j = (1 + j)^-0.5, rotated by a Haar matrix (seed + 1) and
    L2-normalised.  Points are left in generation order (not grouped by
    component).
    """
    dev = torch.device(device)
    g = _generator(seed, dev)
    mu = torch.randn(n_comp, d, generator=g, device=dev, dtype=torch.float32)
    if decay:
        scale = torch.pow(torch.arange(d, device=dev, dtype=torch.float64) + 1.0, -0.25).to(torch.float32)
        rot_t = haar_rotation(d, seed + 1).to(dev, torch.float32).t().contiguous()
    if out is None:
        out = torch.empty(n, d, device=dev, dtype=torch.float32)
    for lo in range(0, n, chunk):
        hi = min(n, lo + chunk)
        comp = torch.randint(0, n_comp, (hi - lo,), generator=g, device=dev)
        eps = torch.randn(hi - lo, d, generator=g, device=dev, dtype=torch.float32)
        x = mu.index_select(0, comp) + std * eps
        if decay:
            x = (x * scale) @ rot_t
            x = x / torch.linalg.vector_norm(x, dim=1, keepdim=True).clamp_min(1e-30)
        out[lo:hi].copy_(x)
    return out


def hadamard_signs(D: int, seed: int) -> torch.Tensor:
    """Seeded +-1 vector of length D (float32, CPU) for a randomized Hadamard
    rotation."""
    g = _generator(seed + 3, "cpu")
    return (torch.randint(0, 2, (D,), generator=g) * 2 - 1).to(torch.float32)


def forgy_indices(n: int, k: int, seed: int) -> torch.Tensor:
    """First k entries of a seeded uniform permutation of range(n) (int64, CPU)."""
    g = _generator(seed + 2, "cpu")
    return torch.randperm(n, generator=g)[:k].clone()


def workload_points(spec: WorkloadSpec, seed: int = 0, device="cpu", n: int | None = None) -> torch.Tensor:
    """Points of a named workload (optionally only the first n rows' recipe at a smaller n)."""
    return gmm_points(
        spec.n if n is None else n,
        spec.d,
        spec.n_comp,
        seed,
        decay=spec.decay,
        std=spec.std,
        device=device,
    )

