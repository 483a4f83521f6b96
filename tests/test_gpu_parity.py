"""GPU path vs the CPU oracle, element by element, through the C ABI.

Integer paths (SQ8 codes/distances/assignments/centroids, RBQ1 estimates,
assignments and centroids given identical codes) must be bit-exact; the fp32
and bf16 paths must agree on >= 99.9% of assignments with every disagreement
at an oracle top-2 relative gap <= 1e-5, centroids within 1e-4 relative L2
given identical assignments, objectives within 1e-4 relative."""
import ctypes
import math

import numpy as np
import pytest
import torch

import oracle
import synth

pytestmark = pytest.mark.gpu

GAP_TOL = 1e-5
AGREE = 0.999


@pytest.fixture(scope="module")
def skm(cuda_ok):
    import paper_2608_14648_gb300 as skm

    skm.lib()
    return skm


DEV = "cuda"


def _points(n, d, seed, decay=True, ncomp=40):
    return synth.gmm_points(n, d, ncomp, seed=seed, decay=decay)


def _check_f32(a_gpu, dist_gpu, best, second, a_or, what):
    a_gpu = np.asarray(a_gpu)
    agree = a_gpu == a_or
    frac = agree.mean()
    assert frac >= AGREE, f"{what}: agreement {frac}"
    if not agree.all():
        gap = (second - best) / np.maximum(best, 1e-30)
        assert np.all(gap[~agree] <= GAP_TOL), f"{what}: disagreement at gap {gap[~agree].max()}"
    if dist_gpu is not None:
        d = np.asarray(dist_gpu)
        np.testing.assert_allclose(d[agree], best[agree], rtol=2e-5, atol=1e-6)


# ----------------------------------------------------------------- fp32 path
@pytest.mark.parametrize("n,d,k", [(1000, 128, 100), (777, 33, 7), (3001, 768, 300), (200, 1, 5),
                                   (513, 64, 257), (64, 200, 64)])
def test_assign_f32_vs_oracle(skm, n, d, k):
    X = _points(n, d, seed=n + d)
    idx = synth.forgy_indices(n, k, seed=d)
    C = X[idx].clone()
    C += 0.01 * torch.randn(C.shape, generator=torch.Generator().manual_seed(1))
    pts = skm.Points(skm.REPR_F32, X.to(DEV), d)
    a, dist = skm.skm_assign(pts, C.to(DEV))
    a_or, best, second = oracle.assign_f32(X.numpy(), C.numpy())
    _check_f32(a.cpu().numpy(), dist.cpu().numpy(), best, second, a_or, f"f32 n={n} d={d} k={k}")
    # the same through a screening copy built once
    a2, dist2 = skm.skm_assign(pts.with_screen(), C.to(DEV))
    assert torch.equal(a2, a) and torch.equal(dist2, dist)


def test_assign_f32_edge_cases(skm):
    X = _points(300, 40, seed=3)
    Xd = X.to(DEV)
    pts = skm.Points(skm.REPR_F32, Xd, 40)
    # k = 1
    a, _ = skm.skm_assign(pts, Xd[:1].clone())
    assert torch.all(a == 0)
    # n = k with centroids = points: identity, zero distance
    a, dist = skm.skm_assign(pts, Xd.clone())
    assert torch.equal(a.cpu(), torch.arange(300, dtype=torch.int32))
    assert float(dist.abs().max()) == 0.0
    # duplicated centroids: ties go to the lowest index
    C = torch.cat([Xd[5:6], Xd[5:6], Xd[9:10], Xd[9:10]]).contiguous()
    sub = skm.Points(skm.REPR_F32, Xd[[5, 9]].contiguous(), 40)
    a, _ = skm.skm_assign(sub, C)
    assert a.tolist() == [0, 2]


def test_update_f32_vs_oracle(skm):
    n, d, k = 5000, 100, 37
    X = _points(n, d, seed=4)
    a = torch.randint(0, k - 1, (n,), generator=torch.Generator().manual_seed(2), dtype=torch.int32)
    C0 = torch.randn(k, d, generator=torch.Generator().manual_seed(3))
    pts = skm.Points(skm.REPR_F32, X.to(DEV), d)
    C, counts = skm.skm_update(pts, a.to(DEV), C0.to(DEV).clone())
    Co, co = oracle.update_f32(X.numpy(), a.numpy(), C0.numpy())
    np.testing.assert_array_equal(counts.cpu().numpy(), co)
    Cg = C.cpu().numpy().astype(np.float64)
    rel = np.linalg.norm(Cg - Co, axis=1) / np.maximum(np.linalg.norm(Co, axis=1), 1e-30)
    assert rel.max() <= 1e-4
    np.testing.assert_array_equal(C.cpu().numpy()[k - 1], C0.numpy()[k - 1])  # empty cluster kept


@pytest.mark.parametrize("n,d,k", [(3000, 64, 300), (257, 256, 4000)])
def test_assign_f32_screen_overflow_fallback(skm, n, d, k):
    """Clusters of near-identical centroids (10 copies of each base point,
    relative perturbations ~1e-6, far inside the screen's bound) leave more
    than 4 candidates per row, so every row takes the exact fp32 fallback
    scan, with the centroids split across the grid when the row list is short."""
    X = _points(n, d, seed=7)
    g = torch.Generator().manual_seed(8)
    base = X[torch.randperm(n, generator=g)[: k // 10]]
    C = base.repeat_interleave(10, dim=0)
    C = (C * (1.0 + 1e-6 * torch.randn(C.shape, generator=g))).contiguous()
    pts = skm.Points(skm.REPR_F32, X.to(DEV), d)
    a, dist = skm.skm_assign(pts, C.to(DEV))
    if k <= n:  # skm_fit requires k <= n; it reports how many rows fell back
        _, _, _, _, st = skm.skm_fit(pts, k, 0, C_init=C.to(DEV), want_objective=False, want_dist=False)
        assert st["fallback_rows"] >= n // 2
    a_or, best, second = oracle.assign_f32(X.numpy(), C.numpy())
    # the copies are near ties by construction, so agreement is not the test:
    # every disagreement must sit at an oracle top-2 gap <= 1e-5, and the
    # reported distance must be the fp32 distance to the chosen centroid
    ag = a.cpu().numpy()
    gap = (second - best) / np.maximum(best, 1e-30)
    assert np.all(gap[ag != a_or] <= GAP_TOL)
    dch = ((X.numpy().astype(np.float64) - C.numpy().astype(np.float64)[ag]) ** 2).sum(1)
    np.testing.assert_allclose(dist.cpu().numpy(), dch, rtol=2e-5, atol=1e-6)


def _skewed_assign(n, k, seed):
    """60% of the points in cluster 0, the rest spread over 1..k-2 (k-1 stays
    empty), and every 997th point outside [0, k) (skipped by the update)."""
    g = torch.Generator().manual_seed(seed)
    a = torch.randint(1, k - 1, (n,), generator=g, dtype=torch.int32)
    a[torch.rand(n, generator=g) < 0.6] = 0
    a[::997] = -1
    return a


def _mixed_size_assign(n, k, seed):
    """Cluster sizes from {1, 2, 3, 5, 31, 32, 33, 64, 97, 200} in random
    order (so 32-row chunks of the sorted order hold one, two or many
    clusters), the rows shuffled, every 501st row outside [0, k)."""
    g = torch.Generator().manual_seed(seed)
    choices = torch.tensor([1, 2, 3, 5, 31, 32, 33, 64, 97, 200])
    sizes = choices[torch.randint(0, len(choices), (k,), generator=g)]
    lab = torch.repeat_interleave(torch.arange(k, dtype=torch.int32), sizes)
    lab = torch.cat([lab, torch.randint(0, k, (max(0, n - lab.numel()),), generator=g, dtype=torch.int32)])[:n]
    a = lab[torch.randperm(n, generator=g)].clone()
    a[::501] = -1
    return a


@pytest.mark.parametrize("d", [128, 384, 768, 1024])
@pytest.mark.parametrize("pattern", ["tiny", "mixed"])
def test_rbq1_update_transposed_table_sums(skm, d, pattern):
    """The 1-bit fused decode-average sums (bit transposes and subset-sum
    tables): chunks of 32 sorted rows from one cluster, from two (two table
    passes), and from many (rows one at a time), ragged last runs and skipped
    rows, against the oracle bit for bit."""
    n = 9973
    if pattern == "tiny":
        k = 3000
        a = torch.randint(0, k, (n,), generator=torch.Generator().manual_seed(d), dtype=torch.int32)
        a[::211] = -1
    else:
        k = 150
        a = _mixed_size_assign(n, k, seed=d + 1)
    X = _points(n, d, seed=d + 5)
    r = skm.skm_quantize(skm.REPR_RBQ1, X.to(DEV))
    pts = skm.rbq1_points(r, d)
    h = _rbq1_host(r)
    ok = (a >= 0).numpy()
    C0 = X[:k].clone()
    Cn, counts = skm.skm_update(pts, a.to(DEV), C0.to(DEV).clone())
    Co, co = oracle.rbq1_update(h["codes"][ok], h["F"][ok], d, h["m"], pts.rbq1_exp, a.numpy()[ok], C0.numpy())
    np.testing.assert_array_equal(counts.cpu().numpy(), co)
    np.testing.assert_array_equal(Cn.cpu().numpy(), Co)


@pytest.mark.parametrize("repr_name,n,d,k", [("f32", 70001, 128, 500), ("f32", 9000, 1536, 40),
                                             ("bf16", 20011, 1024, 300), ("bf16", 70001, 256, 500),
                                             ("bf16", 9001, 200, 40), ("bf16", 20011, 512, 300),
                                             ("rbq1", 70001, 128, 500),
                                             ("rbq1", 20011, 1024, 300), ("sq8", 70001, 128, 500),
                                             ("sq8", 20011, 1024, 300), ("sq8", 5003, 48, 20)])
def test_update_skewed_clusters(skm, repr_name, n, d, k):
    """Runs of the sorted order that cross many small clusters and one giant
    cluster shared by hundreds of runs; ragged last run; skipped points."""
    X = _points(n, d, seed=n + d)
    a = _skewed_assign(n, k, seed=d)
    ok = (a >= 0).numpy()
    C0 = X[:k].clone()
    if repr_name == "sq8":
        q = skm.skm_quantize(skm.REPR_SQ8, X.to(DEV))
        pts = skm.Points(skm.REPR_SQ8, q["codes"], d)
        codes = q["codes"].cpu().numpy()
        Cc = q["codes"][:k].clone()
        Cn, counts = skm.skm_update(pts, a.to(DEV), Cc.clone())
        Co, co = oracle.update_sq8(codes[ok], a.numpy()[ok], Cc.cpu().numpy())
        np.testing.assert_array_equal(counts.cpu().numpy(), co)
        np.testing.assert_array_equal(Cn.cpu().numpy(), Co)
        return
    if repr_name == "rbq1":
        r = skm.skm_quantize(skm.REPR_RBQ1, X.to(DEV))
        pts = skm.rbq1_points(r, d)
        h = _rbq1_host(r)
        Cn, counts = skm.skm_update(pts, a.to(DEV), C0.to(DEV).clone())
        Co, co = oracle.rbq1_update(h["codes"][ok], h["F"][ok], d, h["m"], pts.rbq1_exp,
                                    a.numpy()[ok], C0.numpy())
        np.testing.assert_array_equal(counts.cpu().numpy(), co)
        np.testing.assert_array_equal(Cn.cpu().numpy(), Co)
        return
    if repr_name == "bf16":
        Xb = X.to(torch.bfloat16)
        pts = skm.Points(skm.REPR_BF16, Xb.view(torch.int16).to(DEV), d)
        Co, co = oracle.update_bf16(Xb.view(torch.int16).numpy().view(np.uint16)[ok], a.numpy()[ok],
                                    C0.numpy())
    else:
        pts = skm.Points(skm.REPR_F32, X.to(DEV), d)
        Co, co = oracle.update_f32(X.numpy()[ok], a.numpy()[ok], C0.numpy())
    Cn, counts = skm.skm_update(pts, a.to(DEV), C0.to(DEV).clone())
    np.testing.assert_array_equal(counts.cpu().numpy(), co)
    Cg = Cn.cpu().numpy().astype(np.float64)
    rel = np.linalg.norm(Cg - Co, axis=1) / np.maximum(np.linalg.norm(Co, axis=1), 1e-30)
    assert rel.max() <= 1e-4
    np.testing.assert_array_equal(Cn.cpu().numpy()[k - 1], C0.numpy()[k - 1])  # empty cluster kept


def test_fit_f32_tiny_workload(skm):
    spec = synth.WORKLOADS["tiny_f32"]
    X = synth.workload_points(spec, seed=0)
    idx = synth.forgy_indices(spec.n, spec.k, seed=0)
    pts = skm.Points(skm.REPR_F32, X.to(DEV), spec.d)
    C, a, dist, obj, stats = skm.skm_fit(pts, spec.k, spec.iters, init_idx=idx.to(DEV))
    print("tiny fit stats", stats)
    assert stats["fallback_rows"] < 0.01 * spec.n * (spec.iters + 1)
    Co, ao, objo = oracle.lloyd_f32(X.numpy(), X.numpy()[idx.numpy()], spec.iters)
    agree = (a.cpu().numpy() == ao).mean()
    assert agree >= AGREE
    assert abs(obj[-1] - objo[-1]) / objo[-1] <= 1e-4
    # the GPU trajectory's objective is non-increasing too
    for t in range(1, len(obj)):
        assert obj[t] <= obj[t - 1] * (1 + 1e-6)
    # final objective recomputed in fp64 from the GPU's own outputs
    full = oracle.objective_f32(X.numpy(), C.cpu().numpy(), a.cpu().numpy())
    assert abs(full - objo[-1]) / objo[-1] <= 1e-4


# ------------------------------------------------------------------ SQ8 path
@pytest.mark.parametrize("n,d", [(2000, 64), (777, 33), (1500, 1024), (50, 1), (333, 36), (257, 1500), (5000, 772)])
def test_quantize_sq8_bitexact(skm, n, d):
    X = _points(n, d, seed=n)
    q = skm.skm_quantize(skm.REPR_SQ8, X.to(DEV))
    b, s = oracle.sq8_fit(X.numpy())
    np.testing.assert_array_equal(q["b"].cpu().numpy(), b)
    np.testing.assert_array_equal(q["s"].cpu().numpy(), s)
    np.testing.assert_array_equal(q["codes"].cpu().numpy(), oracle.sq8_encode(X.numpy(), b, s))
    Y = skm.skm_sq8_decode(q["codes"], q["b"], q["s"])
    np.testing.assert_array_equal(Y.cpu().numpy(), oracle.sq8_decode(q["codes"].cpu().numpy(), b, s))


@pytest.mark.parametrize("bits", [8, 4])
def test_quantize_sq8_half_integer_quotients(skm, bits):
    """Fixed (b, s) per column, including scales whose reciprocal is subnormal or
    infinite, and points whose quotients (x - b)/s sit at or one or two ulps
    around every half-integer of the code range and beyond both ends."""
    g = np.random.default_rng(bits)
    d, n = 512, 600
    L = 255 if bits == 8 else 15
    b = g.uniform(-2, 2, size=d).astype(np.float32)
    s = (g.uniform(0.01, 3, size=d) / L).astype(np.float32)
    s[:4] = [1.0, 1.5 * 2.0 ** 127, 1e-40, 2.0 ** -126]
    b[:4] = [0.0, 0.0, 0.0, 0.0]
    m = g.integers(-4, 2 * L + 6, size=(n, d)).astype(np.float32) * np.float32(0.5)
    with np.errstate(over="ignore", invalid="ignore"):
        X = (b[None, :] + m * s[None, :]).astype(np.float32)
    X[~np.isfinite(X)] = 0.0
    nud = g.integers(-2, 3, size=(n, d))
    for _k in range(2):
        X = np.where(nud > 0, np.nextafter(X, np.float32(np.inf)), X)
        X = np.where(nud < 0, np.nextafter(X, np.float32(-np.inf)), X)
        nud = nud - np.sign(nud)
    X = X.astype(np.float32)
    q = skm.skm_quantize(skm.REPR_SQ8, torch.from_numpy(X).to(DEV), fit=False, b=torch.from_numpy(b).to(DEV),
                         s=torch.from_numpy(s).to(DEV), bits=bits)
    np.testing.assert_array_equal(q["codes"].cpu().numpy(), oracle.sq8_encode(X, b, s, bits=bits))


@pytest.mark.parametrize("n,d,k", [(2000, 64, 50), (777, 33, 7), (1024, 1024, 129), (300, 5, 300),
                                   (600, 1500, 40), (1000, 1024, 1)])
def test_assign_update_sq8_bitexact(skm, n, d, k):
    g = np.random.default_rng(n + d)
    Xc = g.integers(0, 256, size=(n, d)).astype(np.uint8)
    Cc = Xc[g.choice(n, k, replace=False)].copy()
    if k > 3:
        Cc[3] = Cc[1]  # duplicate
    pts = skm.Points(skm.REPR_SQ8, torch.from_numpy(Xc).to(DEV), d)
    a, dist = skm.skm_assign(pts, torch.from_numpy(Cc).to(DEV))
    ao, bo = oracle.assign_sq8(Xc, Cc)
    np.testing.assert_array_equal(a.cpu().numpy(), ao)
    np.testing.assert_array_equal(dist.cpu().numpy(), bo.astype(np.float32))
    C, counts = skm.skm_update(pts, a, torch.from_numpy(Cc).to(DEV).clone())
    Co, co = oracle.update_sq8(Xc, ao, Cc)
    np.testing.assert_array_equal(counts.cpu().numpy(), co)
    np.testing.assert_array_equal(C.cpu().numpy(), Co)


def test_fit_sq8_trajectory_bitexact(skm):
    n, d, k, iters = 6000, 256, 64, 6
    X = _points(n, d, seed=8)
    q = skm.skm_quantize(skm.REPR_SQ8, X.to(DEV))
    idx = synth.forgy_indices(n, k, seed=8)
    C, a, _, _, _ = skm.skm_fit(skm.Points(skm.REPR_SQ8, q["codes"], d), k, iters, init_idx=idx.to(DEV))
    codes = q["codes"].cpu().numpy()
    Co, ao = oracle.lloyd_sq8(codes, codes[idx.numpy()], iters)
    np.testing.assert_array_equal(a.cpu().numpy(), ao)
    np.testing.assert_array_equal(C.cpu().numpy(), Co)


# ---------------------------------------------------------------- RBQ1 path
def _rbq1_host(r):
    h = {k: v.cpu().numpy() for k, v in r.items()}
    h["codes"] = h["codes"].view(np.uint32)
    return h


@pytest.mark.parametrize("n,d", [(3000, 768), (777, 33), (500, 32), (400, 31), (100, 1), (333, 36), (257, 1500),
                                 (5000, 1024), (4999, 516)])
def test_encode_rbq1_vs_oracle(skm, n, d):
    X = _points(n, d, seed=n + 1)
    r = skm.skm_quantize(skm.REPR_RBQ1, X.to(DEV))
    h = _rbq1_host(r)
    m = oracle.rbq1_mean(X.numpy())
    np.testing.assert_array_equal(h["m"], m)  # the fixed-point mean, bit for bit
    # codes from the GPU's own mean must match the oracle's encoder bit for bit
    codes, nx2, F, popx = oracle.rbq1_encode(X.numpy(), h["m"])
    np.testing.assert_array_equal(h["codes"], codes)
    np.testing.assert_array_equal(h["popx"], popx)
    np.testing.assert_allclose(h["nx2"], nx2, rtol=1e-6)
    np.testing.assert_allclose(h["F"], F, rtol=1e-6)
    # unused high bits of the last word are zero
    if d % 32:
        assert np.all(h["codes"][:, -1] >> (d % 32) == 0)


@pytest.mark.parametrize("n,d,k", [(3000, 768, 300), (777, 33, 7), (500, 64, 1), (1000, 1024, 65),
                                   (600, 1500, 40), (2000, 100, 129), (1300, 1000, 300), (257, 128, 513)])
def test_assign_update_rbq1_bitexact(skm, n, d, k):
    X = _points(n, d, seed=n + 2)
    r = skm.skm_quantize(skm.REPR_RBQ1, X.to(DEV))
    pts = skm.rbq1_points(r, d)
    h = _rbq1_host(r)
    assert pts.rbq1_exp == oracle.rbq1_exponent(h["F"])
    C = X[synth.forgy_indices(n, k, seed=5)].clone()
    a, est = skm.skm_assign(pts, C.to(DEV))
    prep = oracle.rbq1_centroid_sq4(C.numpy(), h["m"])
    ao, esto = oracle.rbq1_assign(h["codes"], h["nx2"], h["F"], h["popx"], d, prep)
    np.testing.assert_array_equal(a.cpu().numpy(), ao)
    np.testing.assert_array_equal(est.cpu().numpy(), esto)
    Cn, counts = skm.skm_update(pts, a, C.to(DEV).clone())
    Co, co = oracle.rbq1_update(h["codes"], h["F"], d, h["m"], pts.rbq1_exp, ao, C.numpy())
    np.testing.assert_array_equal(counts.cpu().numpy(), co)
    np.testing.assert_array_equal(Cn.cpu().numpy(), Co)


@pytest.mark.parametrize("d", [128, 768, 1000])
def test_assign_rbq1_packed_codes_equal_expanded_copy(skm, d):
    """Without a screening copy the tensor-core kernel reads 16-byte aligned
    codes packed (converter warps expand each point tile into a per-CTA slot);
    with the e4m3 copy, or for misaligned codes, it reads the copy.  All give
    the oracle's assignment and estimates bit for bit."""
    n, k = 3001, 260
    X = _points(n, d, seed=d + 31)
    r = skm.skm_quantize(skm.REPR_RBQ1, X.to(DEV))
    pts = skm.rbq1_points(r, d)
    codes = r["codes"].view(torch.int32).reshape(n, -1)
    W = codes.shape[1]
    buf = torch.zeros(n * W + 1, dtype=torch.int32, device=DEV)
    buf[1:] = codes.reshape(-1)
    off = buf[1:].view(n, W)  # 4 bytes past a 16-byte boundary
    assert off.data_ptr() % 16 == 4 and pts.x.data_ptr() % 16 == 0
    pts_off = skm.Points(skm.REPR_RBQ1, off, d, pts.nx2, pts.F, pts.popx, pts.m, pts.rbq1_exp)
    C = X[synth.forgy_indices(n, k, seed=3)].clone().to(DEV)
    a, est = skm.skm_assign(pts, C)
    a2, est2 = skm.skm_assign(pts_off, C)
    a3, est3 = skm.skm_assign(pts.with_screen(), C)
    h = _rbq1_host(r)
    ao, esto = oracle.rbq1_assign(h["codes"], h["nx2"], h["F"], h["popx"], d,
                                  oracle.rbq1_centroid_sq4(C.cpu().numpy(), h["m"]))
    np.testing.assert_array_equal(a.cpu().numpy(), ao)
    np.testing.assert_array_equal(est.cpu().numpy(), esto)
    assert torch.equal(a, a2) and torch.equal(est, est2)
    assert torch.equal(a, a3) and torch.equal(est, est3)


def test_fit_rbq1_trajectory_bitexact(skm):
    n, d, k, iters = 8000, 256, 50, 6
    X = _points(n, d, seed=9)
    r = skm.skm_quantize(skm.REPR_RBQ1, X.to(DEV))
    pts = skm.rbq1_points(r, d)
    idx = synth.forgy_indices(n, k, seed=9)
    C, a, _, _, _ = skm.skm_fit(pts, k, iters, init_idx=idx.to(DEV))
    h = _rbq1_host(r)
    C0 = oracle.rbq1_decode_points(h["codes"], h["F"], d, h["m"], pts.rbq1_exp, idx.numpy())
    Co, ao = oracle.lloyd_rbq1(h["codes"], h["nx2"], h["F"], h["popx"], d, h["m"], C0, iters, pts.rbq1_exp)
    np.testing.assert_array_equal(a.cpu().numpy(), ao)
    np.testing.assert_array_equal(C.cpu().numpy(), Co)


# ------------------------------------------------------ projection and bf16
@pytest.mark.parametrize("n,d,dout,path", [(1000, 128, 128, "tc"), (777, 100, 33, "tc"), (2048, 1024, 256, "tc"),
                                          (3000, 96, 96, "chunked"), (777, 100, 33, "cuda_cores"),
                                          (1000, 768, 768, "tc"), (129, 8, 3, "tc")])
def test_project_vs_oracle(skm, n, d, dout, path):
    """Tensor-core projection (bf16 parts, six products, one pass or in row
    chunks) and the CUDA-core kernel: fp32 accuracy against the fp64 oracle."""
    X = _points(n, d, seed=d)
    P = synth.haar_rotation(d, 4)[:, :dout].to(torch.float32).contiguous()
    mu = X.mean(0)
    kw = {"cuda_cores": True} if path == "cuda_cores" else ({"max_ws_bytes": 1} if path == "chunked" else {})
    Y = skm.skm_project(X.to(DEV), P.to(DEV), mu.to(DEV), **kw)
    Yo = oracle.project(X.numpy(), P.numpy(), mu.numpy())
    scale = np.linalg.norm(X.numpy() - mu.numpy(), axis=1)[:, None]
    assert np.max(np.abs(Y.cpu().numpy() - Yo) / scale) < 2e-6
    Yb = skm.skm_project(X.to(DEV), P.to(DEV), mu.to(DEV), out_dtype=skm.DTYPE_BF16, **kw)
    yb = Yb.view(torch.int16).cpu().numpy().view(np.uint16)
    ybo = oracle.round_bf16(Yo)
    # bf16 of the fp32 result vs the fp64 result: within half a bf16 ulp of
    # the value plus the fp32 accumulation error; identical codes for almost all
    err = np.abs(oracle.bf16_to_f32(yb).astype(np.float64) - Yo)
    assert np.all(err <= 2.0 ** -8 * np.abs(Yo) + 2e-6 * scale)
    assert (yb == ybo).mean() > 0.99


@pytest.mark.parametrize("n,d,k", [(2000, 256, 100), (777, 64, 13), (300, 32, 300)])
def test_assign_update_bf16_vs_oracle(skm, n, d, k):
    X = _points(n, d, seed=n)
    Xb = X.to(DEV).to(torch.bfloat16)
    xb = Xb.view(torch.int16).cpu().numpy().view(np.uint16)
    C = oracle.bf16_to_f32(xb[synth.forgy_indices(n, k, seed=3).numpy()]).copy()
    pts = skm.Points(skm.REPR_BF16, Xb.view(torch.int16), d)
    a, dist = skm.skm_assign(pts, torch.from_numpy(C).to(DEV))
    a_or, best, second = oracle.assign_bf16(xb, C)
    _check_f32(a.cpu().numpy(), dist.cpu().numpy(), best, second, a_or, "bf16")
    Cn, counts = skm.skm_update(pts, torch.from_numpy(a_or).to(DEV), torch.from_numpy(C).to(DEV).clone())
    Co, co = oracle.update_bf16(xb, a_or, C)
    np.testing.assert_array_equal(counts.cpu().numpy(), co)
    rel = np.linalg.norm(Cn.cpu().numpy() - Co, axis=1) / np.maximum(np.linalg.norm(Co, axis=1), 1e-30)
    assert rel.max() <= 1e-4


def test_pca_fit_vs_oracle(skm):
    n, d, dout = 20000, 64, 16
    X = _points(n, d, seed=12)
    mean, P, w = skm.skm_pca_fit(X.to(DEV), dout)
    mu, Po, wo = oracle.pca_fit(X.numpy(), dout)
    np.testing.assert_allclose(mean.cpu().numpy(), mu, rtol=1e-5, atol=1e-7)
    np.testing.assert_allclose(w.cpu().numpy(), wo, rtol=1e-4)
    # eigenvectors agree where the spectrum is separated (sign fixed on both sides)
    gaps = np.abs(np.diff(np.concatenate([wo, [0.0]]))) / wo
    sep = gaps > 1e-2
    sep[1:] &= gaps[:-1] > 1e-2
    Pg = P.cpu().numpy()
    for j in np.where(sep)[0]:
        assert abs(float(Pg[:, j] @ Po[:, j])) > 0.999


# --------------------------------------------------------- sharded update
@pytest.mark.parametrize("repr_name", ["f32", "sq8", "rbq1", "bf16"])
def test_sharded_update_matches_single(skm, repr_name):
    n, d, k = 4000, 64, 20
    X = _points(n, d, seed=21)
    Xd = X.to(DEV)
    if repr_name == "f32":
        pts = skm.Points(skm.REPR_F32, Xd, d)
        C = Xd[:k].clone()
        pdt, pshape = torch.float64, (k, d)
    elif repr_name == "bf16":  # rows of 128 bytes: the direct register path, fp64 partials
        Xb = Xd.to(torch.bfloat16).view(torch.int16)
        pts = skm.Points(skm.REPR_BF16, Xb, d)
        C = (Xb[:k].to(torch.int32) << 16).view(torch.float32).contiguous()
        pdt, pshape = torch.float64, (k, d)
    elif repr_name == "sq8":
        q = skm.skm_quantize(skm.REPR_SQ8, Xd)
        pts = skm.Points(skm.REPR_SQ8, q["codes"], d)
        C = q["codes"][:k].clone()
        pdt, pshape = torch.int64, (k, d)
    else:
        r = skm.skm_quantize(skm.REPR_RBQ1, Xd)
        pts = skm.rbq1_points(r, d)
        C = Xd[:k].clone()
        pdt, pshape = torch.int64, (k, d + 1)
    a, _ = skm.skm_assign(pts, C)
    C_single, cnt_single = skm.skm_update(pts, a, C.clone())
    bounds = [0, 1000, 1001, 2777, n]
    total = torch.zeros(pshape, dtype=pdt, device=DEV)
    counts = torch.zeros(k, dtype=torch.int64, device=DEV)
    for lo, hi in zip(bounds[:-1], bounds[1:]):
        part = torch.zeros(pshape, dtype=pdt, device=DEV)
        sub_x = pts.x[lo:hi].contiguous()
        extra = {}
        if repr_name == "rbq1":
            extra = dict(nx2=pts.nx2[lo:hi].contiguous(), F=pts.F[lo:hi].contiguous(),
                         popx=pts.popx[lo:hi].contiguous(), m=pts.m, rbq1_exp=pts.rbq1_exp)
        sp = skm.Points(pts.repr, sub_x, d, **extra)
        skm.skm_update(sp, a[lo:hi].contiguous(), None, counts=counts, partial=part)
        skm.skm_merge_partials(total, part)
    C_merged = skm.skm_update_finalize(pts, total, counts, C.clone())
    assert torch.equal(counts, cnt_single)
    if repr_name in ("f32", "bf16"):
        rel = (C_merged - C_single).norm(dim=1) / C_single.norm(dim=1)
        assert float(rel.max()) <= 1e-5
    else:
        assert torch.equal(C_merged, C_single)


# -------------------------------------------------- exact dimension pruning
@pytest.mark.parametrize("repr_name,n,d,k", [("bf16", 3000, 256, 300), ("bf16", 777, 64, 13),
                                             ("f32", 2000, 768, 200), ("f32", 500, 33, 40)])
def test_prune_assign_vs_oracle_and_seed_independent(skm, repr_name, n, d, k):
    X = _points(n, d, seed=n + k)
    if repr_name == "bf16":
        Xd = X.to(DEV).to(torch.bfloat16).view(torch.int16)
        xb = Xd.cpu().numpy().view(np.uint16)
        C = oracle.bf16_to_f32(xb[synth.forgy_indices(n, k, seed=4).numpy()]).copy()
        pts = skm.Points(skm.REPR_BF16, Xd, d)
        a_or, best, second = oracle.assign_bf16(xb, C)
    else:
        Xd = X.to(DEV)
        C = X[synth.forgy_indices(n, k, seed=4)].numpy().copy()
        pts = skm.Points(skm.REPR_F32, Xd, d)
        a_or, best, second = oracle.assign_f32(X.numpy(), C)
    Cd = torch.from_numpy(C).to(DEV)
    pp = pts.with_flags(skm.FLAG_PRUNE)
    a0, d0 = skm.skm_assign(pp, Cd)
    _check_f32(a0.cpu().numpy(), d0.cpu().numpy(), best, second, a_or, f"prune {repr_name}")
    # the seed of the bound changes the work, never the result
    prev = torch.randint(0, k, (n,), generator=torch.Generator().manual_seed(7), dtype=torch.int32).to(DEV)
    ws = skm.workspace(skm.OP_ASSIGN, pp, k)
    a1, d1 = skm.skm_assign(pp, Cd, prev_assign=prev, ws=ws)
    st1 = skm.skm_assign_prune_stats(ws)
    a2, d2 = skm.skm_assign(pp, Cd, prev_assign=a0.clone(), ws=ws)
    st2 = skm.skm_assign_prune_stats(ws)  # counters restart with every call
    assert torch.equal(a1, a0) and torch.equal(a2, a0)
    assert torch.equal(d1, d0) and torch.equal(d2, d0)
    nb = (d + 31) // 32
    for st in (st1, st2):
        if st["prune_front_dims"]:
            # bf16 with a seed: the tensor-core front screened 128 dimensions
            # of every pair; every row keeps at least its seed; complete pairs
            # evaluated all nb blocks on CUDA cores
            assert repr_name == "bf16" and d >= 256 and st["prune_front_dims"] == 128
            assert n <= st["prune_first_block"] <= n * k
            assert 0 <= st["prune_complete"] <= st["prune_first_block"]
            assert st["prune_rows_finished"] + st["prune_rows_full"] <= n
            assert st["prune_complete"] * nb <= st["prune_blocks"]
            assert st["prune_blocks"] <= (st["prune_first_block"] + st["prune_rows_full"] * k) * nb
            continue
        # every pair evaluates its first block; a pair alive after block b
        # evaluates block b + 1; complete pairs evaluated all nb blocks
        assert 0 < st["prune_complete"] <= st["prune_first_block"] <= n * k
        assert st["prune_complete"] * (nb - 1) <= st["prune_blocks"] <= st["prune_first_block"] * (nb - 1)
    # the bound from the nearest centroid leaves no more work than a random one
    assert st2["prune_blocks"] <= st1["prune_blocks"] and st2["prune_first_block"] <= st1["prune_first_block"]
    # and the tensor-core screen reaches the same assignment
    a3, _ = skm.skm_assign(pts, Cd)
    assert (a3 == a0).float().mean().item() >= AGREE


@pytest.mark.parametrize("n,d,k", [(3000, 256, 1000), (1000, 512, 300), (700, 1024, 257), (5000, 256, 13),
                                   (130, 256, 600), (20000, 256, 1000), (1500, 264, 300), (900, 1000, 200)])
def test_prune_front_tensor_cores_bitexact(skm, n, d, k):
    """bf16 points with a seed assignment: the first 128 dimensions of every
    pair screened on tensor cores, survivors finished on CUDA cores (Section
    3.1 "SuperKMeans", a GEMM over the front dimensions, then pruning).  The
    result equals the CUDA-core pruning's (seed 0, no front) bit for bit,
    assignments and distances, with good seeds (most rows decided by the
    front), in place (seed array = output), and with random seeds (lists
    overflow to the full pruning: one CTA per row, or at 20,000 rows the
    tiled kernel over the row list); and it matches the oracle."""
    X = _points(n, d, seed=n + d + k)
    Xd = X.to(DEV).to(torch.bfloat16).view(torch.int16)
    xb = Xd.cpu().numpy().view(np.uint16)
    g = torch.Generator().manual_seed(k)
    # fp32 centroids off the bf16 grid (the bound's residual terms matter)
    C = torch.from_numpy(oracle.bf16_to_f32(xb[synth.forgy_indices(n, k, seed=5).numpy()]).copy())
    C = (C + 0.01 * C.std() * torch.randn(C.shape, generator=g)).contiguous()
    Cd = C.to(DEV)
    pp = skm.Points(skm.REPR_BF16, Xd, d, flags=skm.FLAG_PRUNE)
    a0, d0 = skm.skm_assign(pp, Cd)  # no seed: CUDA cores only
    a_or, best, second = oracle.assign_bf16(xb, C.numpy())
    _check_f32(a0.cpu().numpy(), d0.cpu().numpy(), best, second, a_or, f"prune n={n} d={d} k={k}")
    seed_good, _ = skm.skm_assign(skm.Points(skm.REPR_BF16, Xd, d).with_screen(), Cd)
    ws = skm.workspace(skm.OP_ASSIGN, pp, k)
    a1, d1 = skm.skm_assign(pp, Cd, prev_assign=seed_good, ws=ws)
    st = skm.skm_assign_prune_stats(ws)
    assert torch.equal(a1, a0) and torch.equal(d1, d0)
    assert st["prune_front_dims"] == 128
    assert n <= st["prune_first_block"] <= n * k
    assert st["prune_rows_finished"] + st["prune_rows_full"] <= n
    inplace = seed_good.clone()
    dd = torch.empty(n, device=DEV, dtype=torch.float32)
    skm.skm_assign(pp, Cd, prev_assign=inplace, ws=ws, out=inplace, dist_out=dd)
    assert torch.equal(inplace, a0) and torch.equal(dd, d0)
    seed_bad = torch.randint(0, k, (n,), generator=g, dtype=torch.int32).to(DEV)
    a2, d2 = skm.skm_assign(pp, Cd, prev_assign=seed_bad, ws=ws)
    st2 = skm.skm_assign_prune_stats(ws)
    assert torch.equal(a2, a0) and torch.equal(d2, d0)
    assert st2["prune_first_block"] >= st["prune_first_block"]
    if k >= 300:
        assert st2["prune_rows_full"] > 0  # random seeds keep more than a list holds (128)
    # CUDA cores only (no front), seeded alike: the same result
    wsc = skm.workspace(skm.OP_ASSIGN, pp.with_flags(skm.FLAG_PRUNE | skm.FLAG_PRUNE_CUDA_CORES), k)
    a4, d4 = skm.skm_assign(pp.with_flags(skm.FLAG_PRUNE | skm.FLAG_PRUNE_CUDA_CORES), Cd, prev_assign=seed_good,
                            ws=wsc)
    assert torch.equal(a4, a0) and torch.equal(d4, d0)
    assert skm.skm_assign_prune_stats(wsc)["prune_front_dims"] == 0
    # without distances, and seeds outside [0, k) (centroid 0)
    seed_out = seed_good.clone()
    seed_out[::7] = -1
    seed_out[3::7] = k
    a3, _ = skm.skm_assign(pp, Cd, prev_assign=seed_out, ws=ws, want_dist=False)
    assert torch.equal(a3, a0)


def test_prune_front_kept_bounds_across_lloyd_steps(skm):
    """SKM_FLAG_WARM with the tensor-core pruning front: after the first call
    each row's threshold comes from the bound the previous call left, grown
    by its centroid's move, without reading the points.  Every Lloyd step's
    assignment equals the CUDA-core pruning's bit for bit; a call that wants
    distances gets the exact ones and keeps the state usable; a workspace
    holding another point set's state (same shapes) is cleared by skm_fit."""
    n, d, k = 4000, 256, 300
    X = _points(n, d, seed=77)
    Xd = X.to(DEV).to(torch.bfloat16).view(torch.int16)
    xb = Xd.cpu().numpy().view(np.uint16)
    C = torch.from_numpy(oracle.bf16_to_f32(xb[synth.forgy_indices(n, k, seed=9).numpy()]).copy()).to(DEV)
    pw = skm.Points(skm.REPR_BF16, Xd, d, flags=skm.FLAG_PRUNE | skm.FLAG_WARM)
    pc = skm.Points(skm.REPR_BF16, Xd, d, flags=skm.FLAG_PRUNE)
    ws = skm.workspace(skm.OP_ASSIGN, pw, k)
    a_prev, _ = skm.skm_assign(pc, C)  # no seed: CUDA cores
    for it in range(6):
        a_c, d_c = skm.skm_assign(pc, C)
        if it == 3:  # distances wanted: exact seed distances this call
            a_w, d_w = skm.skm_assign(pw, C, prev_assign=a_prev, ws=ws)
            assert torch.equal(d_w, d_c)
        else:
            a_w, _ = skm.skm_assign(pw, C, prev_assign=a_prev, ws=ws, want_dist=False)
        assert torch.equal(a_w, a_c), f"step {it}"
        st = skm.skm_assign_prune_stats(ws)
        assert st["prune_front_dims"] == 128 and n <= st["prune_first_block"]
        C = C.clone()
        skm.skm_update(pc, a_c, C)
        a_prev = a_w
    # skm_fit on a second point set of the same shapes, in a workspace that
    # holds the first set's state: the same result as in a fresh workspace
    X2 = _points(n, d, seed=78)
    X2d = X2.to(DEV).to(torch.bfloat16).view(torch.int16)
    x2b = X2d.cpu().numpy().view(np.uint16)
    C2 = torch.from_numpy(oracle.bf16_to_f32(x2b[synth.forgy_indices(n, k, seed=10).numpy()]).copy()).to(DEV)
    p1 = skm.Points(skm.REPR_BF16, Xd, d, flags=skm.FLAG_PRUNE)
    p2 = skm.Points(skm.REPR_BF16, X2d, d, flags=skm.FLAG_PRUNE)
    wsf = skm.workspace(skm.OP_FIT, p1, k)
    skm.skm_fit(p1, k, 4, C_init=C2.clone(), ws=wsf, want_objective=False)
    Ca, aa, _, _, _ = skm.skm_fit(p2, k, 4, C_init=C2.clone(), ws=wsf, want_objective=False)
    Cb, ab, _, _, _ = skm.skm_fit(p2, k, 4, C_init=C2.clone(), want_objective=False)
    assert torch.equal(aa, ab)
    # (the fp32 update's sums are accumulated in an order that varies)
    rel = (Ca - Cb).norm(dim=1) / Cb.norm(dim=1).clamp_min(1e-30)
    assert float(rel.max()) <= 1e-6


@pytest.mark.parametrize("repr_name", ["bf16", "f32"])
def test_warm_screen_bounds_across_lloyd_steps(skm, repr_name):
    """SKM_FLAG_WARM: each call starts every row's screen threshold from the
    bound the previous call left, grown by the centroid's move.  Over Lloyd
    steps (assign, update) the warm calls give the cold calls' assignment
    and distances (disagreements only at oracle near-ties) and pass the
    oracle's checks."""
    n, d, k, steps = 20011, 256, 300, 4
    X = _points(n, d, seed=77)
    if repr_name == "bf16":
        Xd = X.to(DEV).to(torch.bfloat16).view(torch.int16)
        xb = Xd.cpu().numpy().view(np.uint16)
        pts = skm.Points(skm.REPR_BF16, Xd, d)
        C = torch.from_numpy(oracle.bf16_to_f32(xb[synth.forgy_indices(n, k, seed=6).numpy()]).copy()).to(DEV)
    else:
        Xd = X.to(DEV)
        pts = skm.Points(skm.REPR_F32, Xd, d)
        C = X[synth.forgy_indices(n, k, seed=6)].clone().to(DEV)
    warm = pts.with_flags(skm.FLAG_WARM)
    ws = skm.workspace(skm.OP_ASSIGN, warm, k)
    for step in range(steps):
        a_w, d_w = skm.skm_assign(warm, C, ws=ws)
        a_c, d_c = skm.skm_assign(pts, C)
        same = (a_w == a_c).float().mean().item()
        assert same >= 0.9999, f"step {step}: warm and cold agree on {same}"
        if repr_name == "bf16":
            a_or, best, second = oracle.assign_bf16(xb, C.cpu().numpy())
        else:
            a_or, best, second = oracle.assign_f32(X.numpy(), C.cpu().numpy())
        _check_f32(a_w.cpu().numpy(), d_w.cpu().numpy(), best, second, a_or, f"warm step {step}")
        C, _ = skm.skm_update(pts, a_w, C.clone())


def test_warm_screen_restarts_cold_on_other_shapes_and_after_abort(skm):
    """A workspace stamped by a call with another k starts cold; a call that
    gave up (injected wait) leaves no stamp, so the next warm call starts
    cold too; every result still equals the cold call's."""
    n, d = 9000, 128
    X = _points(n, d, seed=78).to(DEV)
    pts = skm.Points(skm.REPR_F32, X, d).with_flags(skm.FLAG_WARM)
    ws = skm.workspace(skm.OP_ASSIGN, pts, 400)
    C1, C2 = X[:400].clone(), X[1000:1250].clone()
    skm.skm_assign(pts, C1, ws=ws)
    a_w, _ = skm.skm_assign(pts, C2, ws=ws)  # k changed: cold
    a_c, _ = skm.skm_assign(pts.with_flags(0), C2)
    assert (a_w == a_c).float().mean().item() >= 0.9999
    skm.skm_assign(pts, C2, ws=ws)  # warm
    skm.skm_inject_fault(4, 1)  # SKM_FAULT_WAIT: this call's screen gives up before any load
    skm.skm_assign(pts, (C2 * 1.01).contiguous(), ws=ws)  # asynchronous: its outputs are not used
    torch.cuda.synchronize()
    assert skm.skm_fault_armed(4) == 0
    C3 = (C2 * 0.99).contiguous()
    a_w, d_w = skm.skm_assign(pts, C3, ws=ws)
    a_c, d_c = skm.skm_assign(pts.with_flags(0), C3)
    assert (a_w == a_c).float().mean().item() >= 0.9999


def test_prune_fit_bf16(skm):
    """skm_fit with SKM_FLAG_PRUNE on bf16 points (d = 256): the dense screen
    for the first iterations, the pruned assignment (tensor-core front) once
    fewer than 1% of the rows change cluster; the trajectory matches the
    oracle's."""
    n, d, k, iters = 6000, 256, 64, 12
    X = _points(n, d, seed=33)
    Xd = X.to(DEV).to(torch.bfloat16).view(torch.int16)
    xb = Xd.cpu().numpy().view(np.uint16)
    idx = synth.forgy_indices(n, k, seed=33)
    C0 = oracle.bf16_to_f32(xb[idx.numpy()]).copy()
    pts = skm.Points(skm.REPR_BF16, Xd, d, flags=skm.FLAG_PRUNE)
    C, a, _, obj, stats = skm.skm_fit(pts, k, iters, C_init=torch.from_numpy(C0).to(DEV))
    Co, ao, objo = oracle.lloyd_bf16(xb, C0, iters)
    assert (a.cpu().numpy() == ao).mean() >= AGREE
    assert abs(obj[-1] - objo[-1]) / objo[-1] <= 1e-4
    total = n * k * (iters + 1)
    print("prune stats", stats, "first-block survival", stats["prune_first_block"] / total)
    assert stats["prune_front_dims"] == 128  # the pruned assignment ran
    assert n <= stats["prune_first_block"] <= total
    assert 0 <= stats["prune_complete"] <= stats["prune_first_block"]


# ------------------------------------------------------ empty-cluster split
def _dup_init(n, k, seed):
    """Forgy indices where every 4th entry repeats its predecessor: identical
    centroids tie for every point, so the later copy ends up empty."""
    idx = synth.forgy_indices(n, k, seed=seed).clone()
    idx[1::4] = idx[0::4][: idx[1::4].numel()]
    return idx


@pytest.mark.parametrize("kind", ["f32", "sq8"])
def test_split_empty_matches_oracle(skm, kind):
    g = np.random.default_rng(11)
    k, d = 300, 40
    counts = g.integers(0, 6, size=k).astype(np.int64)
    counts[g.choice(k, 40, replace=False)] = 0
    counts[7] = counts[19] = 50  # a tie between the two largest
    if kind == "sq8":
        C = g.integers(0, 256, size=(k, d)).astype(np.uint8)
        pts = skm.Points(skm.REPR_SQ8, torch.zeros(1, d, dtype=torch.uint8, device=DEV), d)
    else:
        C = g.normal(size=(k, d)).astype(np.float32)
        pts = skm.Points(skm.REPR_F32, torch.zeros(1, d, device=DEV), d)
    Cg = torch.from_numpy(C.copy()).to(DEV)
    skm.skm_split_empty(pts, Cg, torch.from_numpy(counts).to(DEV))
    Co, ns = oracle.split_empty(C, counts)
    assert ns == int((counts == 0).sum())
    np.testing.assert_array_equal(Cg.cpu().numpy(), Co)


def test_fit_sq8_with_split_trajectory_bitexact(skm):
    n, d, k, iters = 6000, 64, 48, 6
    X = _points(n, d, seed=21)
    q = skm.skm_quantize(skm.REPR_SQ8, X.to(DEV))
    codes = q["codes"].cpu().numpy()
    idx = _dup_init(n, k, seed=21)
    C, a, _, _, st = skm.skm_fit(skm.Points(skm.REPR_SQ8, q["codes"], d), k, iters, init_idx=idx.to(DEV),
                                 empty_policy=skm.EMPTY_SPLIT)
    Co, ao = oracle.lloyd_sq8(codes, codes[idx.numpy()], iters, split=True)
    np.testing.assert_array_equal(a.cpu().numpy(), ao)
    np.testing.assert_array_equal(C.cpu().numpy(), Co)
    # without the split the duplicated centroids stay empty
    _, a0, _, _, st0 = skm.skm_fit(skm.Points(skm.REPR_SQ8, q["codes"], d), k, iters, init_idx=idx.to(DEV))
    assert st0["empty_clusters"] > st["empty_clusters"]


def test_fit_rbq1_with_split_trajectory_bitexact(skm):
    n, d, k, iters = 8000, 128, 40, 5
    X = _points(n, d, seed=22)
    r = skm.skm_quantize(skm.REPR_RBQ1, X.to(DEV))
    pts = skm.rbq1_points(r, d)
    idx = _dup_init(n, k, seed=22)
    C, a, _, _, _ = skm.skm_fit(pts, k, iters, init_idx=idx.to(DEV), empty_policy=skm.EMPTY_SPLIT)
    h = _rbq1_host(r)
    C0 = oracle.rbq1_decode_points(h["codes"], h["F"], d, h["m"], pts.rbq1_exp, idx.numpy())
    Co, ao = oracle.lloyd_rbq1(h["codes"], h["nx2"], h["F"], h["popx"], d, h["m"], C0, iters, pts.rbq1_exp,
                               split=True)
    np.testing.assert_array_equal(a.cpu().numpy(), ao)
    np.testing.assert_array_equal(C.cpu().numpy(), Co)


def test_fit_f32_with_split_vs_oracle(skm):
    n, d, k, iters = 5000, 32, 40, 5
    X = _points(n, d, seed=23)
    idx = _dup_init(n, k, seed=23)
    pts = skm.Points(skm.REPR_F32, X.to(DEV), d)
    C, a, _, obj, st = skm.skm_fit(pts, k, iters, init_idx=idx.to(DEV), empty_policy=skm.EMPTY_SPLIT)
    Co, ao, objo = oracle.lloyd_f32(X.numpy(), X.numpy()[idx.numpy()], iters, split=True)
    assert (a.cpu().numpy() == ao).mean() >= AGREE
    assert abs(obj[-1] - objo[-1]) / objo[-1] <= 1e-4
    # the duplicated centroids would stay empty without the split
    _, a0, _, _, _ = skm.skm_fit(pts, k, iters, init_idx=idx.to(DEV))
    empty = lambda v: int((np.bincount(v, minlength=k) == 0).sum())  # noqa: E731
    assert empty(a.cpu().numpy()) < empty(a0.cpu().numpy())


# ------------------------------------------------------------------- SQ4
@pytest.mark.parametrize("n,d,k", [(3000, 64, 40), (1500, 1024, 33), (777, 33, 7)])
def test_sq4_quantize_assign_update_fit_bitexact(skm, n, d, k):
    """4-bit codes through the SQ8 entry points: encode, exact code-domain
    assignment and update, and a whole Lloyd trajectory, against the oracle."""
    X = _points(n, d, seed=n + 4)
    q = skm.skm_quantize(skm.REPR_SQ8, X.to(DEV), bits=4)
    b, s = oracle.sq8_fit(X.numpy(), bits=4)
    np.testing.assert_array_equal(q["b"].cpu().numpy(), b)
    np.testing.assert_array_equal(q["s"].cpu().numpy(), s)
    codes = q["codes"].cpu().numpy()
    np.testing.assert_array_equal(codes, oracle.sq8_encode(X.numpy(), b, s, bits=4))
    assert codes.max() <= 15
    pts = skm.Points(skm.REPR_SQ8, q["codes"], d)
    idx = synth.forgy_indices(n, k, seed=4)
    C, a, dist, _, _ = skm.skm_fit(pts, k, 4, init_idx=idx.to(DEV))
    Co, ao = oracle.lloyd_sq8(codes, codes[idx.numpy()], 4)
    np.testing.assert_array_equal(a.cpu().numpy(), ao)
    np.testing.assert_array_equal(C.cpu().numpy(), Co)
    assert C.cpu().numpy().max() <= 15


# ------------------------------------------------ randomized Hadamard rotation
@pytest.mark.parametrize("n,d,D", [(1000, 33, 64), (777, 100, 128), (3000, 768, 1024), (500, 1024, 1024),
                                   (300, 2000, 2048), (64, 4096, 4096), (50, 20, 32)])
def test_project_hadamard_vs_oracle(skm, n, d, D):
    X = _points(n, d, seed=d + 1)
    sigma = synth.hadamard_signs(D, seed=d)
    mean = X.mean(0) if d % 2 else None
    Y = skm.skm_project_hadamard(X.to(DEV), sigma.to(DEV), None if mean is None else mean.to(DEV))
    Yo = oracle.hadamard_rotate(X.numpy(), sigma.numpy(), None if mean is None else mean.numpy())
    Yg = Y.cpu().numpy().astype(np.float64)
    err = np.linalg.norm(Yg - Yo, axis=1) / np.maximum(np.linalg.norm(Yo, axis=1), 1e-30)
    assert err.max() <= 2e-6
    # bf16 output: the fp32 result rounded to nearest even
    Yb = skm.skm_project_hadamard(X.to(DEV), sigma.to(DEV), None if mean is None else mean.to(DEV),
                                  out_dtype=skm.DTYPE_BF16).float().cpu().numpy()
    assert np.all(np.abs(Yb - Yo) <= 2.0 ** -8 * np.abs(Yo) + 1e-6)


# ------------------------------------------------------- segmented assignment
_SEG_SIZES = [1, 127, 129, 300, 5, 1000, 64, 257, 2, 700]
_SEG_KS = [1, 3, 200, 2, 40, 300, 7, 1, 2, 90]


def _segments():
    group = np.repeat(np.arange(len(_SEG_SIZES)), _SEG_SIZES).astype(np.int32)
    base = np.concatenate([[0], np.cumsum(_SEG_KS)]).astype(np.int32)
    return group, base


@pytest.mark.parametrize("kind", ["f32", "bf16", "sq8", "rbq1"])
def test_assign_segmented_vs_oracle_per_group(skm, kind):
    group, base = _segments()
    n, k, d = group.size, int(base[-1]), 96
    X = _points(n, d, seed=41)
    g = torch.from_numpy(group).to(DEV)
    bt = torch.from_numpy(base).to(DEV)
    Cf = _points(k, d, seed=42)
    if kind in ("f32", "bf16"):
        if kind == "bf16":
            Xb = X.to(torch.bfloat16)
            xb = Xb.view(torch.int16).numpy().view(np.uint16)
            pts = skm.Points(skm.REPR_BF16, Xb.view(torch.int16).to(DEV), d)
        else:
            pts = skm.Points(skm.REPR_F32, X.to(DEV), d)
        a, dist = skm.skm_assign_segmented(pts, Cf.to(DEV), g, bt)
        ag = a.cpu().numpy()
        for s in range(len(_SEG_SIZES)):
            rows = np.nonzero(group == s)[0]
            Cs = Cf.numpy()[base[s]:base[s + 1]]
            if kind == "bf16":
                ao, best, second = oracle.assign_bf16(xb[rows], Cs)
            else:
                ao, best, second = oracle.assign_f32(X.numpy()[rows], Cs)
            _check_f32(ag[rows] - base[s], dist.cpu().numpy()[rows], best, second, ao, f"segment {s}")
    elif kind == "sq8":
        q = skm.skm_quantize(skm.REPR_SQ8, X.to(DEV))
        codes = q["codes"].cpu().numpy()
        Cc = torch.from_numpy(np.random.default_rng(43).integers(0, 256, (k, d)).astype(np.uint8))
        pts = skm.Points(skm.REPR_SQ8, q["codes"], d)
        a, dist = skm.skm_assign_segmented(pts, Cc.to(DEV), g, bt)
        for s in range(len(_SEG_SIZES)):
            rows = np.nonzero(group == s)[0]
            ao, bo = oracle.assign_sq8(codes[rows], Cc.numpy()[base[s]:base[s + 1]])
            np.testing.assert_array_equal(a.cpu().numpy()[rows] - base[s], ao)
            np.testing.assert_array_equal(dist.cpu().numpy()[rows], bo.astype(np.float32))
    else:
        r = skm.skm_quantize(skm.REPR_RBQ1, X.to(DEV))
        pts = skm.rbq1_points(r, d)
        h = _rbq1_host(r)
        a, est = skm.skm_assign_segmented(pts, Cf.to(DEV), g, bt)
        for s in range(len(_SEG_SIZES)):
            rows = np.nonzero(group == s)[0]
            prep = oracle.rbq1_centroid_sq4(Cf.numpy()[base[s]:base[s + 1]], h["m"])
            ao, eo = oracle.rbq1_assign(h["codes"][rows], h["nx2"][rows], h["F"][rows], h["popx"][rows], d, prep)
            np.testing.assert_array_equal(a.cpu().numpy()[rows] - base[s], ao)
            np.testing.assert_array_equal(est.cpu().numpy()[rows], eo)


# ------------------------------------------------------ hierarchical k-means
def _hier_points(n, d, seed):
    return _points(n, d, seed=seed, ncomp=24)


@pytest.mark.parametrize("refine", [False, True])
def test_fit_hierarchical_sq8_bitexact(skm, refine):
    n, d, k, m = 9000, 64, 60, 8
    X = _hier_points(n, d, 51)
    q = skm.skm_quantize(skm.REPR_SQ8, X.to(DEV))
    codes = q["codes"].cpu().numpy()
    idx = synth.forgy_indices(n, m, seed=51)
    C, a, meso, kf, _ = skm.skm_fit_hierarchical(skm.Points(skm.REPR_SQ8, q["codes"], d), k, m, idx.to(DEV), 3, 4,
                                                 refine=refine)
    Co, ao, amo, kfo = oracle.hierarchical("sq8", codes, k, m, idx.numpy(), 3, 4, refine=refine)
    assert kf == kfo and sum(kf) == k
    np.testing.assert_array_equal(meso.cpu().numpy(), amo)
    np.testing.assert_array_equal(a.cpu().numpy(), ao)
    np.testing.assert_array_equal(C.cpu().numpy(), Co)


def test_fit_hierarchical_rbq1_bitexact(skm):
    n, d, k, m = 8000, 128, 48, 6
    X = _hier_points(n, d, 52)
    r = skm.skm_quantize(skm.REPR_RBQ1, X.to(DEV))
    pts = skm.rbq1_points(r, d)
    h = _rbq1_host(r)
    idx = synth.forgy_indices(n, m, seed=52)
    C, a, meso, kf, _ = skm.skm_fit_hierarchical(pts, k, m, idx.to(DEV), 3, 3)
    data = {"codes": h["codes"], "nx2": h["nx2"], "F": h["F"], "popx": h["popx"], "d": d, "m": h["m"],
            "e": pts.rbq1_exp}
    Co, ao, amo, kfo = oracle.hierarchical("rbq1", data, k, m, idx.numpy(), 3, 3)
    assert kf == kfo
    np.testing.assert_array_equal(meso.cpu().numpy(), amo)
    np.testing.assert_array_equal(a.cpu().numpy(), ao)
    np.testing.assert_array_equal(C.cpu().numpy(), Co)


def test_fit_hierarchical_f32_vs_oracle(skm):
    n, d, k, m = 12000, 48, 64, 8
    X = _hier_points(n, d, 53)
    idx = synth.forgy_indices(n, m, seed=53)
    C, a, meso, kf, _ = skm.skm_fit_hierarchical(skm.Points(skm.REPR_F32, X.to(DEV), d), k, m, idx.to(DEV), 3, 4,
                                                 refine=True)
    Co, ao, amo, kfo = oracle.hierarchical("f32", X.numpy(), k, m, idx.numpy(), 3, 4, refine=True)
    assert (meso.cpu().numpy() == amo).mean() >= AGREE
    if kf == kfo and (meso.cpu().numpy() == amo).all():
        assert (a.cpu().numpy() == ao).mean() >= AGREE
    wg = oracle.objective_f32(X.numpy(), C.cpu().numpy(), a.cpu().numpy())
    wo = oracle.objective_f32(X.numpy(), Co, ao)
    assert abs(wg - wo) / wo <= 1e-3


# ------------------------------------------- host-to-device copy by the SMs
@pytest.mark.parametrize("nbytes,offset", [(6 * 1024 * 1024 + 48, 0), (1000003, 3), (15, 1), (16, 0)])
def test_copy_from_host(skm, nbytes, offset):
    g = torch.Generator().manual_seed(nbytes)
    src_all = torch.randint(0, 256, (nbytes + offset,), dtype=torch.uint8, generator=g).pin_memory()
    src = src_all[offset:]
    dst_all = torch.zeros(nbytes + 1, dtype=torch.uint8, device=DEV)
    dst = dst_all[1:] if offset else dst_all[:nbytes]
    skm.skm_copy_from_host(dst, src)
    torch.cuda.synchronize()
    assert torch.equal(dst.cpu(), src)
    # the guard byte outside the destination is untouched
    assert int(dst_all[0 if offset else nbytes].item()) == 0


def test_copy_from_host_pageable_memory(skm):
    """Ordinary (pageable) host memory: copied where the device addresses all
    host memory (a hardware-coherent host link), else refused before any launch."""
    src = torch.arange(4096, dtype=torch.float32)
    dst = torch.zeros(4096, dtype=torch.float32, device=DEV)
    try:
        skm.skm_copy_from_host(dst, src)
        refused = False
    except skm.SkmError:
        refused = True
    torch.cuda.synchronize()
    if refused:
        assert float(dst.abs().sum().item()) == 0.0
    else:
        assert torch.equal(dst.cpu(), src)


# ------------------------------------- centroids back in the original space
@pytest.mark.parametrize("k,d,dout", [(300, 96, 32), (1000, 1024, 256), (17, 50, 50)])
def test_unproject_vs_oracle(skm, k, d, dout):
    g = torch.Generator().manual_seed(k + d)
    Y = torch.randn(k, dout, generator=g)
    P = torch.randn(d, dout, generator=g)
    mu = torch.randn(d, generator=g)
    X = skm.skm_unproject(Y.to(DEV), P.to(DEV), mu.to(DEV)).cpu().numpy()
    Xo = oracle.unproject(Y.numpy(), P.numpy(), mu.numpy())
    err = np.linalg.norm(X - Xo, axis=1) / np.maximum(np.linalg.norm(Xo, axis=1), 1e-30)
    assert err.max() <= 1e-5


def test_raw_vector_last_update_and_full_dimensional_centroids(skm):
    """RabitQ's raw-vector last update and PCA's approach 1 are an update with
    the raw float32 points and the quantized / projected run's assignment:
    the oracle's mean of members, and (for fixed assignments) no other
    centroids have a lower WCSS."""
    n, d, k = 6000, 128, 40
    X = _points(n, d, seed=61)
    r = skm.skm_quantize(skm.REPR_RBQ1, X.to(DEV))
    pts = skm.rbq1_points(r, d)
    idx = synth.forgy_indices(n, k, seed=61)
    C, a, _, _, _ = skm.skm_fit(pts, k, 4, init_idx=idx.to(DEV))
    Craw, counts = skm.skm_update(skm.Points(skm.REPR_F32, X.to(DEV), d), a, C.clone())
    Co, co = oracle.update_f32(X.numpy(), a.cpu().numpy(), C.cpu().numpy())
    np.testing.assert_array_equal(counts.cpu().numpy(), co)
    rel = np.linalg.norm(Craw.cpu().numpy() - Co, axis=1) / np.maximum(np.linalg.norm(Co, axis=1), 1e-30)
    assert rel.max() <= 1e-4
    ah = a.cpu().numpy()
    assert oracle.objective_f32(X.numpy(), Craw.cpu().numpy(), ah) <= \
        oracle.objective_f32(X.numpy(), C.cpu().numpy(), ah) * (1 + 1e-7)
    # PCA: cluster the projection, then approach 2 (unproject) and approach 1 (members)
    mean, P, _ = skm.skm_pca_fit(X.to(DEV), 32)
    Yp = skm.skm_project(X.to(DEV), P, mean)
    Cp, ap, _, _, _ = skm.skm_fit(skm.Points(skm.REPR_F32, Yp, 32), k, 4, init_idx=idx.to(DEV))
    Cu = skm.skm_unproject(Cp, P, mean).cpu().numpy()
    Cuo = oracle.unproject(Cp.cpu().numpy(), P.cpu().numpy(), mean.cpu().numpy())
    np.testing.assert_allclose(Cu, Cuo, rtol=1e-5, atol=1e-6)
    Cm, _ = skm.skm_update(skm.Points(skm.REPR_F32, X.to(DEV), d), ap, torch.from_numpy(Cu).to(DEV))
    Cmo, _ = oracle.update_f32(X.numpy(), ap.cpu().numpy(), Cu)
    rel = np.linalg.norm(Cm.cpu().numpy() - Cmo, axis=1) / np.maximum(np.linalg.norm(Cmo, axis=1), 1e-30)
    assert rel.max() <= 1e-4


# --------------------------------------------------------------------- LVQ4
def _lvq4_host(q, d):
    words = q["codes"].cpu().numpy().view(np.uint32)
    return {"words": words, "codes": oracle.lvq4_unpack(words, d), "fac": q["lvq"].cpu().numpy()}


@pytest.mark.parametrize("n,d", [(3000, 768), (777, 33), (500, 32), (400, 31), (100, 1), (300, 2048), (333, 36),
                                 (257, 1020), (100, 1024)])
def test_encode_lvq4_bitexact(skm, n, d):
    X = _points(n, d, seed=n + 3)
    q = skm.skm_quantize(skm.REPR_LVQ4, X.to(DEV))
    h = _lvq4_host(q, d)
    codes, fac, _ = oracle.lvq4_encode(X.numpy())
    np.testing.assert_array_equal(h["words"], oracle.lvq4_pack(codes))
    np.testing.assert_array_equal(h["fac"], fac)


@pytest.mark.parametrize("d", [768, 36])
def test_encode_lvq4_half_integer_quotients(skm, d):
    """Quotients (x - b)/s at, and one or two ulps around, every half-integer
    0.5 .. 14.5 (where rounding half to even decides the code), with s = 1 and
    with scales that are not powers of two."""
    g = np.random.default_rng(d)
    rows = []
    for lo, span in [(0.0, 15.0), (-3.25, 1.5), (0.1, 15.0 * 0.37), (1e-3, 2.2e-3)]:
        for _ in range(40):
            s = np.float32(np.float32(span) / np.float32(15.0))
            m = g.integers(0, 30, size=d).astype(np.float32) * np.float32(0.5)
            x = (np.float32(lo) + m * s).astype(np.float32)
            nud = g.integers(-2, 3, size=d)
            for _k in range(2):
                x = np.where(nud > 0, np.nextafter(x, np.float32(np.inf)), x)
                x = np.where(nud < 0, np.nextafter(x, np.float32(-np.inf)), x)
                nud = nud - np.sign(nud)
            x[0], x[1] = np.float32(lo), np.float32(np.float32(lo) + np.float32(span))
            rows.append(x.astype(np.float32))
    X = torch.from_numpy(np.stack(rows))
    q = skm.skm_quantize(skm.REPR_LVQ4, X.to(DEV))
    h = _lvq4_host(q, d)
    codes, fac, _ = oracle.lvq4_encode(X.numpy())
    np.testing.assert_array_equal(h["words"], oracle.lvq4_pack(codes))
    np.testing.assert_array_equal(h["fac"], fac)


@pytest.mark.parametrize("n,d,k", [(3000, 768, 300), (777, 33, 7), (500, 64, 1), (1000, 1024, 65),
                                   (600, 1500, 40), (300, 5, 300), (2100, 128, 513), (1300, 992, 300)])
def test_assign_update_lvq4_bitexact(skm, n, d, k):
    X = _points(n, d, seed=n + 4)
    q = skm.skm_quantize(skm.REPR_LVQ4, X.to(DEV))
    pts = skm.lvq4_points(q, d)
    h = _lvq4_host(q, d)
    assert pts.rbq1_exp == oracle.lvq4_exponent(h["fac"])
    C = X[synth.forgy_indices(n, k, seed=6)].clone()
    a, dist = skm.skm_assign(pts, C.to(DEV))
    ao, do = oracle.lvq4_assign(h["codes"], h["fac"], oracle.lvq4_encode(C.numpy()))
    np.testing.assert_array_equal(a.cpu().numpy(), ao)
    np.testing.assert_array_equal(dist.cpu().numpy(), do)
    Cn, counts = skm.skm_update(pts, a, C.to(DEV).clone())
    Co, co = oracle.lvq4_update(h["codes"], h["fac"], pts.rbq1_exp, ao, C.numpy())
    np.testing.assert_array_equal(counts.cpu().numpy(), co)
    np.testing.assert_array_equal(Cn.cpu().numpy(), Co)


@pytest.mark.parametrize("d", [128, 768, 992])
def test_assign_lvq4_packed_codes_equal_expanded_copy(skm, d):
    """Without a screening copy the tensor-core kernel reads 16-byte aligned
    LVQ4 nibble words packed (converter warps expand each point tile through
    a byte -> two e4m3 codes table); misaligned words or a caller-built copy
    are read from the e4m3 copy.  All give the oracle's result bit for bit."""
    n, k = 3001, 260
    X = _points(n, d, seed=d + 37)
    q = skm.skm_quantize(skm.REPR_LVQ4, X.to(DEV))
    pts = skm.lvq4_points(q, d)
    words = q["codes"].view(torch.int32).reshape(n, -1)
    W = words.shape[1]
    buf = torch.zeros(n * W + 1, dtype=torch.int32, device=DEV)
    buf[1:] = words.reshape(-1)
    off = buf[1:].view(n, W)  # 4 bytes past a 16-byte boundary
    assert off.data_ptr() % 16 == 4 and pts.x.data_ptr() % 16 == 0
    pts_off = skm.Points(skm.REPR_LVQ4, off, d, rbq1_exp=pts.rbq1_exp, lvq=pts.lvq)
    C = X[synth.forgy_indices(n, k, seed=3)].clone().to(DEV)
    a, dist = skm.skm_assign(pts, C)
    a2, dist2 = skm.skm_assign(pts_off, C)
    a3, dist3 = skm.skm_assign(pts.with_screen(), C)
    h = _lvq4_host(q, d)
    ao, do = oracle.lvq4_assign(h["codes"], h["fac"], oracle.lvq4_encode(C.cpu().numpy()))
    np.testing.assert_array_equal(a.cpu().numpy(), ao)
    np.testing.assert_array_equal(dist.cpu().numpy(), do)
    assert torch.equal(a, a2) and torch.equal(dist, dist2)
    assert torch.equal(a, a3) and torch.equal(dist, dist3)


@pytest.mark.parametrize("d", [1024, 777])
def test_assign_lvq4_large_code_products_exact(skm, d):
    """Codes near 15 everywhere (P close to 225 d, the largest the tensor path
    meets): the e4m3 accumulator must still give the exact integer P, seen
    through bit-exact distances."""
    rng = np.random.default_rng(d)
    n, k = 700, 300
    X = np.ones((n, d), np.float32)
    X[np.arange(n), rng.integers(0, d, n)] = 0.0  # one code 0 per row, the rest 15
    X[: n // 2] -= rng.integers(0, 2, (n // 2, d)).astype(np.float32) / 15.0  # codes 14 / 15 mixed
    X[: n // 2, 0] = 0.0
    C = np.ones((k, d), np.float32)
    C[np.arange(k), rng.integers(0, d, k)] = 0.0
    C[k // 2:] -= rng.integers(0, 3, (k - k // 2, d)).astype(np.float32) / 15.0
    q = skm.skm_quantize(skm.REPR_LVQ4, torch.from_numpy(X).to(DEV))
    pts = skm.lvq4_points(q, d)
    h = _lvq4_host(q, d)
    assert h["codes"].mean() > 14.0
    a, dist = skm.skm_assign(pts, torch.from_numpy(C).to(DEV))
    ao, do = oracle.lvq4_assign(h["codes"], h["fac"], oracle.lvq4_encode(C))
    np.testing.assert_array_equal(a.cpu().numpy(), ao)
    np.testing.assert_array_equal(dist.cpu().numpy(), do)


@pytest.mark.parametrize("split", [False, True])
def test_fit_lvq4_trajectory_bitexact(skm, split):
    n, d, k, iters = 8000, 256, 50, 6
    X = _points(n, d, seed=10)
    q = skm.skm_quantize(skm.REPR_LVQ4, X.to(DEV))
    pts = skm.lvq4_points(q, d)
    idx = synth.forgy_indices(n, k, seed=10)
    policy = skm.EMPTY_SPLIT if split else skm.EMPTY_KEEP
    C, a, dist, obj, _ = skm.skm_fit(pts, k, iters, init_idx=idx.to(DEV), empty_policy=policy)
    h = _lvq4_host(q, d)
    C0 = oracle.lvq4_decode_points(h["codes"], h["fac"], pts.rbq1_exp, idx.numpy())
    Co, ao = oracle.lloyd_lvq4(h["codes"], h["fac"], C0, iters, pts.rbq1_exp, split=split)
    np.testing.assert_array_equal(a.cpu().numpy(), ao)
    np.testing.assert_array_equal(C.cpu().numpy(), Co)
    _, do = oracle.lvq4_assign(h["codes"], h["fac"], oracle.lvq4_encode(Co))
    np.testing.assert_array_equal(dist.cpu().numpy(), do)
    assert math.isclose(obj[-1], float(do.astype(np.float64).sum()), rel_tol=1e-12)


def test_sharded_update_lvq4_matches_single(skm):
    n, d, k = 4000, 64, 20
    X = _points(n, d, seed=22)
    q = skm.skm_quantize(skm.REPR_LVQ4, X.to(DEV))
    pts = skm.lvq4_points(q, d)
    C = X[:k].clone().to(DEV)
    a, _ = skm.skm_assign(pts, C)
    C_single, cnt_single = skm.skm_update(pts, a, C.clone())
    total = torch.zeros((k, d + 1), dtype=torch.int64, device=DEV)
    counts = torch.zeros(k, dtype=torch.int64, device=DEV)
    for lo, hi in zip([0, 999, 1000, 3001], [999, 1000, 3001, n]):
        part = torch.zeros((k, d + 1), dtype=torch.int64, device=DEV)
        sp = skm.Points(skm.REPR_LVQ4, pts.x[lo:hi].contiguous(), d, rbq1_exp=pts.rbq1_exp,
                        lvq=pts.lvq[lo:hi].contiguous())
        skm.skm_update(sp, a[lo:hi].contiguous(), None, counts=counts, partial=part)
        skm.skm_merge_partials(total, part)
    C_merged = skm.skm_update_finalize(pts, total, counts, C.clone())
    assert torch.equal(counts, cnt_single)
    assert torch.equal(C_merged, C_single)


def test_assign_segmented_lvq4_per_group(skm):
    group, base = _segments()
    n, k, d = group.size, int(base[-1]), 96
    X = _points(n, d, seed=44)
    Cf = _points(k, d, seed=45)
    q = skm.skm_quantize(skm.REPR_LVQ4, X.to(DEV))
    pts = skm.lvq4_points(q, d)
    h = _lvq4_host(q, d)
    a, dist = skm.skm_assign_segmented(pts, Cf.to(DEV), torch.from_numpy(group).to(DEV),
                                       torch.from_numpy(base).to(DEV))
    for s in range(len(_SEG_SIZES)):
        rows = np.nonzero(group == s)[0]
        ao, do = oracle.lvq4_assign(h["codes"][rows], h["fac"][rows],
                                    oracle.lvq4_encode(Cf.numpy()[base[s]:base[s + 1]]))
        np.testing.assert_array_equal(a.cpu().numpy()[rows] - base[s], ao)
        np.testing.assert_array_equal(dist.cpu().numpy()[rows], do)


@pytest.mark.parametrize("refine", [False, True])
def test_fit_hierarchical_lvq4_bitexact(skm, refine):
    n, d, k, m = 8000, 128, 48, 6
    X = _hier_points(n, d, 53)
    q = skm.skm_quantize(skm.REPR_LVQ4, X.to(DEV))
    pts = skm.lvq4_points(q, d)
    h = _lvq4_host(q, d)
    idx = synth.forgy_indices(n, m, seed=53)
    C, a, meso, kf, _ = skm.skm_fit_hierarchical(pts, k, m, idx.to(DEV), 3, 3, refine=refine)
    data = {"codes": h["codes"], "fac": h["fac"], "e": pts.rbq1_exp}
    Co, ao, amo, kfo = oracle.hierarchical("lvq4", data, k, m, idx.numpy(), 3, 3, refine=refine)
    assert kf == kfo
    np.testing.assert_array_equal(meso.cpu().numpy(), amo)
    np.testing.assert_array_equal(a.cpu().numpy(), ao)
    np.testing.assert_array_equal(C.cpu().numpy(), Co)


# ------------------------------------------------- SQ8 with exact pruning
@pytest.mark.parametrize("n,d,k", [(3000, 256, 300), (777, 33, 13), (500, 1024, 40), (2000, 64, 1)])
def test_prune_sq8_bitexact_and_seed_independent(skm, n, d, k):
    """SuperKMeans on SQ8 codes: integer partial distances make the pruning
    exact, so the result is the oracle's code-space argmin bit for bit,
    whatever seeds the bound."""
    X = _points(n, d, seed=n + d)
    q = skm.skm_quantize(skm.REPR_SQ8, X.to(DEV))
    codes = q["codes"].cpu().numpy()
    Cc = q["codes"][synth.forgy_indices(n, k, seed=8).to(DEV)].clone()
    ao, bo = oracle.assign_sq8(codes, Cc.cpu().numpy())
    pp = skm.Points(skm.REPR_SQ8, q["codes"], d, flags=skm.FLAG_PRUNE)
    a0, d0 = skm.skm_assign(pp, Cc)
    np.testing.assert_array_equal(a0.cpu().numpy(), ao)
    np.testing.assert_array_equal(d0.cpu().numpy(), bo.astype(np.float32))
    prev = torch.randint(0, k, (n,), generator=torch.Generator().manual_seed(9), dtype=torch.int32).to(DEV)
    a1, d1 = skm.skm_assign(pp, Cc, prev_assign=prev)
    assert torch.equal(a1, a0) and torch.equal(d1, d0)


def test_prune_fit_sq8_trajectory_bitexact(skm):
    n, d, k, iters = 6000, 128, 40, 5
    X = _points(n, d, seed=34)
    q = skm.skm_quantize(skm.REPR_SQ8, X.to(DEV))
    codes = q["codes"].cpu().numpy()
    idx = synth.forgy_indices(n, k, seed=34)
    pp = skm.Points(skm.REPR_SQ8, q["codes"], d, flags=skm.FLAG_PRUNE)
    C, a, _, _, st = skm.skm_fit(pp, k, iters, init_idx=idx.to(DEV))
    Co, ao = oracle.lloyd_sq8(codes, codes[idx.numpy()], iters)
    np.testing.assert_array_equal(a.cpu().numpy(), ao)
    np.testing.assert_array_equal(C.cpu().numpy(), Co)
    assert 0 < st["prune_complete"] <= st["prune_first_block"] <= (iters + 1) * n * k


@pytest.mark.parametrize("d", [1024, 1000])
def test_assign_rbq1_extreme_code_sums_exact(skm, d):
    """The tensor path takes 2P - sum ybar straight from the e4m3 accumulator
    (points as +-1): rows whose bits are all 1 or all 0 against centroids whose
    SQ4 codes are almost all 15 push it to +-15 d; the estimates must still
    equal the oracle's bit for bit."""
    rng = np.random.default_rng(d + 1)
    n, k = 512, 256
    X = rng.standard_normal((n, d)).astype(np.float32)
    X[: n // 3] = np.abs(X[: n // 3]) + 0.5  # all residuals > 0 once centred on m = 0
    X[n // 3: 2 * n // 3] = -np.abs(X[n // 3: 2 * n // 3]) - 0.5  # all <= 0
    m = torch.zeros(d, dtype=torch.float32, device=DEV)
    r = skm.skm_quantize(skm.REPR_RBQ1, torch.from_numpy(X).to(DEV), fit=False, m=m)
    pts = skm.rbq1_points(r, d)
    h = _rbq1_host(r)
    C = np.full((k, d), 2.0, np.float32)
    C[np.arange(k), rng.integers(0, d, k)] = -1.0  # one code 0, the rest 15
    C[k // 2:] += rng.integers(0, 2, (k - k // 2, d)).astype(np.float32) * 0.2
    a, est = skm.skm_assign(pts, torch.from_numpy(C).to(DEV))
    prep = oracle.rbq1_centroid_sq4(C, h["m"])
    assert prep[0].mean() > 12.0
    ao, esto = oracle.rbq1_assign(h["codes"], h["nx2"], h["F"], h["popx"], d, prep)
    np.testing.assert_array_equal(a.cpu().numpy(), ao)
    np.testing.assert_array_equal(est.cpu().numpy(), esto)


# ------------------------------------------- symmetric 1-bit (XOR + POPCOUNT)
@pytest.mark.parametrize("n,d,k", [(3000, 768, 300), (777, 33, 7), (1000, 1024, 65), (600, 1500, 40),
                                   (400, 2048, 33)])
def test_assign_rbq1_symmetric_bitexact(skm, n, d, k):
    X = _points(n, d, seed=n + 7)
    r = skm.skm_quantize(skm.REPR_RBQ1, X.to(DEV))
    pts = skm.rbq1_points(r, d).with_flags(skm.FLAG_SYMMETRIC)
    h = _rbq1_host(r)
    C = X[synth.forgy_indices(n, k, seed=11)].clone()
    a, est = skm.skm_assign(pts, C.to(DEV))
    ao, eo = oracle.rbq1_assign_sym(h["codes"], h["nx2"], h["F"], d, oracle.rbq1_centroid_sym(C.numpy(), h["m"]))
    np.testing.assert_array_equal(a.cpu().numpy(), ao)
    np.testing.assert_array_equal(est.cpu().numpy(), eo)


def test_fit_rbq1_symmetric_trajectory_bitexact(skm):
    n, d, k, iters = 8000, 256, 50, 5
    X = _points(n, d, seed=12)
    r = skm.skm_quantize(skm.REPR_RBQ1, X.to(DEV))
    pts = skm.rbq1_points(r, d).with_flags(skm.FLAG_SYMMETRIC)
    idx = synth.forgy_indices(n, k, seed=12)
    C, a, _, _, _ = skm.skm_fit(pts, k, iters, init_idx=idx.to(DEV))
    h = _rbq1_host(r)
    C0 = oracle.rbq1_decode_points(h["codes"], h["F"], d, h["m"], pts.rbq1_exp, idx.numpy())
    Co, ao = oracle.lloyd_rbq1_sym(h["codes"], h["nx2"], h["F"], h["popx"], d, h["m"], C0, iters, pts.rbq1_exp)
    np.testing.assert_array_equal(a.cpu().numpy(), ao)
    np.testing.assert_array_equal(C.cpu().numpy(), Co)


def test_fit_seeded_forgy_matches_oracle(skm):
    """skm_fit with neither C_init nor init_idx draws its Forgy points from
    the seed (STEP 1); the oracle draws its own from the same seed, and the
    SQ8 trajectories from them are bit-exact."""
    n, d, k, iters, seed = 9001, 48, 37, 4, 2**33 + 5
    X = _points(n, d, seed=71)
    q = skm.skm_quantize(skm.REPR_SQ8, X.to(DEV))
    codes = q["codes"].cpu().numpy()
    C, a, _, _, _ = skm.skm_fit(skm.Points(skm.REPR_SQ8, q["codes"], d), k, iters, seed=seed)
    idx = oracle.forgy_indices(seed, n, k)
    Co, ao = oracle.lloyd_sq8(codes, codes[idx], iters)
    np.testing.assert_array_equal(a.cpu().numpy(), ao)
    np.testing.assert_array_equal(C.cpu().numpy(), Co)


def test_fit_balance_statistics(skm):
    """skm_stats: the per-iteration empty-cluster counts and the cluster-size
    standard deviation of the final assignment (the balance column of the
    paper's Table 3) equal the ones of the oracle's SQ8 trajectory (bit-exact
    assignments, so the counts are the same integers)."""
    n, d, k, iters = 3000, 32, 200, 5
    X = _points(n, d, seed=81, ncomp=12)
    q = skm.skm_quantize(skm.REPR_SQ8, X.to(DEV))
    codes = q["codes"].cpu().numpy()
    idx = synth.forgy_indices(n, k, seed=81)
    idx[1:20:2] = idx[0:20:2]  # ten duplicated initial centroids: the higher copies start empty
    _, a, _, _, st = skm.skm_fit(skm.Points(skm.REPR_SQ8, q["codes"], d), k, iters, init_idx=idx.to(DEV))
    Cc = codes[idx.numpy()].copy()
    empties = []
    for _ in range(iters):
        ao, _ = oracle.assign_sq8(codes, Cc)
        Cc, co = oracle.update_sq8(codes, ao, Cc)
        empties.append(int((co == 0).sum()))
    ao, _ = oracle.assign_sq8(codes, Cc)
    np.testing.assert_array_equal(a.cpu().numpy(), ao)
    assert st["empty_per_iter"] == empties and max(empties) > 0
    assert st["empty_clusters"] == empties[-1]
    sizes = np.bincount(ao, minlength=k).astype(np.float64)
    assert math.isclose(st["cluster_size_std"], float(sizes.std()), rel_tol=1e-12)


@pytest.mark.parametrize("d", [768, 33])
def test_sharded_rbq1_mean_codes_and_update_match_single(skm, d):
    """Three uneven row shards: the merged fixed-point mean (shard max |x|,
    scale from the global max and total rows, shard int64 column sums added)
    equals the single-process skm_quantize mean bit for bit, so the shards'
    codes and the merged fused decode-average equal the single-process ones."""
    n, k = 5003, 23
    X = _points(n, d, seed=91).to(DEV)
    whole = skm.skm_quantize(skm.REPR_RBQ1, X)
    bounds = [0, 17, 2950, n]
    shards = [X[lo:hi].contiguous() for lo, hi in zip(bounds[:-1], bounds[1:])]
    amax = max(skm.skm_column_absmax(xs) for xs in shards)
    s = skm.skm_mean_scale(amax, n)
    S = torch.zeros(d, dtype=torch.int64, device=DEV)
    for xs in shards:
        skm.skm_column_sums_fixed(xs, s, S)
    m = skm.skm_mean_from_sums(S, n, s)
    assert torch.equal(m, whole["m"])
    pw = skm.rbq1_points(whole, d)
    C = X[:k].clone()
    a, _ = skm.skm_assign(pw, C)
    C_single, cnt_single = skm.skm_update(pw, a, C.clone())
    total = torch.zeros(k, d + 1, dtype=torch.int64, device=DEV)
    counts = torch.zeros(k, dtype=torch.int64, device=DEV)
    for (lo, hi), xs in zip(zip(bounds[:-1], bounds[1:]), shards):
        q = skm.skm_quantize(skm.REPR_RBQ1, xs, fit=False, m=m.clone())
        assert torch.equal(q["codes"], whole["codes"][lo:hi])
        assert torch.equal(q["F"], whole["F"][lo:hi]) and torch.equal(q["nx2"], whole["nx2"][lo:hi])
        sp = skm.Points(skm.REPR_RBQ1, q["codes"], d, q["nx2"], q["F"], q["popx"], m, pw.rbq1_exp)
        part = torch.zeros(k, d + 1, dtype=torch.int64, device=DEV)
        skm.skm_update(sp, a[lo:hi].contiguous(), None, counts=counts, partial=part)
        skm.skm_merge_partials(total, part)
    C_merged = skm.skm_update_finalize(pw, total, counts, C.clone())
    assert torch.equal(counts, cnt_single) and torch.equal(C_merged, C_single)


# ---------------------------------- SuperKMeans with RabitQ codes (checkpoints)
def _skm_rbq1(skm, n, d, seed):
    X = _points(n, d, seed=seed).to(DEV)
    q = skm.skm_quantize(skm.REPR_RBQ1, X)
    seg = skm.skm_rbq1_segments(X, q["m"])
    pts = skm.rbq1_points(q, d).with_segments(seg).with_flags(skm.FLAG_PRUNE)
    return X, q, seg, pts


@pytest.mark.parametrize("n,d,k", [(3001, 768, 300), (1000, 1024, 129), (777, 200, 40), (500, 128, 7)])
def test_rbq1_segment_pruning_bitexact(skm, n, d, k):
    """Segment factors against the oracle's definitions; the checkpoint-pruned
    assignment and its D3 equal the oracle's bit for bit (the GPU's factors
    handed over) for several seeds of the bound."""
    X, q, seg, pts = _skm_rbq1(skm, n, d, seed=n + d)
    h = _rbq1_host(q)
    nx2o, Fo, pco = oracle.rbq1_seg_encode(X.cpu().numpy(), h["m"])
    segh = tuple(v.cpu().numpy() for v in seg)
    np.testing.assert_allclose(segh[0], nx2o, rtol=1e-6, atol=1e-12)
    np.testing.assert_allclose(segh[1], Fo, rtol=1e-6, atol=1e-12)
    np.testing.assert_array_equal(segh[2], pco)
    C = X[torch.from_numpy(synth.forgy_indices(n, k, seed=3).numpy()).to(DEV)].clone()
    C += 0.05 * torch.randn(C.shape, generator=torch.Generator().manual_seed(4)).to(DEV)
    prep = oracle.rbq1_seg_centroid(C.cpu().numpy(), h["m"])
    a_plain, _ = skm.skm_assign(skm.rbq1_points(q, d), C)
    g = torch.Generator().manual_seed(5)
    for prev in (None, a_plain, torch.randint(0, k, (n,), generator=g, dtype=torch.int32).to(DEV)):
        a, est = skm.skm_assign(pts, C, prev_assign=prev)
        ao, esto = oracle.rbq1_seg_assign(h["codes"], segh, d, prep,
                                          prev=None if prev is None else prev.cpu().numpy())
        np.testing.assert_array_equal(a.cpu().numpy(), ao)
        np.testing.assert_array_equal(est.cpu().numpy(), esto)


def test_fit_rbq1_segment_pruning_trajectory_bitexact(skm):
    """skm_fit with the checkpoints (each iteration's bound from the previous
    assignment) against the oracle's loop of pruned assignments and fused
    decode-average updates: bit-exact, with pruning statistics reported."""
    n, d, k, iters = 4000, 256, 60, 4
    X, q, seg, pts = _skm_rbq1(skm, n, d, seed=77)
    idx = synth.forgy_indices(n, k, seed=7)
    C, a, _, _, st = skm.skm_fit(pts, k, iters, init_idx=idx.to(DEV))
    h = _rbq1_host(q)
    segh = tuple(v.cpu().numpy() for v in seg)
    e = pts.rbq1_exp
    Co = oracle.rbq1_decode_points(h["codes"], h["F"], d, h["m"], e, idx.numpy())
    prev = None
    for _ in range(iters):
        ao, _ = oracle.rbq1_seg_assign(h["codes"], segh, d, oracle.rbq1_seg_centroid(Co, h["m"]), prev=prev)
        Co, _ = oracle.rbq1_update(h["codes"], h["F"], d, h["m"], e, ao, Co)
        prev = ao
    ao, _ = oracle.rbq1_seg_assign(h["codes"], segh, d, oracle.rbq1_seg_centroid(Co, h["m"]), prev=prev)
    np.testing.assert_array_equal(a.cpu().numpy(), ao)
    np.testing.assert_array_equal(C.cpu().numpy(), Co)
    assert 0 < st["prune_complete"] < st["prune_first_block"] < (iters + 1) * n * k


def test_kernel_timer_times_the_tensor_core_launch(skm):
    """skm_kernel_timer: events around each tensor-core kernel launch; the
    last launch's duration is positive and below the whole call's."""
    n, d, k = 50000, 256, 1000
    X = _points(n, d, seed=91)
    Xd = X.to(DEV).to(torch.bfloat16).view(torch.int16)
    C = (Xd[synth.forgy_indices(n, k, seed=3).to(DEV)].to(torch.int32) << 16).view(torch.float32).contiguous()
    pts = skm.Points(skm.REPR_BF16, Xd, d).with_screen()
    ws = skm.workspace(skm.OP_ASSIGN, pts, k)
    skm.skm_assign(pts, C, ws=ws)
    skm.skm_kernel_timer(True)
    try:
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        skm.skm_assign(pts, C, ws=ws)
        e1.record()
        ms = skm.skm_kernel_timer_ms()
        torch.cuda.synchronize()
        assert 0.0 < ms <= e0.elapsed_time(e1)
    finally:
        skm.skm_kernel_timer(False)
