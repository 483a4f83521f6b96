"""Pins for the CPU oracle: each check ties the oracle to something other than
itself (a library routine, a closed form, an invariant, brute force on tiny
inputs, or the hand-worked example in tests/golden/).  No GPU needed."""
import json
import math
import os

import numpy as np
import pytest
import scipy.cluster.vq as vq
from scipy.spatial.distance import cdist

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rng(seed=0):
    return np.random.default_rng(seed)


# ---------------------------------------------------------------- assignment
@pytest.mark.parametrize("d", [1, 31, 32, 33, 64])
@pytest.mark.parametrize("n,k", [(64, 8), (17, 3), (5, 1)])
def test_assign_f32_matches_cdist_brute_force(n, k, d):
    r = _rng(d * 100 + k)
    X = r.standard_normal((n, d)).astype(np.float32)
    C = r.standard_normal((k, d)).astype(np.float32)
    a, best, second = oracle.assign_f32(X, C)
    D = cdist(X.astype(np.float64), C.astype(np.float64), "sqeuclidean")
    np.testing.assert_array_equal(a, np.argmin(D, axis=1))
    np.testing.assert_allclose(best, D.min(axis=1), rtol=1e-12, atol=1e-12)
    if k > 1:
        np.testing.assert_allclose(second, np.sort(D, axis=1)[:, 1], rtol=1e-12, atol=1e-12)
    # invariant: the assigned distance is <= every other centroid's distance
    assert np.all(best[:, None] <= D + 1e-12)


def test_assign_f32_special_cases():
    r = _rng(1)
    X = r.standard_normal((40, 7)).astype(np.float32)
    # K = 1: everything goes to centroid 0
    a, _, _ = oracle.assign_f32(X, X[:1])
    assert np.all(a == 0)
    # N = K with centroids = points: identity assignment, objective 0
    a, best, _ = oracle.assign_f32(X, X)
    np.testing.assert_array_equal(a, np.arange(40))
    assert best.sum() == 0.0
    # duplicate centroids: ties go to the lowest index
    C = np.concatenate([X[3:4], X[3:4], X[5:6], X[5:6]])
    a, _, _ = oracle.assign_f32(X[[3, 5]], C)
    np.testing.assert_array_equal(a, [0, 2])
    # a point exactly halfway between two centroids goes to the lower index
    C = np.array([[1.0, 0.0], [-1.0, 0.0]], np.float32)
    a, _, _ = oracle.assign_f32(np.zeros((1, 2), np.float32), C[::-1].copy())
    assert a[0] == 0


def test_assign_bf16_matches_cdist():
    r = _rng(2)
    Xf = r.standard_normal((50, 33))
    Xb = oracle.round_bf16(Xf)
    C = r.standard_normal((6, 33)).astype(np.float32)
    a, best, _ = oracle.assign_bf16(Xb, C)
    D = cdist(oracle.bf16_to_f32(Xb).astype(np.float64), C.astype(np.float64), "sqeuclidean")
    np.testing.assert_array_equal(a, np.argmin(D, axis=1))
    np.testing.assert_allclose(best, D.min(axis=1), rtol=1e-12)


# -------------------------------------------------------------------- update
def test_update_f32_is_member_mean_and_keeps_empty():
    r = _rng(3)
    X = r.standard_normal((200, 9)).astype(np.float32)
    k = 6
    a = r.integers(0, k - 1, size=200).astype(np.int32)  # cluster k-1 stays empty
    C0 = r.standard_normal((k, 9)).astype(np.float32)
    C, counts = oracle.update_f32(X, a, C0)
    assert counts.sum() == 200 and counts[k - 1] == 0
    for j in range(k - 1):
        np.testing.assert_allclose(C[j], X[a == j].astype(np.float64).mean(axis=0), rtol=1e-6, atol=1e-7)
    np.testing.assert_array_equal(C[k - 1], C0[k - 1])
    # K = 1: the global mean
    C1, _ = oracle.update_f32(X, np.zeros(200, np.int32), C0[:1])
    np.testing.assert_allclose(C1[0], X.astype(np.float64).mean(axis=0), rtol=1e-6, atol=1e-7)


def test_lloyd_f32_matches_scipy_kmeans2_and_is_monotone():
    import synth

    X = synth.gmm_points(3000, 16, 20, seed=5, decay=False).numpy()
    idx = synth.forgy_indices(3000, 20, seed=5).numpy()
    C0 = X[idx].copy()
    C, a, objs = oracle.lloyd_f32(X, C0, 10)
    # scipy's kmeans2 with given initial centroids is the same Lloyd loop
    # (assign, mean of members, empty clusters keep their centroid), in fp64.
    # kmeans2 returns the labels of its last assignment, made before its last
    # update; the final STEP 2 on its returned centroids is vq.vq.
    Cs, _ = vq.kmeans2(X.astype(np.float64), C0.astype(np.float64), iter=10, minit="matrix", missing="warn")
    labs, _ = vq.vq(X.astype(np.float64), Cs)
    assert np.mean(labs == a) > 0.999
    np.testing.assert_allclose(C, Cs, rtol=1e-4, atol=1e-5)
    # Lloyd's objective never increases (fp32 centroids: allow 1e-6 slack)
    for t in range(1, len(objs)):
        assert objs[t] <= objs[t - 1] * (1 + 1e-6)


def test_objective_is_wcss():
    r = _rng(4)
    X = r.standard_normal((100, 5)).astype(np.float32)
    C = r.standard_normal((4, 5)).astype(np.float32)
    a = r.integers(0, 4, 100).astype(np.int32)
    want = float(((X.astype(np.float64) - C[a].astype(np.float64)) ** 2).sum())
    assert math.isclose(oracle.objective_f32(X, C, a), want, rel_tol=1e-12)


# ----------------------------------------------------------------------- SQ8
def test_sq8_grid_data_reproduces_codes():
    r = _rng(6)
    n, d = 300, 37
    codes = r.integers(0, 256, size=(n, d)).astype(np.uint8)
    codes[0, :] = 0
    codes[1, :] = 255
    s0 = (2.0 ** -r.integers(3, 9, size=d)).astype(np.float32)
    b0 = (r.integers(-50, 50, size=d) * s0).astype(np.float32)
    X = (codes.astype(np.float32) * s0 + b0).astype(np.float32)
    b, s = oracle.sq8_fit(X)
    np.testing.assert_array_equal(b, b0)
    np.testing.assert_array_equal(s, s0)
    np.testing.assert_array_equal(oracle.sq8_encode(X, b, s), codes)
    np.testing.assert_array_equal(oracle.sq8_decode(codes, b, s), X)


def test_sq8_roundtrip_error_bound_and_flat_dims():
    r = _rng(7)
    X = r.standard_normal((500, 20)).astype(np.float32)
    X[:, 3] = 0.25  # flat dimension
    b, s = oracle.sq8_fit(X)
    assert s[3] == 1.0 and b[3] == 0.25
    np.testing.assert_array_equal(b, X.min(axis=0))
    codes = oracle.sq8_encode(X, b, s)
    assert codes[:, 3].max() == 0
    np.testing.assert_array_equal(codes.min(axis=0)[np.arange(20) != 3], 0)
    np.testing.assert_array_equal(codes.max(axis=0)[np.arange(20) != 3], 255)
    err = np.abs(oracle.sq8_decode(codes, b, s).astype(np.float64) - X)
    assert np.all(err <= s.astype(np.float64) / 2 * (1 + 1e-5) + 1e-7)


def test_sq4_grid_data_reproduces_codes_and_roundtrip_bound():
    """4-bit codes (Section 3.1 "SQ8 and SQ4"): 15 levels between min and max.
    Data on the grid b + s * code with s a power of two reproduces its codes;
    generic data decodes within s/2 and uses the full 0..15 range."""
    r = _rng(16)
    n, d = 200, 21
    codes = r.integers(0, 16, size=(n, d)).astype(np.uint8)
    codes[0, :] = 0
    codes[1, :] = 15
    s0 = (2.0 ** -r.integers(2, 7, size=d)).astype(np.float32)
    b0 = (r.integers(-40, 40, size=d) * s0).astype(np.float32)
    X = (codes.astype(np.float32) * s0 + b0).astype(np.float32)
    b, s = oracle.sq8_fit(X, bits=4)
    np.testing.assert_array_equal(b, b0)
    np.testing.assert_array_equal(s, s0)
    np.testing.assert_array_equal(oracle.sq8_encode(X, b, s, bits=4), codes)
    Y = r.standard_normal((400, 9)).astype(np.float32)
    b, s = oracle.sq8_fit(Y, bits=4)
    np.testing.assert_allclose(s, (Y.max(0) - Y.min(0)) / np.float32(15), rtol=1e-7)
    c = oracle.sq8_encode(Y, b, s, bits=4)
    assert c.max() == 15 and c.min() == 0
    err = np.abs(oracle.sq8_decode(c, b, s).astype(np.float64) - Y)
    assert np.all(err <= s.astype(np.float64) / 2 * (1 + 1e-5) + 1e-7)


def test_assign_and_update_sq8_exact_integers():
    r = _rng(8)
    Xc = r.integers(0, 256, size=(120, 45)).astype(np.uint8)
    Cc = r.integers(0, 256, size=(7, 45)).astype(np.uint8)
    Cc[5] = Cc[2]  # duplicate: ties to the lower index
    a, best = oracle.assign_sq8(Xc, Cc)
    D = cdist(Xc.astype(np.float64), Cc.astype(np.float64), "sqeuclidean")  # exact below 2^53
    np.testing.assert_array_equal(a, np.argmin(D, axis=1))
    np.testing.assert_array_equal(best, D.min(axis=1).astype(np.int64))
    assert not np.any(a == 5)
    a2 = r.integers(0, 6, 120).astype(np.int32)  # cluster 6 empty
    Cn, counts = oracle.update_sq8(Xc, a2, Cc)
    for j in range(6):
        S = Xc[a2 == j].astype(np.int64).sum(axis=0)
        np.testing.assert_array_equal(Cn[j], np.rint(S / counts[j]).astype(np.uint8))
    np.testing.assert_array_equal(Cn[6], Cc[6])
    # exact halves round to even
    Xh = np.array([[2], [3], [0], [1], [5], [6]], np.uint8)
    Cn, _ = oracle.update_sq8(Xh, np.array([0, 0, 1, 1, 2, 2], np.int32), np.zeros((3, 1), np.uint8))
    np.testing.assert_array_equal(Cn[:, 0], [2, 0, 6])  # 2.5 -> 2, 0.5 -> 0, 5.5 -> 6


# ------------------------------------------------------------------ RabitQ
def _sign_constant_points(r, n, d, m, amp):
    sg = np.where(r.random((n, d)) < 0.5, -1.0, 1.0)
    return (m[None, :].astype(np.float64) + amp[:, None] * sg).astype(np.float32), sg


def test_rbq1_encode_bits_and_factors():
    r = _rng(9)
    n, d = 40, 70
    X = r.standard_normal((n, d)).astype(np.float32)
    m = oracle.rbq1_mean(X)
    np.testing.assert_allclose(m, X.astype(np.float64).mean(axis=0), rtol=1e-6, atol=1e-7)
    codes, nx2, F, popx = oracle.rbq1_encode(X, m)
    R = X - m[None, :]
    bits = (R > 0).astype(np.uint8)
    packed = np.packbits(np.pad(bits, ((0, 0), (0, 96 - d))), axis=1, bitorder="little").view(np.uint32)
    np.testing.assert_array_equal(codes, packed)
    np.testing.assert_array_equal(popx, bits.sum(axis=1))
    R64 = R.astype(np.float64)
    np.testing.assert_allclose(nx2, (R64 ** 2).sum(axis=1), rtol=1e-6)
    # <xbar, x> = ||r||_1 / (sqrt(d) ||r||); F = ||r|| / <xbar, x>
    cosq = np.abs(R64).sum(axis=1) / (math.sqrt(d) * np.linalg.norm(R64, axis=1))
    np.testing.assert_allclose(F, np.linalg.norm(R64, axis=1) / cosq, rtol=1e-6)
    # Cauchy-Schwarz (Section 4, "Closing RabitQ's gap"): decoded radius F >= ||r||
    assert np.all(F >= np.sqrt(nx2) * (1 - 1e-6))
    # degenerate residual r = 0
    _, nx2z, Fz, popz = oracle.rbq1_encode(m[None, :].copy(), m)
    assert nx2z[0] == 0 and Fz[0] == 0 and popz[0] == 0


def test_rbq1_decode_exact_for_sign_constant_residuals():
    r = _rng(10)
    n, d = 30, 96
    m = r.standard_normal(d).astype(np.float32) * 0.1
    amp = r.uniform(0.5, 2.0, n)
    X, sg = _sign_constant_points(r, n, d, m, amp)
    codes, nx2, F, popx = oracle.rbq1_encode(X, m)
    e = oracle.rbq1_exponent(F)
    Cdec = oracle.rbq1_decode_points(codes, F, d, m, e, np.arange(n))
    np.testing.assert_allclose(Cdec, X, rtol=1e-6, atol=1e-6)


def test_rbq1_estimator_matches_direct_sum_and_is_exact_on_grid():
    r = _rng(11)
    n, d, k = 25, 64, 1
    m = np.zeros(d, np.float32)
    amp = r.uniform(0.5, 2.0, n)
    X, sg = _sign_constant_points(r, n, d, m, amp)
    codes, nx2, F, popx = oracle.rbq1_encode(X, m)
    # centroid residual exactly on an SQ4 grid: c - m = b + s * ybar
    yb = r.integers(0, 16, size=d)
    yb[0], yb[1] = 0, 15
    b0, s0 = np.float32(-0.75), np.float32(0.125)
    C = (b0 + s0 * yb.astype(np.float32))[None, :].astype(np.float32)
    prep = oracle.rbq1_centroid_sq4(C, m)
    ybar, b, s, sumy, ny2 = prep
    np.testing.assert_array_equal(ybar[0], yb)
    assert b[0] == b0 and s[0] == s0 and sumy[0] == yb.sum()
    a, est = oracle.rbq1_assign(codes, nx2, F, popx, d, prep)
    # direct form of Eq. final:rabitq: (1/sqrt d) sum (2 xbar_i - 1)(b + s ybar_i), fp64
    xbar = (X - m > 0).astype(np.float64)
    ip = ((2 * xbar - 1) * (float(b[0]) + float(s[0]) * yb)).sum(axis=1) / math.sqrt(d)
    direct = nx2.astype(np.float64) + float(ny2[0]) - 2 * F.astype(np.float64) * ip
    np.testing.assert_allclose(est, direct, rtol=2e-6, atol=2e-5)
    # with sign-constant residuals and an on-grid centroid the estimate is the true distance
    true = cdist(X.astype(np.float64), C.astype(np.float64), "sqeuclidean")[:, 0]
    np.testing.assert_allclose(est, true, rtol=2e-6, atol=2e-5)


def test_blocked_sum_of_squares_is_the_sum_of_squares():
    r = _rng(17)
    for d in (1, 31, 32, 33, 768, 1000):
        v = r.standard_normal(d).astype(np.float32)
        exact = math.fsum(float(x) * float(x) for x in v)
        assert math.isclose(oracle.sumsq_blocked(v), exact, rel_tol=1e-14)
    # order matters only through rounding: a permutation inside a block changes nothing
    v = np.arange(32, dtype=np.float32)
    assert oracle.sumsq_blocked(v) == sum(float(x) ** 2 for x in v)


def test_rbq1_hand_worked_d32_example():
    g = json.load(open(os.path.join(GOLDEN, "rbq1_d32_hand_example.json")))
    d = g["d"]
    bits = np.array([(g["x_bits_word0"] >> i) & 1 for i in range(d)])
    X = np.where(bits == 1, 1.0, -1.0).astype(np.float32)[None, :]
    m = np.zeros(d, np.float32)
    C = (np.arange(d) % 16).astype(np.float32)[None, :]
    codes, nx2, F, popx = oracle.rbq1_encode(X, m)
    assert int(codes[0, 0]) == g["x_bits_word0"]
    assert nx2[0] == g["nx2"] and popx[0] == g["popx"]
    assert math.isclose(float(F[0]), g["F"], rel_tol=1e-7)
    prep = oracle.rbq1_centroid_sq4(C, m)
    assert prep[3][0] == g["sumy"] and prep[4][0] == g["ny2"]
    _, est = oracle.rbq1_assign(codes, nx2, F, popx, d, prep)
    assert math.isclose(float(est[0]), g["estimate"], rel_tol=1e-6)
    assert float(((X - C) ** 2).sum()) == g["true_l2"]


def test_rbq1_update_is_mean_of_decoded_members():
    r = _rng(12)
    n, d, k = 300, 50, 5
    X = r.standard_normal((n, d)).astype(np.float32)
    m = oracle.rbq1_mean(X)
    codes, nx2, F, popx = oracle.rbq1_encode(X, m)
    e = oracle.rbq1_exponent(F)
    mx = float(F.max())
    assert 2.0 ** 23 < mx * 2.0 ** e <= 2.0 ** 24
    a = r.integers(0, k - 1, n).astype(np.int32)  # cluster k-1 empty
    C0 = r.standard_normal((k, d)).astype(np.float32)
    C, counts = oracle.rbq1_update(codes, F, d, m, e, a, C0)
    xbar = (X - m > 0).astype(np.float64)
    dec = m.astype(np.float64) + F.astype(np.float64)[:, None] * (2 * xbar - 1) / math.sqrt(d)
    for j in range(k - 1):
        np.testing.assert_allclose(C[j], dec[a == j].mean(axis=0), rtol=1e-6, atol=1e-7)
    np.testing.assert_array_equal(C[k - 1], C0[k - 1])


def test_rbq1_assign_argmin_of_estimates_brute_force():
    r = _rng(13)
    n, d, k = 60, 40, 7
    X = r.standard_normal((n, d)).astype(np.float32)
    C = r.standard_normal((k, d)).astype(np.float32)
    m = oracle.rbq1_mean(X)
    codes, nx2, F, popx = oracle.rbq1_encode(X, m)
    prep = oracle.rbq1_centroid_sq4(C, m)
    a, est = oracle.rbq1_assign(codes, nx2, F, popx, d, prep)
    ybar, b, s, sumy, ny2 = prep
    xbar = (X - m > 0).astype(np.float64)
    ipd = ((2 * xbar[:, None, :] - 1) * (b[None, :, None] + s[None, :, None] * ybar[None, :, :])).sum(-1) / math.sqrt(d)
    estd = nx2[:, None] + ny2[None, :] - 2 * F[:, None] * ipd
    top2 = np.sort(estd, axis=1)
    clear = (top2[:, 1] - top2[:, 0]) > 1e-3 * np.abs(top2[:, 0]).max()
    np.testing.assert_array_equal(a[clear], np.argmin(estd, axis=1)[clear])


# ------------------------------------------------------- projection and PCA
def test_project_matches_matmul_and_rotation_preserves_distances():
    import synth

    r = _rng(14)
    X = r.standard_normal((40, 24)).astype(np.float32)
    Q = synth.haar_rotation(24, 3).numpy()
    np.testing.assert_allclose(Q.T @ Q, np.eye(24), atol=1e-12)
    mu = X.mean(axis=0).astype(np.float32)
    Y = oracle.project(X, Q.astype(np.float32), mu)
    np.testing.assert_allclose(Y, (X.astype(np.float64) - mu) @ Q.astype(np.float32).astype(np.float64), rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(cdist(Y, Y), cdist(X.astype(np.float64), X.astype(np.float64)), rtol=1e-5, atol=1e-5)


def test_pca_recovers_axes_of_diagonal_covariance():
    r = _rng(15)
    lam = np.array([9.0, 4.0, 2.0, 1.0, 0.25, 0.05])
    X = (r.standard_normal((20000, 6)) * np.sqrt(lam)).astype(np.float32)
    mu0, cov0 = oracle.mean_cov(X)
    np.testing.assert_allclose(cov0, np.cov(X.astype(np.float64).T, bias=True), rtol=1e-9, atol=1e-12)
    mu, P, w = oracle.pca_fit(X, 4)
    np.testing.assert_allclose(np.abs(P), np.eye(6)[:, :4], atol=0.03)
    assert np.all(np.diag(P[:4, :4]) > 0)  # sign fix: largest entry positive
    np.testing.assert_allclose(w, lam[:4], rtol=0.05)
    # full-rank PCA is a rotation: pairwise distances are preserved
    _, Pf, _ = oracle.pca_fit(X[:500], 6)
    Y = oracle.project(X[:50], Pf.astype(np.float32), mu0.astype(np.float32))
    np.testing.assert_allclose(cdist(Y, Y), cdist(X[:50].astype(np.float64), X[:50].astype(np.float64)), rtol=1e-5, atol=1e-5)


def test_round_bf16_matches_torch_and_ties_to_even():
    import torch

    r = _rng(16)
    f = r.standard_normal(4000).astype(np.float32)
    want = torch.from_numpy(f).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(oracle.round_bf16(f.astype(np.float64)), want)
    # exact halfway cases: 1 + 2^-8 lies between 1 and 1 + 2^-7 -> even (1.0)
    got = oracle.round_bf16(np.array([1 + 2.0 ** -8, 1 + 3 * 2.0 ** -8, 1 + 2.0 ** -8 + 2.0 ** -30]))
    np.testing.assert_array_equal(oracle.bf16_to_f32(got), np.array([1.0, 1 + 2.0 ** -6, 1 + 2.0 ** -7], np.float32))


# ----------------------------------------------------- empty-cluster split
def test_split_empty_takes_the_largest_cluster_and_halves_it():
    """Empty clusters 1 and 3 (visited in that order) each split the cluster
    with the most members left (ties to the lowest index): 1 takes half of
    cluster 0 (5 members: 3 stay, 2 move to 1); then cluster 0 (3) is still
    larger than clusters 1 and 2 (2 each), so 3 splits 0 again."""
    rng = np.random.default_rng(3)
    C = rng.normal(size=(5, 6)).astype(np.float32)
    counts = np.array([5, 0, 2, 0, 1], np.int64)
    Cn, ns = oracle.split_empty(C, counts)
    assert ns == 2
    # untouched clusters keep their centroids
    np.testing.assert_array_equal(Cn[2], C[2])
    np.testing.assert_array_equal(Cn[4], C[4])
    # the pair (1, 0) after the first split straddles the old centroid 0:
    # each coordinate moved by a relative 2^-10 in opposite directions
    eps = 2.0 ** -10
    c0 = C[0].astype(np.float64)
    first_j = c0 * np.where(np.arange(6) % 2 == 0, 1 + eps, 1 - eps)
    np.testing.assert_allclose(Cn[1], first_j, rtol=2 ** -23)
    # cluster 3 split the (already moved) cluster 0: midpoint of 3 and 0 is
    # the moved centroid, and 3 differs from 1
    moved0 = c0 * np.where(np.arange(6) % 2 == 0, 1 - eps, 1 + eps)
    mid = (Cn[3].astype(np.float64) + Cn[0].astype(np.float64)) / 2
    np.testing.assert_allclose(mid, moved0, rtol=1e-6)
    assert not np.array_equal(Cn[3], Cn[1])


def test_split_empty_tie_goes_to_lowest_index_and_singletons_are_not_split():
    C = np.arange(12, dtype=np.float32).reshape(4, 3) + 1.0
    Cn, ns = oracle.split_empty(C, np.array([3, 0, 3, 1], np.int64))
    assert ns == 1
    np.testing.assert_array_equal(Cn[2], C[2])  # tie 3 vs 3: cluster 0 is split
    assert not np.array_equal(Cn[0], C[0])
    Cn2, ns2 = oracle.split_empty(C, np.array([1, 0, 1, 0], np.int64))
    assert ns2 == 0
    np.testing.assert_array_equal(Cn2, C)


def test_split_empty_sq8_moves_codes_by_one_step_with_clipping():
    Cc = np.array([[0, 255, 7, 7], [9, 9, 9, 9]], np.uint8)
    Cn, ns = oracle.split_empty(Cc, np.array([4, 0], np.int64))
    assert ns == 1
    np.testing.assert_array_equal(Cn[1], [1, 254, 8, 6])
    np.testing.assert_array_equal(Cn[0], [0, 255, 6, 8])


def test_lloyd_with_split_leaves_no_empty_cluster_on_separated_data():
    """Two far-apart blobs and 4 centroids started inside one blob: without
    splitting, centroids that lose every member stay empty; with splitting
    every centroid ends with members."""
    rng = np.random.default_rng(5)
    X = np.concatenate([rng.normal(0, 0.1, (200, 4)), rng.normal(10, 0.1, (200, 4))]).astype(np.float32)
    C0 = np.concatenate([X[:1] + 100, X[:1] + 101, X[200:203]]).astype(np.float32)
    C, a, _ = oracle.lloyd_f32(X, C0, 6, split=True)
    counts = np.bincount(a, minlength=5)
    assert np.all(counts > 0)
    C2, a2, _ = oracle.lloyd_f32(X, C0, 6, split=False)
    assert np.any(np.bincount(a2, minlength=5) == 0)


# -------------------------------------------------- randomized Hadamard rotation
def test_hadamard_rotate_small_cases_by_hand():
    # D = 2: (x0 s0 + x1 s1, x0 s0 - x1 s1) / sqrt(2)
    X = np.array([[3.0, 1.0]], np.float32)
    Y = oracle.hadamard_rotate(X, np.array([1.0, -1.0], np.float32))
    np.testing.assert_allclose(Y[0], np.array([2.0, 4.0]) / np.sqrt(2), rtol=1e-7)
    # D = 4 with padding of a 3-dimensional row and a mean: rows of H_4 are
    # (1,1,1,1), (1,-1,1,-1), (1,1,-1,-1), (1,-1,-1,1)
    X = np.array([[2.0, 5.0, -1.0]], np.float32)
    mean = np.array([1.0, 1.0, 1.0], np.float32)
    s = np.array([1.0, 1.0, -1.0, 1.0], np.float32)
    v = np.array([1.0, 4.0, 2.0, 0.0])  # (x - mean) * sigma, padded
    H4 = np.array([[1, 1, 1, 1], [1, -1, 1, -1], [1, 1, -1, -1], [1, -1, -1, 1]], np.float64)
    np.testing.assert_allclose(oracle.hadamard_rotate(X, s, mean)[0], H4 @ v / 2.0, rtol=1e-7)


def test_hadamard_rotate_is_orthogonal_and_preserves_distances():
    r = _rng(21)
    X = r.standard_normal((50, 100)).astype(np.float32)
    s = np.where(r.random(128) < 0.5, -1.0, 1.0).astype(np.float32)
    Y = oracle.hadamard_rotate(X, s).astype(np.float64)
    assert Y.shape == (50, 128)
    Xd = X.astype(np.float64)
    np.testing.assert_allclose(np.linalg.norm(Y, axis=1), np.linalg.norm(Xd, axis=1), rtol=1e-6)
    dX = np.linalg.norm(Xd[:, None] - Xd[None], axis=2)
    dY = np.linalg.norm(Y[:, None] - Y[None], axis=2)
    np.testing.assert_allclose(dY, dX, rtol=1e-5, atol=1e-5)
    # the transform of the unit vectors e_i is the i-th column of H D / sqrt(D):
    # entries +-1/sqrt(D), columns mutually orthogonal
    E = np.eye(128, dtype=np.float32)
    T = oracle.hadamard_rotate(E, s).astype(np.float64)
    np.testing.assert_allclose(np.abs(T), 1 / np.sqrt(128), rtol=1e-7)
    np.testing.assert_allclose(T @ T.T, np.eye(128), atol=1e-6)


# ------------------------------------------------------ hierarchical k-means
def test_fine_counts_apportionment():
    # proportional: 10 clusters over sizes 50/30/20 -> 5/3/2 exactly
    assert oracle.fine_counts([50, 30, 20], 10) == [5, 3, 2]
    # largest remainders: 7 over 5/4/1 (N=10): floors 3,2,0 remainders 5,8,7 -> +1 to 1 and 2
    assert oracle.fine_counts([5, 4, 1], 7) == [3, 3, 1]
    # a tiny non-empty cluster still gets one, taken from the largest
    assert oracle.fine_counts([98, 1, 1], 3) == [1, 1, 1]
    assert oracle.fine_counts([990, 5, 5], 10) == [8, 1, 1]
    # empty meso clusters get none; the total is always k
    kf = oracle.fine_counts([0, 40, 0, 60], 9)
    assert kf[0] == 0 and kf[2] == 0 and sum(kf) == 9
    assert oracle.fine_init_positions(10, 4) == [0, 2, 5, 7]


def test_hierarchical_with_one_meso_cluster_is_plain_lloyd():
    """m = 1: every point is in the single meso cluster, so the fine phase is
    vanilla Lloyd with init at evenly spaced points."""
    r = _rng(31)
    X = r.standard_normal((400, 6)).astype(np.float32)
    C, a, am, kf = oracle.hierarchical("f32", X, 5, 1, np.array([0]), 2, 4)
    assert kf == [5] and np.all(am == 0)
    init = np.array(oracle.fine_init_positions(400, 5))
    Cl, al, _ = oracle.lloyd_f32(X, X[init], 4)
    np.testing.assert_array_equal(a, al)
    np.testing.assert_array_equal(C, Cl)


def test_hierarchical_recovers_separated_blobs_and_refine_does_not_hurt():
    """Four far-apart blobs of 3 sub-blobs each, m = 4 meso and k = 12 fine
    clusters: the meso clusters find the blobs (apportioned 3 each), the fine
    phase the sub-blobs; the refinement iteration does not raise the WCSS."""
    r = _rng(32)
    cent = np.array([[0, 0], [100, 0], [0, 100], [100, 100]], np.float64)
    sub = np.array([[0, 0], [6, 0], [0, 6]], np.float64)
    pts = [c + s + r.normal(0, 0.3, (50, 2)) for c in cent for s in sub]
    X = np.concatenate(pts).astype(np.float32)
    meso_init = np.array([0, 150, 300, 450])
    C, a, am, kf = oracle.hierarchical("f32", X, 12, 4, meso_init, 3, 5)
    assert kf == [3, 3, 3, 3]
    labels = np.repeat(np.arange(12), 50)
    for s in range(12):  # each sub-blob maps to a single fine cluster
        assert len(set(a[labels == s])) == 1
    w = oracle.objective_f32(X, C, a)
    C2, a2, _, _ = oracle.hierarchical("f32", X, 12, 4, meso_init, 3, 5, refine=True)
    assert oracle.objective_f32(X, C2, a2) <= w * (1 + 1e-9)


def test_unproject_inverts_a_full_rank_orthogonal_projection():
    """With an orthogonal d x d matrix, unprojecting the projection gives the
    points back; with the top-d' PCA axes of data that lives in d' dimensions
    it gives them back too."""
    r = _rng(41)
    Q, _ = np.linalg.qr(r.standard_normal((12, 12)))
    Q = Q.astype(np.float32)
    X = r.standard_normal((30, 12)).astype(np.float32)
    mu = X.mean(0).astype(np.float32)
    Y = oracle.project(X, Q, mu).astype(np.float32)
    np.testing.assert_allclose(oracle.unproject(Y, Q, mu), X, atol=1e-5)
    # rank-3 data in 8 dims: 3 axes suffice
    B = np.linalg.qr(r.standard_normal((8, 3)))[0].astype(np.float32)
    Z = (r.standard_normal((40, 3)) @ B.T + 2.0).astype(np.float32)
    mz = Z.mean(0).astype(np.float32)
    Yz = oracle.project(Z, B, mz).astype(np.float32)
    np.testing.assert_allclose(oracle.unproject(Yz, B, mz), Z, atol=1e-5)


# ---------------------------------------------------------------- LVQ4
def test_lvq4_hand_example():
    g = json.load(open(os.path.join(GOLDEN, "lvq4_d8_hand_example.json")))
    x = np.array([g["x"]], np.float32)
    y = np.array([g["y"]], np.float32)
    xc, xf, _ = oracle.lvq4_encode(x)
    yc, yf, Gy = oracle.lvq4_encode(y)
    assert xc[0].tolist() == g["xbar"] and yc[0].tolist() == g["ybar"]
    assert tuple(xf[0]) == (g["s_x"], g["b_x"], g["N_x"], g["A_x"])
    assert (yf[0, 0], yf[0, 1], yf[0, 2], Gy[0]) == (g["s_y"], g["b_y"], g["N_y"], g["G_y"])
    assert int((xc[0].astype(np.int64) * yc[0]).sum()) == g["P"]
    a, dist = oracle.lvq4_assign(xc, xf, (yc, yf, Gy))
    assert a[0] == 0 and float(dist[0]) == g["distance"]
    assert float(((x.astype(np.float64) - y) ** 2).sum()) == g["distance"]


def _lvq4_grid(r, n, d):
    """Vectors exactly on their own 15-step grid: power-of-two scale, bias a
    multiple of it, codes 0 and 15 both present in every row."""
    q = r.integers(0, 16, (n, d))
    q[:, 0] = 0
    q[:, 1] = 15
    for p in range(n):
        q[p] = q[p][r.permutation(d)]
    s = 2.0 ** r.integers(-6, 1, n)
    b = s * r.integers(-40, 40, n)
    return (b[:, None] + s[:, None] * q).astype(np.float32), q, s, b


def test_lvq4_encode_grid_exact_and_error_bound():
    r = _rng(40)
    X, q, s, b = _lvq4_grid(r, 50, 37)
    codes, fac, G = oracle.lvq4_encode(X)
    np.testing.assert_array_equal(codes, q)
    np.testing.assert_array_equal(fac[:, 0], s.astype(np.float32))
    np.testing.assert_array_equal(fac[:, 1], b.astype(np.float32))
    # random vectors: codes in range, extremes at 0 and 15, error <= s/2
    X = (r.standard_normal((200, 65)) * r.uniform(0.01, 5, (200, 1)) + r.uniform(-3, 3, (200, 1))).astype(np.float32)
    codes, fac, G = oracle.lvq4_encode(X)
    assert codes.max() <= 15
    np.testing.assert_array_equal(codes[np.arange(200), X.argmin(1)], 0)
    np.testing.assert_array_equal(codes[np.arange(200), X.argmax(1)], 15)
    dec = fac[:, 1:2].astype(np.float64) + fac[:, 0:1].astype(np.float64) * codes
    err = np.abs(dec - X)
    assert np.all(err <= fac[:, 0:1] * (0.5 + 1e-5))
    np.testing.assert_array_equal(fac[:, 1], X.min(1))


def test_lvq4_encode_flat_vector():
    X = np.full((2, 10), 0.75, np.float32)
    X[1] = -3.0
    codes, fac, G = oracle.lvq4_encode(X)
    assert codes.max() == 0
    np.testing.assert_array_equal(fac[:, 0], [1.0, 1.0])
    np.testing.assert_array_equal(fac[:, 1], [0.75, -3.0])
    np.testing.assert_array_equal(fac[:, 2], [10 * 0.75 ** 2, 90.0])
    np.testing.assert_array_equal(fac[:, 3], [7.5, -30.0])
    np.testing.assert_array_equal(G, [0.0, 0.0])


def test_lvq4_terms_are_norm_and_sum_of_decoded_vector():
    r = _rng(41)
    X = (r.standard_normal((100, 96)) + 0.3).astype(np.float32)
    codes, fac, G = oracle.lvq4_encode(X)
    dec = fac[:, 1:2].astype(np.float64) + fac[:, 0:1].astype(np.float64) * codes
    np.testing.assert_allclose(fac[:, 2], (dec ** 2).sum(1), rtol=2e-7)
    np.testing.assert_allclose(fac[:, 3], dec.sum(1), rtol=2e-7, atol=1e-5)
    np.testing.assert_allclose(G, fac[:, 0].astype(np.float64) * codes.sum(1), rtol=1e-7)


def test_lvq4_distance_is_l2_of_decoded_vectors():
    """Eq. final:lvq against the fp64 squared distance of the decoded vectors;
    points and centroids with different scales and biases, so a swapped or
    dropped term shows."""
    r = _rng(42)
    n, k, d = 300, 12, 48
    X = (r.standard_normal((n, d)) * r.uniform(0.5, 2, (n, 1)) + r.uniform(-1, 1, (n, 1))).astype(np.float32)
    C = (r.standard_normal((k, d)) * r.uniform(0.5, 2, (k, 1)) + r.uniform(-1, 1, (k, 1))).astype(np.float32)
    xc, xf, _ = oracle.lvq4_encode(X)
    prep = oracle.lvq4_encode(C)
    yc, yf, _ = prep
    a, dist = oracle.lvq4_assign(xc, xf, prep)
    dx = xf[:, 1:2].astype(np.float64) + xf[:, 0:1] * xc.astype(np.float64)
    dy = yf[:, 1:2].astype(np.float64) + yf[:, 0:1] * yc.astype(np.float64)
    D = cdist(dx, dy, "sqeuclidean")
    scale = xf[:, 2:3].astype(np.float64) + yf[None, :, 2]
    true_best = D[np.arange(n), a]
    assert np.all(np.abs(dist - true_best) <= 1e-5 * scale[np.arange(n), a] + 1e-6)
    srt = np.sort(D, 1)
    ok = a == D.argmin(1)
    gap = (srt[:, 1] - srt[:, 0]) / scale.max(1)
    assert np.all(ok | (gap < 1e-5))
    assert ok.mean() > 0.98


def test_lvq4_exact_grid_assignment_and_ties():
    """Small power-of-two grids make every fp32 step exact: the argmin is the
    brute-force one, duplicated centroids resolve to the lower index."""
    r = _rng(43)
    X, _, _, _ = _lvq4_grid(r, 60, 16)
    C, _, _, _ = _lvq4_grid(r, 5, 16)
    C = np.concatenate([C, C[2:3]])  # centroid 5 duplicates centroid 2
    xc, xf, _ = oracle.lvq4_encode(X)
    a, dist = oracle.lvq4_assign(xc, xf, oracle.lvq4_encode(C))
    D = cdist(X.astype(np.float64), C.astype(np.float64), "sqeuclidean")
    np.testing.assert_array_equal(a, D.argmin(1))
    np.testing.assert_array_equal(dist, D.min(1).astype(np.float32))
    assert not np.any(a == 5)


def test_lvq4_exponent_and_update_is_mean_of_decoded_members():
    r = _rng(44)
    n, d, k = 400, 40, 6
    X = (r.standard_normal((n, d)) + 0.2).astype(np.float32)
    codes, fac, _ = oracle.lvq4_encode(X)
    e = oracle.lvq4_exponent(fac)
    M = float(np.maximum(fac[:, 0], np.abs(fac[:, 1])).max())
    assert 2.0 ** 30 < M * 2.0 ** e <= 2.0 ** 31
    a = r.integers(0, k - 1, n).astype(np.int32)  # cluster k-1 stays empty
    C0 = r.standard_normal((k, d)).astype(np.float32)
    C, counts = oracle.lvq4_update(codes, fac, e, a, C0)
    dec = fac[:, 1:2].astype(np.float64) + fac[:, 0:1] * codes.astype(np.float64)
    for j in range(k - 1):
        np.testing.assert_allclose(C[j], dec[a == j].mean(0), rtol=1e-6, atol=1e-7)
        assert counts[j] == (a == j).sum()
    np.testing.assert_array_equal(C[k - 1], C0[k - 1])
    assert counts[k - 1] == 0
    # K = 1: the global mean of the decoded points
    C1, _ = oracle.lvq4_update(codes, fac, e, np.zeros(n, np.int32), C0[:1])
    np.testing.assert_allclose(C1[0], dec.mean(0), rtol=1e-6, atol=1e-7)
    # members exactly representable in fixed point: the mean is exact
    G, _, _, _ = _lvq4_grid(r, 4, 8)
    gc, gf, _ = oracle.lvq4_encode(G)
    Cg, _ = oracle.lvq4_update(gc, gf, oracle.lvq4_exponent(gf), np.zeros(4, np.int32), np.zeros((1, 8), np.float32))
    np.testing.assert_array_equal(Cg[0], G.astype(np.float64).mean(0).astype(np.float32))


def test_lvq4_pack_layout():
    codes = np.zeros((2, 11), np.uint8)
    codes[0, 0] = 1
    codes[0, 7] = 15
    codes[0, 8] = 3
    codes[1, 10] = 9
    w = oracle.lvq4_pack(codes)
    assert w.shape == (2, 2)
    assert int(w[0, 0]) == 1 | (15 << 28) and int(w[0, 1]) == 3
    assert int(w[1, 1]) == 9 << 8
    r = _rng(45)
    c = r.integers(0, 16, (7, 29)).astype(np.uint8)
    np.testing.assert_array_equal(oracle.lvq4_unpack(oracle.lvq4_pack(c), 29), c)


def test_lloyd_lvq4_points_as_centroids():
    """N = K with the decoded points as initial centroids: every point keeps
    its own centroid (the re-encoded decoded point reproduces its codes)."""
    r = _rng(46)
    X = r.standard_normal((24, 32)).astype(np.float32)
    codes, fac, _ = oracle.lvq4_encode(X)
    e = oracle.lvq4_exponent(fac)
    C0 = oracle.lvq4_decode_points(codes, fac, e, np.arange(24))
    yc, _, _ = oracle.lvq4_encode(C0)
    np.testing.assert_array_equal(yc, codes)
    C, a = oracle.lloyd_lvq4(codes, fac, C0, 3, e=e)
    np.testing.assert_array_equal(a, np.arange(24))


def test_hierarchical_lvq4_one_meso_cluster_equals_lloyd():
    """m = 1: the fine phase is plain LVQ4 Lloyd from the evenly spaced
    members (positions floor(t n / k))."""
    r = _rng(47)
    n, d, k = 600, 24, 6
    X = r.standard_normal((n, d)).astype(np.float32)
    codes, fac, _ = oracle.lvq4_encode(X)
    e = oracle.lvq4_exponent(fac)
    data = {"codes": codes, "fac": fac, "e": e}
    C, a, am, kf = oracle.hierarchical("lvq4", data, k, 1, np.array([3]), 2, 3)
    assert kf == [k] and np.all(am == 0)
    init = (np.arange(k) * n) // k
    C2, a2 = oracle.lloyd_lvq4(codes, fac, oracle.lvq4_decode_points(codes, fac, e, init), 3, e=e)
    np.testing.assert_array_equal(C, C2)
    np.testing.assert_array_equal(a, a2)


# ------------------------------------------------- symmetric 1-bit (XOR + POPCOUNT)
def test_rbq1_symmetric_estimate_matches_formula_and_hamming():
    """Estimate = nx2 + ny2 - 2 F_x F_y (d - 2 h) / d with h the Hamming
    distance of the sign codes (numpy popcount of the XOR), in fp64."""
    r = _rng(48)
    n, d, k = 80, 70, 9
    X = r.standard_normal((n, d)).astype(np.float32)
    C = r.standard_normal((k, d)).astype(np.float32)
    m = oracle.rbq1_mean(X)
    codes, nx2, F, popx = oracle.rbq1_encode(X, m)
    yb, fy, ny2 = oracle.rbq1_centroid_sym(C, m)
    # the centroid side is the point encoder's sign code and factor
    cc, cn2, cF, _ = oracle.rbq1_encode(C, m)
    np.testing.assert_array_equal(yb, cc)
    np.testing.assert_allclose(ny2, cn2, rtol=1e-6)
    np.testing.assert_allclose(fy * d, cF, rtol=1e-5)
    a, est = oracle.rbq1_assign_sym(codes, nx2, F, d, (yb, fy, ny2))
    bx = np.unpackbits(codes.view(np.uint8), axis=1, bitorder="little")[:, :d].astype(np.int64)
    by = np.unpackbits(yb.view(np.uint8), axis=1, bitorder="little")[:, :d].astype(np.int64)
    h = (bx[:, None, :] != by[None, :, :]).sum(-1)
    E = nx2[:, None].astype(np.float64) + ny2[None, :] - 2.0 * F[:, None] * cF[None, :] * (d - 2 * h) / d
    np.testing.assert_allclose(est, E[np.arange(n), a], rtol=2e-5, atol=1e-4)
    srt = np.sort(E, 1)
    clear = (srt[:, 1] - srt[:, 0]) > 1e-4 * np.abs(srt).max()
    np.testing.assert_array_equal(a[clear], E.argmin(1)[clear])


def test_rbq1_symmetric_exact_for_sign_constant_vectors():
    """Residuals of constant magnitude are reconstructed exactly by
    F (2 bit - 1) / sqrt(d), so the symmetric estimate is the true squared
    distance (up to rounding)."""
    r = _rng(49)
    n, k, d = 20, 6, 64
    m = np.zeros(d, np.float32)
    X = (r.choice([-1.0, 1.0], (n, d)) * r.uniform(0.5, 2.0, (n, 1))).astype(np.float32)
    C = (r.choice([-1.0, 1.0], (k, d)) * r.uniform(0.5, 2.0, (k, 1))).astype(np.float32)
    codes, nx2, F, _ = oracle.rbq1_encode(X, m)
    a, est = oracle.rbq1_assign_sym(codes, nx2, F, d, oracle.rbq1_centroid_sym(C, m))
    D = cdist(X.astype(np.float64), C.astype(np.float64), "sqeuclidean")
    np.testing.assert_allclose(est, D[np.arange(n), a], rtol=1e-5)
    np.testing.assert_array_equal(a, D.argmin(1))


# ------------------------------------- hierarchical SQ8 / RBQ1, bf16 update and objective
def test_hierarchical_sq8_with_one_meso_cluster_is_plain_lloyd():
    """m = 1: the fine phase is plain SQ8 Lloyd (pinned against exact integer
    means above) from the evenly spaced members floor(t n / k)."""
    r = _rng(51)
    n, d, k = 500, 12, 7
    codes = r.integers(0, 256, (n, d)).astype(np.uint8)
    C, a, am, kf = oracle.hierarchical("sq8", codes, k, 1, np.array([4]), 2, 4)
    assert kf == [k] and np.all(am == 0)
    init = np.array(oracle.fine_init_positions(n, k))
    Cl, al = oracle.lloyd_sq8(codes, codes[init], 4)
    np.testing.assert_array_equal(a, al)
    np.testing.assert_array_equal(C, Cl)


def test_hierarchical_rbq1_with_one_meso_cluster_is_plain_lloyd():
    """m = 1: the fine phase is plain RabitQ Lloyd from the decoded evenly
    spaced members."""
    r = _rng(52)
    n, d, k = 400, 40, 5
    X = r.standard_normal((n, d)).astype(np.float32)
    m = oracle.rbq1_mean(X)
    codes, nx2, F, popx = oracle.rbq1_encode(X, m)
    e = oracle.rbq1_exponent(F)
    data = {"codes": codes, "nx2": nx2, "F": F, "popx": popx, "d": d, "m": m, "e": e}
    C, a, am, kf = oracle.hierarchical("rbq1", data, k, 1, np.array([7]), 2, 3)
    assert kf == [k] and np.all(am == 0)
    init = np.array(oracle.fine_init_positions(n, k))
    C0 = oracle.rbq1_decode_points(codes, F, d, m, e, init)
    Cl, al = oracle.lloyd_rbq1(codes, nx2, F, popx, d, m, C0, 3, e)
    np.testing.assert_array_equal(a, al)
    np.testing.assert_array_equal(C, Cl)


def _blobs(r, d, sep, sub, noise, per=50):
    """Four far-apart blobs of three sub-blobs each (labels 0..11 in order):
    blob centres sep * e_b, sub-blob offsets sub * e_{4 + s} along axes of
    their own, isotropic Gaussian noise."""
    pts, labels = [], []
    for b in range(4):
        for s in range(3):
            c = np.zeros(d)
            c[b] = sep
            c[4 + 3 * b + s] = sub
            pts.append(c + r.normal(0, noise, (per, d)))
            labels.append(np.full(per, 3 * b + s))
    return np.concatenate(pts).astype(np.float32), np.concatenate(labels)


def _assert_blobs_recovered(a, am, kf, labels):
    assert kf == [3, 3, 3, 3]
    for b in range(4):  # each blob is one meso cluster
        assert len(set(am[labels // 3 == b])) == 1
    for s in range(12):  # each sub-blob is one fine cluster, and they are distinct
        assert len(set(a[labels == s])) == 1
    assert len({int(a[labels == s][0]) for s in range(12)}) == 12


def test_hierarchical_sq8_recovers_separated_blobs():
    """SQ8 codes of four far-apart blobs of three sub-blobs each, m = 4 meso
    and k = 12 fine clusters: meso clusters are the blobs (3 fine clusters
    each), fine clusters the sub-blobs."""
    r = _rng(53)
    X, labels = _blobs(r, 16, 100.0, 20.0, 0.5)
    b, s = oracle.sq8_fit(X)
    codes = oracle.sq8_encode(X, b, s)
    meso_init = np.array([0, 150, 300, 450])
    C, a, am, kf = oracle.hierarchical("sq8", codes, 12, 4, meso_init, 3, 5)
    _assert_blobs_recovered(a, am, kf, labels)
    C2, a2, _, _ = oracle.hierarchical("sq8", codes, 12, 4, meso_init, 3, 5, refine=True)
    np.testing.assert_array_equal(a2, a)  # a fixed point: refinement changes nothing


def _sign_blobs(r, per=50):
    """Four blobs of three sub-blobs each (labels 0..11 in order) for 1-bit
    codes, which see only the signs of x - m: on dimensions 0..31 each blob
    has a +-30 pattern (every dimension + for two blobs and - for the other
    two, so the data mean is 0 there), on dimensions 32..63 each sub-blob a
    pattern of +10, -10 and 0 (a permutation per blob and dimension, mean 0),
    plus Gaussian noise 0.5.  Blobs are then ~8x farther apart than
    sub-blobs, and every blob and sub-blob has a sign code of its own."""
    pats = [(1, 1, -1, -1), (1, -1, 1, -1), (1, -1, -1, 1), (-1, -1, 1, 1), (-1, 1, -1, 1), (-1, 1, 1, -1)]
    B = np.array([pats[r.integers(0, 6)] for _ in range(32)], np.float64).T * 30.0  # [4][32]
    S = np.zeros((4, 3, 32))
    for b in range(4):
        for i in range(32):
            S[b, :, i] = r.permutation([10.0, -10.0, 0.0])
    pts, labels = [], []
    for b in range(4):
        for s in range(3):
            c = np.concatenate([B[b], S[b, s]])
            pts.append(c + r.normal(0, 0.5, (per, 64)))
            labels.append(np.full(per, 3 * b + s))
    return np.concatenate(pts).astype(np.float32), np.concatenate(labels)


def test_hierarchical_rbq1_recovers_separated_blobs():
    """Blobs and sub-blobs with sign codes of their own, as RabitQ 1-bit
    codes (d = 64), m = 4 meso and k = 12 fine clusters: meso clusters are
    the blobs, fine clusters the sub-blobs."""
    r = _rng(54)
    X, labels = _sign_blobs(r)
    m = oracle.rbq1_mean(X)
    codes, nx2, F, popx = oracle.rbq1_encode(X, m)
    e = oracle.rbq1_exponent(F)
    data = {"codes": codes, "nx2": nx2, "F": F, "popx": popx, "d": 64, "m": m, "e": e}
    meso_init = np.array([0, 150, 300, 450])
    C, a, am, kf = oracle.hierarchical("rbq1", data, 12, 4, meso_init, 3, 5)
    _assert_blobs_recovered(a, am, kf, labels)


def test_update_bf16_is_member_mean_of_decoded_rows_and_keeps_empty():
    r = _rng(55)
    n, d, k = 300, 21, 6
    Xb = oracle.round_bf16(r.standard_normal((n, d)))
    Xf = oracle.bf16_to_f32(Xb).astype(np.float64)
    a = r.integers(0, k - 1, n).astype(np.int32)  # cluster k-1 stays empty
    C0 = r.standard_normal((k, d)).astype(np.float32)
    C, counts = oracle.update_bf16(Xb, a, C0)
    np.testing.assert_array_equal(counts, np.bincount(a, minlength=k))
    for j in range(k - 1):
        np.testing.assert_allclose(C[j], Xf[a == j].mean(axis=0), rtol=1e-6, atol=1e-7)
    np.testing.assert_array_equal(C[k - 1], C0[k - 1])


def test_objective_bf16_is_wcss_of_decoded_rows():
    r = _rng(56)
    n, d, k = 120, 19, 5
    Xb = oracle.round_bf16(r.standard_normal((n, d)))
    C = r.standard_normal((k, d)).astype(np.float32)
    a = r.integers(0, k, n).astype(np.int32)
    D = cdist(oracle.bf16_to_f32(Xb).astype(np.float64), C.astype(np.float64), "sqeuclidean")
    want = float(D[np.arange(n), a].sum())
    assert math.isclose(oracle.objective_bf16(Xb, C, a), want, rel_tol=1e-12)


# ------------------------------------------------------- seeded Forgy (STEP 1)
def test_philox4x32_10_known_answer_vectors():
    """The published known-answer vectors of Philox4x32-10 (Salmon et al.,
    SC'11; the Random123 distribution's kat_vectors)."""
    kat = [((0, 0, 0, 0), (0, 0), (0x6627E8D5, 0xE169C58D, 0xBC57AC4C, 0x9B00DBD8)),
           ((0xFFFFFFFF,) * 4, (0xFFFFFFFF,) * 2, (0x408F276D, 0x41C83B0E, 0xA20BC7C6, 0x6D5451FD)),
           ((0x243F6A88, 0x85A308D3, 0x13198A2E, 0x03707344), (0xA4093822, 0x299F31D0),
            (0xD16CFE09, 0x94FDCCEB, 0x5001E420, 0x24126EA1))]
    for ctr, key, want in kat:
        assert tuple(int(v) for v in oracle.philox4x32_10(ctr, key)) == want


def test_forgy_indices_are_a_permutation_prefix():
    for seed in (0, 1, 2**40 + 7):
        full = oracle.forgy_indices(seed, 1000, 1000)
        assert sorted(full.tolist()) == list(range(1000))  # k = n: a permutation
        part = oracle.forgy_indices(seed, 1000, 37)
        np.testing.assert_array_equal(part, full[:37])  # a prefix of the same permutation
    a = oracle.forgy_indices(5, 10_000_000, 1000)
    assert len(set(a.tolist())) == 1000 and a.min() >= 0 and a.max() < 10_000_000
    assert not np.array_equal(oracle.forgy_indices(6, 10_000_000, 1000), a)
    assert oracle.forgy_indices(9, 1, 1).tolist() == [0]


def test_forgy_indices_are_uniform():
    """First and second entries over 20,000 seeds with n = 10: every value
    (and every ordered pair) about equally often (chi-square)."""
    from scipy.stats import chisquare

    n, trials = 10, 20_000
    first = np.empty(trials, np.int64)
    second = np.empty(trials, np.int64)
    for s in range(trials):
        f = oracle.forgy_indices(s, n, 2)
        first[s], second[s] = f
    assert np.all(first != second)
    assert chisquare(np.bincount(first, minlength=n)).pvalue > 1e-4
    pairs = np.bincount(first * n + second, minlength=n * n).reshape(n, n)
    off = pairs[~np.eye(n, dtype=bool)]
    assert chisquare(off).pvalue > 1e-4


# ------------------------------------------ RabitQ dataset mean in fixed point
def test_mean_scale_by_hand():
    # 1.0 = 0.5 * 2^1 -> E = 1; n = 1 -> L = 0; s = 61 - 0 - 1
    assert oracle.mean_scale(1.0, 1) == 60
    assert oracle.mean_scale(0.75, 1024) == 61 - 10 - 0
    assert oracle.mean_scale(0.75, 1025) == 61 - 11 - 0
    assert oracle.mean_scale(0.0, 100) == 0
    assert oracle.mean_scale(2.0 ** -140, 2) == 61 - 1 + 139  # 2^-140 = 0.5 * 2^-139


def test_rbq1_mean_is_the_mean_within_the_fixed_point_bound():
    r = _rng(57)
    n, d = 1000, 13
    X = (r.standard_normal((n, d)) * np.logspace(-3, 1, d)).astype(np.float32)
    m = oracle.rbq1_mean(X)
    s = oracle.mean_scale(float(np.abs(X).max()), n)
    exact = X.astype(np.float64).mean(axis=0)
    bound = 2.0 ** -(s + 1) + np.abs(exact) * 2.0 ** -24 + 1e-300
    assert np.all(np.abs(m.astype(np.float64) - exact) <= bound)


def test_rbq1_mean_of_grid_data_is_exact():
    """Coordinates on a 2^-10 grid: the fixed-point sums are the exact sums,
    so m is the fp64 mean (exact sum, one division) rounded to fp32."""
    r = _rng(58)
    X = (r.integers(-4000, 4000, (777, 11)) / 1024.0).astype(np.float32)
    want = (X.astype(np.float64).sum(axis=0) / 777).astype(np.float32)
    np.testing.assert_array_equal(oracle.rbq1_mean(X), want)


def test_rbq1_mean_shard_sums_add_up():
    """Uneven row shards summed at the global scale give the whole-data sums,
    hence the single-process mean bit for bit."""
    r = _rng(59)
    X = r.standard_normal((1001, 17)).astype(np.float32)
    s = oracle.mean_scale(float(np.abs(X).max()), 1001)
    parts = [X[:13], X[13:600], X[600:]]
    S = sum(oracle.column_sums_fixed(p, s) for p in parts)
    np.testing.assert_array_equal(S, oracle.column_sums_fixed(X, s))
    np.testing.assert_array_equal(oracle.mean_from_sums(S, 1001, s), oracle.rbq1_mean(X))


# ---------------------------------- SuperKMeans with RabitQ: segment estimates
def test_rbq1_seg_bounds():
    assert oracle.rbq1_seg_bounds(1024) == (128, 256)  # 12.5% and 25% of d
    assert oracle.rbq1_seg_bounds(768) == (96, 192)
    assert oracle.rbq1_seg_bounds(128) == (32, 64)


def test_rbq1_seg_factors_are_their_definitions():
    r = _rng(61)
    n, d = 30, 256
    X = r.standard_normal((n, d)).astype(np.float32)
    m = oracle.rbq1_mean(X)
    d1, d2 = oracle.rbq1_seg_bounds(d)
    nx2, F, pc = oracle.rbq1_seg_encode(X, m)
    R = X.astype(np.float64) - m.astype(np.float64)
    for t, (lo, hi) in enumerate([(0, d1), (d1, d2), (d2, d)]):
        Rt = R[:, lo:hi]
        s2, s1 = (Rt ** 2).sum(1), np.abs(Rt).sum(1)
        np.testing.assert_allclose(nx2[:, t], s2, rtol=1e-6)
        np.testing.assert_allclose(F[:, t], math.sqrt(hi - lo) * s2 / s1, rtol=1e-6)
        np.testing.assert_array_equal(pc[:, t], ((X[:, lo:hi] - m[lo:hi]) > 0).sum(1))


def test_rbq1_seg_whole_d_is_plain_rabitq():
    """One segment spanning all of d (the other two empty): the segment
    estimate is the plain RabitQ estimate, and with the bound from centroid 0
    the pruned argmin is the plain argmin."""
    r = _rng(62)
    n, d, k = 200, 96, 9
    X = r.standard_normal((n, d)).astype(np.float32)
    C = r.standard_normal((k, d)).astype(np.float32)
    m = oracle.rbq1_mean(X)
    codes, nx2, F, popx = oracle.rbq1_encode(X, m)
    seg = oracle.rbq1_seg_encode(X, m, bounds=(d, d))
    np.testing.assert_array_equal(seg[0][:, 0], nx2)
    np.testing.assert_array_equal(seg[1][:, 0], F)
    np.testing.assert_array_equal(seg[2][:, 0], popx)
    a0, e0 = oracle.rbq1_assign(codes, nx2, F, popx, d, oracle.rbq1_centroid_sq4(C, m))
    a1, e1 = oracle.rbq1_seg_assign(codes, seg, d, oracle.rbq1_seg_centroid(C, m, bounds=(d, d)), bounds=(d, d))
    np.testing.assert_array_equal(a1, a0)
    np.testing.assert_array_equal(e1, e0)


def test_rbq1_seg_estimates_exact_on_grid_and_pruning_keeps_the_nearest():
    """Residuals of constant magnitude within each segment (the 1-bit code
    then reconstructs each segment exactly) and centroids on SQ4 grids: every
    segment estimate is the exact segment distance, the partial estimates are
    partial distances, and the checkpoint pruning with the exact test (g = 1)
    returns the true nearest centroid whatever the seed of its bound."""
    r = _rng(63)
    n, d, k = 60, 256, 8
    d1, d2 = oracle.rbq1_seg_bounds(d)
    m = np.zeros(d, np.float32)
    amp = np.empty((n, d), np.float64)
    for lo, hi in [(0, d1), (d1, d2), (d2, d)]:
        amp[:, lo:hi] = r.uniform(0.25, 2.0, (n, 1))
    X = (amp * np.where(r.random((n, d)) < 0.5, -1.0, 1.0)).astype(np.float32)
    yb = r.integers(0, 16, (k, d))
    yb[:, 0], yb[:, 1] = 0, 15
    b0 = r.choice([-1.0, -0.75, -0.5], k).astype(np.float32)
    s0 = r.choice([0.0625, 0.125, 0.25], k).astype(np.float32)
    C = (b0[:, None] + s0[:, None] * yb).astype(np.float32)
    seg = oracle.rbq1_seg_encode(X, m)
    prep = oracle.rbq1_seg_centroid(C, m)
    codes, _, _, _ = oracle.rbq1_encode(X, m)
    true = cdist(X.astype(np.float64), C.astype(np.float64), "sqeuclidean")
    want = np.argmin(true, axis=1)
    gap = np.sort(true, axis=1)
    assert np.all(gap[:, 1] - gap[:, 0] > 1e-3 * gap[:, 0])  # no near ties
    for prev in (None, np.zeros(n, np.int32), np.full(n, k - 1, np.int32), want.astype(np.int32),
                 r.integers(0, k, n).astype(np.int32)):
        a, est = oracle.rbq1_seg_assign(codes, seg, d, prep, prev=prev, g=np.ones(2, np.float32))
        np.testing.assert_array_equal(a, want)
        np.testing.assert_allclose(est, true[np.arange(n), want], rtol=1e-5)


def test_rbq1_seg_pruning_rule_brute_force():
    """The scaled checkpoint test (ADSampling's factors) against the rule
    restated over every pair's partial estimates: the candidates are the seed
    and every centroid whose partial estimates stay <= fl32(beta g_t), the
    result the candidate with the smallest D3 (lowest index on ties)."""
    r = _rng(64)
    n, d, k = 50, 256, 40
    X = r.standard_normal((n, d)).astype(np.float32)
    C = (X[r.integers(0, n, k)] + 0.3 * r.standard_normal((k, d))).astype(np.float32)
    m = oracle.rbq1_mean(X)
    codes, _, _, _ = oracle.rbq1_encode(X, m)
    seg = oracle.rbq1_seg_encode(X, m)
    prep = oracle.rbq1_seg_centroid(C, m)
    D = oracle.rbq1_seg_partials(codes, seg, d, prep)
    g = oracle.rbq1_seg_factors(d)
    assert 0 < g[0] < g[1] < 1
    prev = r.integers(0, k, n).astype(np.int32)
    a, est = oracle.rbq1_seg_assign(codes, seg, d, prep, prev=prev)
    pruned = 0
    for p in range(n):
        beta = D[p, prev[p], 2]
        keep = (D[p, :, 0] <= np.float32(beta * g[0])) & (D[p, :, 1] <= np.float32(beta * g[1]))
        keep[prev[p]] = True
        pruned += int((~keep).sum())
        cand = np.nonzero(keep)[0]
        want = cand[np.argmin(D[p, cand, 2])]  # np.argmin takes the first (lowest index) on ties
        assert a[p] == want and est[p] == D[p, want, 2]
    assert pruned > 0
    # with no pruning (g = +inf) the result is the argmin of D3 over all centroids
    a_all, _ = oracle.rbq1_seg_assign(codes, seg, d, prep, prev=prev, g=np.full(2, np.inf, np.float32))
    np.testing.assert_array_equal(a_all, np.argmin(D[:, :, 2], axis=1))
