"""CPU oracle for the Lloyd k-means hot path (test infrastructure only).

Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg may import
this package.  It never imports the CUDA library or its Python binding, and the
CUDA path never imports it.

The arithmetic lives in skm_oracle.c (plain C, -O2 -ffp-contract=off, OpenMP
over rows); this module compiles it with gcc on first use, wraps each function
for numpy arrays, and composes the Lloyd loop of Section 2.3 (STEP 2 and STEP 3
repeated, then STEP 2 once more) for each representation.  The PCA
eigen-decomposition is numpy.linalg.eigh on the fp64 covariance (a library
routine used as one step), sorted by descending eigenvalue with each
eigenvector's sign fixed so that its largest-magnitude entry is positive.

Parity status: every function is pinned by tests/test_oracle_pins.py except the
paper's printed dataset-level numbers (WCSS, recall), which need the paper's
datasets: parity unpinned for those.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "skm_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liboracle.so")
_lock = threading.Lock()
_lib = None

GCC_FLAGS = ["-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-ffp-contract=off", "-fno-fast-math"]


def build(force: bool = False) -> str:
    """Compile skm_oracle.c into oracle/_build/liboracle.so (gcc)."""
    os.makedirs(_BUILD, exist_ok=True)
    stale = (not os.path.exists(_LIB_PATH)) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC)
    if force or stale:
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", *GCC_FLAGS, _SRC, "-o", tmp, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _p(a):
    return a.ctypes.data_as(ctypes.c_void_p) if a is not None else None


def lib():
    global _lib
    with _lock:
        if _lib is None:
            build()
            L = ctypes.CDLL(_LIB_PATH)
            vp, i64, i32, f64 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_double
            sig = {
                "or_num_threads": ([], i32),
                "or_set_num_threads": ([i32], None),
                "or_assign_f32": ([vp, i64, i32, vp, i32, vp, vp, vp], None),
                "or_assign_bf16": ([vp, i64, i32, vp, i32, vp, vp, vp], None),
                "or_sq8_fit": ([vp, i64, i32, vp, vp], None),
                "or_sq8_encode": ([vp, i64, i32, vp, vp, vp], None),
                "or_sq_fit": ([vp, i64, i32, i32, vp, vp], None),
                "or_sq_encode": ([vp, i64, i32, i32, vp, vp, vp], None),
                "or_sq8_decode": ([vp, i64, i32, vp, vp, vp], None),
                "or_assign_sq8": ([vp, i64, i32, vp, i32, vp, vp], None),
                "or_update_sq8": ([vp, i64, i32, vp, i32, vp, vp], None),
                "or_update_f32": ([vp, i64, i32, vp, i32, vp, vp], None),
                "or_update_bf16": ([vp, i64, i32, vp, i32, vp, vp], None),
                "or_objective_f32": ([vp, i64, i32, vp, vp], f64),
                "or_objective_bf16": ([vp, i64, i32, vp, vp], f64),
                "or_rbq1_mean": ([vp, i64, i32, vp], None),
                "or_rbq1_encode": ([vp, i64, i32, vp, vp, vp, vp, vp], None),
                "or_rbq1_centroid_sq4": ([vp, i32, i32, vp, vp, vp, vp, vp, vp], None),
                "or_rbq1_assign": ([vp, vp, vp, vp, i64, i32, vp, vp, vp, vp, vp, i32, vp, vp], None),
                "or_rbq1_exponent": ([vp, i64], i32),
                "or_rbq1_centroid_sym": ([vp, i32, i32, vp, vp, vp, vp], None),
                "or_rbq1_assign_sym": ([vp, vp, vp, i64, i32, vp, vp, vp, i32, vp, vp], None),
                "or_rbq1_update": ([vp, vp, i64, i32, vp, i32, vp, i32, vp, vp], None),
                "or_project": ([vp, i64, i32, vp, vp, i32, vp], None),
                "or_mean_cov": ([vp, i64, i32, vp, vp], None),
                "or_round_bf16": ([vp, i64, vp], None),
                "or_sumsq_blocked": ([vp, i32], f64),
                "or_split_empty_f32": ([vp, vp, i32, i32], i32),
                "or_hadamard_rotate": ([vp, i64, i32, vp, vp, i32, vp], None),
                "or_unproject": ([vp, i64, i32, vp, vp, i32, vp], None),
                "or_split_empty_sq8": ([vp, vp, i32, i32], i32),
                "or_lvq4_encode": ([vp, i64, i32, vp, vp, vp], None),
                "or_lvq4_assign": ([vp, vp, i64, i32, vp, vp, vp, i32, vp, vp], None),
                "or_lvq4_exponent": ([vp, i64], i32),
                "or_lvq4_update": ([vp, vp, i64, i32, i32, vp, i32, vp, vp], None),
                "or_philox4x32_10": ([vp, vp, vp], None),
                "or_mean_scale": ([ctypes.c_float, i64], i32),
                "or_rbq1_seg_bounds": ([i32, vp, vp], None),
                "or_rbq1_seg_encode": ([vp, i64, i32, vp, i32, i32, vp, vp, vp], None),
                "or_rbq1_seg_centroid": ([vp, i32, i32, vp, i32, i32, vp, vp, vp, vp, vp], None),
                "or_rbq1_seg_assign": ([vp, vp, vp, vp, i64, i32, i32, i32, vp, vp, vp, vp, vp, i32, vp, vp, vp,
                                        vp], None),
                "or_rbq1_seg_factors": ([i32, i32, i32, f64, vp], None),
                "or_rbq1_seg_partials": ([vp, vp, vp, vp, i64, i32, i32, i32, vp, vp, vp, vp, vp, i32, vp], None),
                "or_column_sums_fixed": ([vp, i64, i32, i32, vp], None),
                "or_mean_from_sums": ([vp, i64, i32, i32, vp], None),
                "or_forgy_indices": ([ctypes.c_uint64, i64, i32, vp], None),
            }
            for name, (args, res) in sig.items():
                fn = getattr(L, name)
                fn.argtypes = args
                fn.restype = res
            _lib = L
    return _lib


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def num_threads() -> int:
    return int(lib().or_num_threads())


def set_num_threads(t: int) -> None:
    lib().or_set_num_threads(int(t))


# --------------------------------------------------------------------------
# STEP 2 (Section 2.3): nearest centroid, plain definition
# --------------------------------------------------------------------------
def assign_f32(X, C):
    """Returns (assign int32[n], best fp64[n], second fp64[n])."""
    X, C = _c(X, np.float32), _c(C, np.float32)
    n, d = X.shape
    k = C.shape[0]
    a = np.empty(n, np.int32)
    b1 = np.empty(n, np.float64)
    b2 = np.empty(n, np.float64)
    lib().or_assign_f32(_p(X), n, d, _p(C), k, _p(a), _p(b1), _p(b2))
    return a, b1, b2


def assign_bf16(Xb, C):
    """Points as bf16 bit patterns (uint16 [n, d]); returns (assign, best, second)."""
    Xb, C = _c(Xb, np.uint16), _c(C, np.float32)
    n, d = Xb.shape
    k = C.shape[0]
    a = np.empty(n, np.int32)
    b1 = np.empty(n, np.float64)
    b2 = np.empty(n, np.float64)
    lib().or_assign_bf16(_p(Xb), n, d, _p(C), k, _p(a), _p(b1), _p(b2))
    return a, b1, b2


def bf16_to_f32(Xb) -> np.ndarray:
    return (np.ascontiguousarray(Xb, np.uint16).astype(np.uint32) << 16).view(np.float32)


def round_bf16(Y) -> np.ndarray:
    """fp64 -> bf16 bit patterns (round half to even, from the fp64 value)."""
    Y = _c(Y, np.float64)
    out = np.empty(Y.shape, np.uint16)
    lib().or_round_bf16(_p(Y), Y.size, _p(out))
    return out


# --------------------------------------------------------------------------
# SQ8 (Section 3.1, per-dimension parameters)
# --------------------------------------------------------------------------
def sq8_fit(X, bits=8):
    """Per-dimension bias and scale of B-bit scalar codes (Section 3.1 "SQ8
    and SQ4"): 2^B - 1 levels between the min and the max."""
    X = _c(X, np.float32)
    n, d = X.shape
    b = np.empty(d, np.float32)
    s = np.empty(d, np.float32)
    if bits == 8:
        lib().or_sq8_fit(_p(X), n, d, _p(b), _p(s))
    else:
        lib().or_sq_fit(_p(X), n, d, (1 << bits) - 1, _p(b), _p(s))
    return b, s


def sq8_encode(X, b, s, bits=8):
    X = _c(X, np.float32)
    n, d = X.shape
    codes = np.empty((n, d), np.uint8)
    if bits == 8:
        lib().or_sq8_encode(_p(X), n, d, _p(_c(b, np.float32)), _p(_c(s, np.float32)), _p(codes))
    else:
        lib().or_sq_encode(_p(X), n, d, (1 << bits) - 1, _p(_c(b, np.float32)), _p(_c(s, np.float32)),
                           _p(codes))
    return codes


def sq8_decode(codes, b, s):
    codes = _c(codes, np.uint8)
    n, d = codes.shape
    Y = np.empty((n, d), np.float32)
    lib().or_sq8_decode(_p(codes), n, d, _p(_c(b, np.float32)), _p(_c(s, np.float32)), _p(Y))
    return Y


def assign_sq8(Xc, Cc):
    Xc, Cc = _c(Xc, np.uint8), _c(Cc, np.uint8)
    n, d = Xc.shape
    k = Cc.shape[0]
    a = np.empty(n, np.int32)
    best = np.empty(n, np.int64)
    lib().or_assign_sq8(_p(Xc), n, d, _p(Cc), k, _p(a), _p(best))
    return a, best


def update_sq8(Xc, assign, Cc):
    Xc = _c(Xc, np.uint8)
    n, d = Xc.shape
    Cn = np.array(Cc, dtype=np.uint8, copy=True, order="C")
    k = Cn.shape[0]
    counts = np.empty(k, np.int64)
    lib().or_update_sq8(_p(Xc), n, d, _p(_c(assign, np.int32)), k, _p(Cn), _p(counts))
    return Cn, counts


# --------------------------------------------------------------------------
# STEP 3: mean of members; objective
# --------------------------------------------------------------------------
def update_f32(X, assign, C):
    X = _c(X, np.float32)
    n, d = X.shape
    Cn = np.array(C, dtype=np.float32, copy=True, order="C")
    k = Cn.shape[0]
    counts = np.empty(k, np.int64)
    lib().or_update_f32(_p(X), n, d, _p(_c(assign, np.int32)), k, _p(Cn), _p(counts))
    return Cn, counts


def update_bf16(Xb, assign, C):
    Xb = _c(Xb, np.uint16)
    n, d = Xb.shape
    Cn = np.array(C, dtype=np.float32, copy=True, order="C")
    k = Cn.shape[0]
    counts = np.empty(k, np.int64)
    lib().or_update_bf16(_p(Xb), n, d, _p(_c(assign, np.int32)), k, _p(Cn), _p(counts))
    return Cn, counts


def objective_f32(X, C, assign) -> float:
    X = _c(X, np.float32)
    n, d = X.shape
    return float(lib().or_objective_f32(_p(X), n, d, _p(_c(C, np.float32)), _p(_c(assign, np.int32))))


def objective_bf16(Xb, C, assign) -> float:
    Xb = _c(Xb, np.uint16)
    n, d = Xb.shape
    return float(lib().or_objective_bf16(_p(Xb), n, d, _p(_c(C, np.float32)), _p(_c(assign, np.int32))))


# --------------------------------------------------------------------------
# RabitQ 1-bit (Section 3.1, Eq. l2_decomp, rabitq_l2, final:rabitq)
# --------------------------------------------------------------------------
def rbq1_mean(X):
    X = _c(X, np.float32)
    n, d = X.shape
    m = np.empty(d, np.float32)
    lib().or_rbq1_mean(_p(X), n, d, _p(m))
    return m


def mean_scale(amax, n) -> int:
    """Fixed-point scale s of the RabitQ mean for a maximum |x| and n rows."""
    return int(lib().or_mean_scale(float(amax), int(n)))


def column_sums_fixed(X, s):
    """int64[d]: per column, the sum of rint(x 2^s) (exact)."""
    X = _c(X, np.float32)
    n, d = X.shape
    S = np.zeros(d, np.int64)
    lib().or_column_sums_fixed(_p(X), n, d, int(s), _p(S))
    return S


def mean_from_sums(S, n, s):
    """fl32(fl64(S) / (n 2^s)) per column."""
    S = _c(S, np.int64)
    m = np.empty(S.shape[0], np.float32)
    lib().or_mean_from_sums(_p(S), int(n), S.shape[0], int(s), _p(m))
    return m


def rbq1_encode(X, m):
    """Returns (codes uint32[n, W], nx2 f32[n], F f32[n], popx int32[n])."""
    X = _c(X, np.float32)
    n, d = X.shape
    W = (d + 31) // 32
    codes = np.empty((n, W), np.uint32)
    nx2 = np.empty(n, np.float32)
    F = np.empty(n, np.float32)
    popx = np.empty(n, np.int32)
    lib().or_rbq1_encode(_p(X), n, d, _p(_c(m, np.float32)), _p(codes), _p(nx2), _p(F), _p(popx))
    return codes, nx2, F, popx


def rbq1_centroid_sq4(C, m):
    """Returns (ybar uint8[k, d], b f32[k], s f32[k], sumy int32[k], ny2 f32[k])."""
    C = _c(C, np.float32)
    k, d = C.shape
    ybar = np.empty((k, d), np.uint8)
    b = np.empty(k, np.float32)
    s = np.empty(k, np.float32)
    sumy = np.empty(k, np.int32)
    ny2 = np.empty(k, np.float32)
    lib().or_rbq1_centroid_sq4(_p(C), k, d, _p(_c(m, np.float32)), _p(ybar), _p(b), _p(s), _p(sumy), _p(ny2))
    return ybar, b, s, sumy, ny2


def sumsq_blocked(r) -> float:
    """||r||^2 in the library's blocked fp64 order (see skm_oracle.c)."""
    r = _c(r, np.float32)
    return float(lib().or_sumsq_blocked(_p(r), r.size))


def rbq1_assign(codes, nx2, F, popx, d, prep):
    """prep = rbq1_centroid_sq4(...). Returns (assign int32[n], est f32[n])."""
    codes = _c(codes, np.uint32)
    n = codes.shape[0]
    ybar, b, s, sumy, ny2 = prep
    k = ybar.shape[0]
    a = np.empty(n, np.int32)
    est = np.empty(n, np.float32)
    lib().or_rbq1_assign(
        _p(codes), _p(_c(nx2, np.float32)), _p(_c(F, np.float32)), _p(_c(popx, np.int32)), n, d,
        _p(_c(ybar, np.uint8)), _p(_c(b, np.float32)), _p(_c(s, np.float32)), _p(_c(sumy, np.int32)),
        _p(_c(ny2, np.float32)), k, _p(a), _p(est),
    )
    return a, est


def rbq1_centroid_sym(C, m):
    """Symmetric 1-bit centroid side: (bits uint32[k, W], fy f32[k], ny2 f32[k])."""
    C = _c(C, np.float32)
    k, d = C.shape
    W = (d + 31) // 32
    yb = np.empty((k, W), np.uint32)
    fy = np.empty(k, np.float32)
    ny2 = np.empty(k, np.float32)
    lib().or_rbq1_centroid_sym(_p(C), k, d, _p(_c(m, np.float32)), _p(yb), _p(fy), _p(ny2))
    return yb, fy, ny2


def rbq1_assign_sym(codes, nx2, F, d, prep):
    """XOR + POPCOUNT estimate against binarized centroids; (assign, est)."""
    codes = _c(codes, np.uint32)
    n = codes.shape[0]
    yb, fy, ny2 = prep
    k = yb.shape[0]
    a = np.empty(n, np.int32)
    est = np.empty(n, np.float32)
    lib().or_rbq1_assign_sym(_p(codes), _p(_c(nx2, np.float32)), _p(_c(F, np.float32)), n, d, _p(_c(yb, np.uint32)),
                             _p(_c(fy, np.float32)), _p(_c(ny2, np.float32)), k, _p(a), _p(est))
    return a, est


def lloyd_rbq1_sym(codes, nx2, F, popx, d, m, C0, iters, e=None):
    """Lloyd with the symmetric estimate in the assignment (the update is the
    fused decode-average of the points, as in the asymmetric variant)."""
    if e is None:
        e = rbq1_exponent(F)
    C = np.array(C0, np.float32, copy=True)
    for _ in range(iters):
        a, _ = rbq1_assign_sym(codes, nx2, F, d, rbq1_centroid_sym(C, m))
        C, _ = rbq1_update(codes, F, d, m, e, a, C)
    a, _ = rbq1_assign_sym(codes, nx2, F, d, rbq1_centroid_sym(C, m))
    return C, a


def rbq1_exponent(F) -> int:
    F = _c(F, np.float32)
    return int(lib().or_rbq1_exponent(_p(F), F.size))


def rbq1_update(codes, F, d, m, e, assign, C):
    codes = _c(codes, np.uint32)
    n = codes.shape[0]
    Cn = np.array(C, dtype=np.float32, copy=True, order="C")
    k = Cn.shape[0]
    counts = np.empty(k, np.int64)
    lib().or_rbq1_update(
        _p(codes), _p(_c(F, np.float32)), n, d, _p(_c(m, np.float32)), int(e),
        _p(_c(assign, np.int32)), k, _p(Cn), _p(counts),
    )
    return Cn, counts


def rbq1_decode_points(codes, F, d, m, e, idx):
    """Decoded points (the fused decode-average of one member each), f32[len(idx), d]."""
    idx = np.asarray(idx, np.int64)
    sub_codes = _c(codes, np.uint32)[idx]
    sub_F = _c(F, np.float32)[idx]
    k = idx.size
    C0 = np.zeros((k, d), np.float32)
    C, _ = rbq1_update(sub_codes, sub_F, d, m, e, np.arange(k, dtype=np.int32), C0)
    return C


# --------------------------------------------------------------------------
# LVQ4 (Section 3.1 "LVQ4", Eq. final:lvq, fused decode-average)
# --------------------------------------------------------------------------
def lvq4_encode(V):
    """Per-vector LVQ4 of V [n, d]: (codes uint8[n, d] in 0..15,
    fac f32[n, 4] = (s, b, N, A), G f32[n] = s * sum(codes))."""
    V = _c(V, np.float32)
    n, d = V.shape
    codes = np.empty((n, d), np.uint8)
    fac = np.empty((n, 4), np.float32)
    G = np.empty(n, np.float32)
    lib().or_lvq4_encode(_p(V), n, d, _p(codes), _p(fac), _p(G))
    return codes, fac, G


def lvq4_pack(codes):
    """Nibble-packed layout of 4-bit codes: uint32 [n, ceil(d/8)], dimension
    8w + j in bits 4j .. 4j + 3 of word w, unused nibbles 0."""
    codes = np.asarray(codes, np.uint8)
    n, d = codes.shape
    W = (d + 7) // 8
    pad = np.zeros((n, 8 * W), np.uint32)
    pad[:, :d] = codes
    out = np.zeros((n, W), np.uint32)
    for j in range(8):
        out |= pad[:, j::8] << np.uint32(4 * j)
    return out


def lvq4_unpack(words, d):
    words = np.asarray(words).view(np.uint32)
    n, W = words.shape
    out = np.empty((n, 8 * W), np.uint8)
    for j in range(8):
        out[:, j::8] = (words >> np.uint32(4 * j)) & np.uint32(15)
    return out[:, :d]


def lvq4_assign(codes, fac, prep):
    """prep = lvq4_encode(C).  Returns (assign int32[n], dist f32[n])."""
    codes = _c(codes, np.uint8)
    n, d = codes.shape
    yc, yfac, Gy = prep
    k = yc.shape[0]
    a = np.empty(n, np.int32)
    dist = np.empty(n, np.float32)
    lib().or_lvq4_assign(_p(codes), _p(_c(fac, np.float32)), n, d, _p(_c(yc, np.uint8)),
                         _p(_c(yfac, np.float32)), _p(_c(Gy, np.float32)), k, _p(a), _p(dist))
    return a, dist


def lvq4_exponent(fac) -> int:
    fac = _c(fac, np.float32)
    return int(lib().or_lvq4_exponent(_p(fac), fac.shape[0]))


def lvq4_update(codes, fac, e, assign, C):
    codes = _c(codes, np.uint8)
    n, d = codes.shape
    Cn = np.array(C, dtype=np.float32, copy=True, order="C")
    k = Cn.shape[0]
    counts = np.empty(k, np.int64)
    lib().or_lvq4_update(_p(codes), _p(_c(fac, np.float32)), n, d, int(e), _p(_c(assign, np.int32)), k,
                         _p(Cn), _p(counts))
    return Cn, counts


def lvq4_decode_points(codes, fac, e, idx):
    """Decoded points (the fused decode-average of one member each)."""
    idx = np.asarray(idx, np.int64)
    sub = _c(codes, np.uint8)[idx]
    k, d = sub.shape
    C, _ = lvq4_update(sub, _c(fac, np.float32)[idx], e, np.arange(k, dtype=np.int32), np.zeros((k, d), np.float32))
    return C


# --------------------------------------------------------------------------
# Projection (rotation / PCA)
# --------------------------------------------------------------------------
def project(X, P, mu=None):
    """Y = (X - mu) P in fp64, returned as fp64 [n, dout]."""
    X = _c(X, np.float32)
    P = _c(P, np.float32)
    n, d = X.shape
    dout = P.shape[1]
    Y = np.empty((n, dout), np.float64)
    lib().or_project(_p(X), n, d, _p(_c(mu, np.float32)) if mu is not None else None, _p(P), dout, _p(Y))
    return Y


def unproject(Y, P, mu=None):
    """x = y P^T + mu in fp64 (P: d x dout), [n, d]."""
    Y = _c(Y, np.float32)
    P = _c(P, np.float32)
    n, dout = Y.shape
    d = P.shape[0]
    X = np.empty((n, d), np.float64)
    lib().or_unproject(_p(Y), n, dout, _p(P), _p(_c(mu, np.float32)) if mu is not None else None, d, _p(X))
    return X


def mean_cov(X):
    X = _c(X, np.float32)
    n, d = X.shape
    mu = np.empty(d, np.float64)
    cov = np.empty((d, d), np.float64)
    lib().or_mean_cov(_p(X), n, d, _p(mu), _p(cov))
    return mu, cov


def pca_fit(X, d_out):
    """Returns (mu fp64[d], P fp64[d, d_out], eigenvalues fp64[d_out]) by descending eigenvalue."""
    mu, cov = mean_cov(X)
    w, V = np.linalg.eigh(cov)
    order = np.argsort(-w, kind="stable")[:d_out]
    w = w[order]
    V = V[:, order]
    piv = np.argmax(np.abs(V), axis=0)
    sgn = np.sign(V[piv, np.arange(V.shape[1])])
    sgn[sgn == 0] = 1.0
    return mu, V * sgn, w


# --------------------------------------------------------------------------
# Lloyd loop (Section 2.3): iters x (STEP 2, STEP 3), then STEP 2 once more.
# objective[t] is the objective of the assignment made at step t.
# --------------------------------------------------------------------------
def hadamard_rotate(X, sigma, mean=None):
    """y = H_D diag(sigma) [x - mean; 0] / sqrt(D), D = len(sigma) (a power of
    two >= d), in fp64 (fast Walsh-Hadamard transform), rounded to fp32."""
    X = _c(X, np.float32)
    n, d = X.shape
    sigma = _c(sigma, np.float32)
    D = sigma.shape[0]
    assert D >= d and D & (D - 1) == 0
    Y = np.empty((n, D), np.float32)
    lib().or_hadamard_rotate(_p(X), n, d, _p(_c(mean, np.float32)) if mean is not None else None, _p(sigma), D,
                             _p(Y))
    return Y


def split_empty(C, counts):
    """Empty clusters take half of the current largest one (the library's
    reading of splitting large clusters, Section 2.3 STEP 3); returns the new
    centroids and the number of splits.  fp32 centroids or SQ8 codes."""
    C = np.array(C, copy=True, order="C")
    k, d = C.shape
    counts = _c(counts, np.int64)
    if C.dtype == np.uint8:
        ns = lib().or_split_empty_sq8(_p(C), _p(counts), k, d)
    else:
        C = C.astype(np.float32)
        ns = lib().or_split_empty_f32(_p(C), _p(counts), k, d)
    return C, int(ns)


def lloyd_f32(X, C0, iters, split=False):
    C = np.array(C0, np.float32, copy=True)
    objs = []
    for _ in range(iters):
        a, best, _ = assign_f32(X, C)
        objs.append(float(best.sum()))
        C, counts = update_f32(X, a, C)
        if split:
            C, _ = split_empty(C, counts)
    a, best, second = assign_f32(X, C)
    objs.append(float(best.sum()))
    return C, a, objs


def lloyd_bf16(Xb, C0, iters):
    C = np.array(C0, np.float32, copy=True)
    objs = []
    for _ in range(iters):
        a, best, _ = assign_bf16(Xb, C)
        objs.append(float(best.sum()))
        C, counts = update_bf16(Xb, a, C)
    a, best, _ = assign_bf16(Xb, C)
    objs.append(float(best.sum()))
    return C, a, objs


def lloyd_sq8(Xc, C0c, iters, split=False):
    Cc = np.array(C0c, np.uint8, copy=True)
    for _ in range(iters):
        a, _ = assign_sq8(Xc, Cc)
        Cc, counts = update_sq8(Xc, a, Cc)
        if split:
            Cc, _ = split_empty(Cc, counts)
    a, best = assign_sq8(Xc, Cc)
    return Cc, a


def lloyd_rbq1(codes, nx2, F, popx, d, m, C0, iters, e=None, split=False):
    if e is None:
        e = rbq1_exponent(F)
    C = np.array(C0, np.float32, copy=True)
    for _ in range(iters):
        prep = rbq1_centroid_sq4(C, m)
        a, _ = rbq1_assign(codes, nx2, F, popx, d, prep)
        C, counts = rbq1_update(codes, F, d, m, e, a, C)
        if split:
            C, _ = split_empty(C, counts)
    prep = rbq1_centroid_sq4(C, m)
    a, est = rbq1_assign(codes, nx2, F, popx, d, prep)
    return C, a


def lloyd_lvq4(codes, fac, C0, iters, e=None, split=False):
    if e is None:
        e = lvq4_exponent(fac)
    C = np.array(C0, np.float32, copy=True)
    for _ in range(iters):
        a, _ = lvq4_assign(codes, fac, lvq4_encode(C))
        C, counts = lvq4_update(codes, fac, e, a, C)
        if split:
            C, _ = split_empty(C, counts)
    a, _ = lvq4_assign(codes, fac, lvq4_encode(C))
    return C, a


# --------------------------------------------------------------------------
# Hierarchical k-means (the paper's MESO- and FINE-CLUSTERING, with the
# optional refinement iteration of vanilla k-means).
# --------------------------------------------------------------------------
def fine_counts(sizes, k):
    """Fine clusters per meso cluster: k apportioned proportionally to the
    meso sizes n_i (floor of k n_i / N, the remaining clusters to the largest
    remainders k n_i mod N, ties to the lower index); a non-empty meso cluster
    left with none takes one from the cluster with the most (ties to the lower
    index).  Empty meso clusters get none.  The paper states sqrt(n_i) fine
    clusters per meso cluster; this reading keeps the total at the requested k."""
    sizes = [int(v) for v in sizes]
    N = sum(sizes)
    m = len(sizes)
    kk = [k * v // N for v in sizes]
    rem = [k * v % N for v in sizes]
    left = k - sum(kk)
    order = sorted(range(m), key=lambda i: (-rem[i], i))
    for i in order[:left]:
        kk[i] += 1
    for i in range(m):
        if sizes[i] > 0 and kk[i] == 0:
            j = min(range(m), key=lambda t: (-kk[t], t))
            kk[j] -= 1
            kk[i] = 1
    return kk


def fine_init_positions(n_i, k_i):
    """Positions (in the meso cluster's members, increasing point index) of the
    initial fine centroids: floor(t n_i / k_i), t < k_i."""
    return [t * n_i // k_i for t in range(k_i)]


def hierarchical(kind, data, k, m, meso_init, meso_iters, fine_iters, refine=False):
    """kind 'f32' (data = X), 'sq8' (data = codes), 'rbq1' (data = dict of
    codes, nx2, F, popx, d, m, e) or 'lvq4' (data = dict of codes (one byte per
    dimension), fac, e).  Returns (centroids [k], assignments [n],
    meso assignments [n], fine counts per meso cluster)."""
    if kind == "f32":
        X = _c(data, np.float32)
        n = X.shape[0]
        Cm, am, _ = lloyd_f32(X, X[meso_init], meso_iters)
    elif kind == "sq8":
        X = _c(data, np.uint8)
        n = X.shape[0]
        Cm, am = lloyd_sq8(X, X[meso_init], meso_iters)
    elif kind == "lvq4":
        r = data
        n = r["codes"].shape[0]
        C0 = lvq4_decode_points(r["codes"], r["fac"], r["e"], meso_init)
        Cm, am = lloyd_lvq4(r["codes"], r["fac"], C0, meso_iters, r["e"])
    else:
        r = data
        n = r["codes"].shape[0]
        C0 = rbq1_decode_points(r["codes"], r["F"], r["d"], r["m"], r["e"], meso_init)
        Cm, am = lloyd_rbq1(r["codes"], r["nx2"], r["F"], r["popx"], r["d"], r["m"], C0, meso_iters, r["e"])
    sizes = np.bincount(am, minlength=m)
    kf = fine_counts(sizes, k)
    base = np.concatenate([[0], np.cumsum(kf)]).astype(np.int64)
    a = np.empty(n, np.int32)
    Cs = []
    for i in range(m):
        members = np.nonzero(am == i)[0]  # increasing point index
        if kf[i] == 0:
            continue
        pos = fine_init_positions(len(members), kf[i])
        init = members[pos]
        if kind == "f32":
            Ci, ai, _ = lloyd_f32(X[members], X[init], fine_iters)
        elif kind == "sq8":
            Ci, ai = lloyd_sq8(X[members], X[init], fine_iters)
        elif kind == "lvq4":
            C0 = lvq4_decode_points(r["codes"], r["fac"], r["e"], init)
            Ci, ai = lloyd_lvq4(r["codes"][members], r["fac"][members], C0, fine_iters, r["e"])
        else:
            C0 = rbq1_decode_points(r["codes"], r["F"], r["d"], r["m"], r["e"], init)
            Ci, ai = lloyd_rbq1(r["codes"][members], r["nx2"][members], r["F"][members], r["popx"][members],
                                r["d"], r["m"], C0, fine_iters, r["e"])
        Cs.append(Ci)
        a[members] = ai + base[i]
    C = np.concatenate(Cs, axis=0)
    if refine:  # one vanilla iteration over all points, then the final assignment
        if kind == "f32":
            C, a, _ = lloyd_f32(X, C, 1)
        elif kind == "sq8":
            C, a = lloyd_sq8(X, C, 1)
        elif kind == "lvq4":
            C, a = lloyd_lvq4(r["codes"], r["fac"], C, 1, r["e"])
        else:
            C, a = lloyd_rbq1(r["codes"], r["nx2"], r["F"], r["popx"], r["d"], r["m"], C, 1, r["e"])
    return C, a, am, kf


# --------------------------------------------------------------------------
# STEP 1 (Section 2.3): seeded Forgy initialisation
# --------------------------------------------------------------------------
def philox4x32_10(ctr, key):
    """Philox4x32-10 of a 4-word counter under a 2-word key (4 uint32 words)."""
    c = np.asarray(ctr, dtype=np.uint32)
    k = np.asarray(key, dtype=np.uint32)
    out = np.empty(4, np.uint32)
    lib().or_philox4x32_10(_p(c), _p(k), _p(out))
    return out


def forgy_indices(seed, n, k):
    """The first k entries of the seeded Fisher-Yates permutation of range(n)
    (int64[k]); the draw is defined in skm_oracle.c."""
    out = np.empty(int(k), np.int64)
    lib().or_forgy_indices(ctypes.c_uint64(int(seed) & (2**64 - 1)), int(n), int(k), _p(out))
    return out


# --------------------------------------------------------------------------
# SuperKMeans with RabitQ codes: segment estimates and checkpoint pruning
# --------------------------------------------------------------------------
def rbq1_seg_bounds(d):
    a, b = ctypes.c_int(0), ctypes.c_int(0)
    lib().or_rbq1_seg_bounds(int(d), ctypes.byref(a), ctypes.byref(b))
    return a.value, b.value


def rbq1_seg_encode(X, m, bounds=None):
    """Per point and segment: (nx2 f32[n, 3], F f32[n, 3], popx int32[n, 3])."""
    X = _c(X, np.float32)
    n, d = X.shape
    d1, d2 = bounds if bounds is not None else rbq1_seg_bounds(d)
    nx2 = np.empty((n, 3), np.float32)
    F = np.empty((n, 3), np.float32)
    pc = np.empty((n, 3), np.int32)
    lib().or_rbq1_seg_encode(_p(X), n, d, _p(_c(m, np.float32)), d1, d2, _p(nx2), _p(F), _p(pc))
    return nx2, F, pc


def rbq1_seg_centroid(C, m, bounds=None):
    """(ybar uint8[k, d], b f32[k], s f32[k], sumy int32[k, 3], ny2 f32[k, 3])."""
    C = _c(C, np.float32)
    k, d = C.shape
    d1, d2 = bounds if bounds is not None else rbq1_seg_bounds(d)
    ybar = np.empty((k, d), np.uint8)
    b = np.empty(k, np.float32)
    s = np.empty(k, np.float32)
    sumy = np.empty((k, 3), np.int32)
    ny2 = np.empty((k, 3), np.float32)
    lib().or_rbq1_seg_centroid(_p(C), k, d, _p(_c(m, np.float32)), d1, d2, _p(ybar), _p(b), _p(s), _p(sumy),
                               _p(ny2))
    return ybar, b, s, sumy, ny2


SEG_EPS0 = 2.1  # ADSampling's default significance parameter


def rbq1_seg_factors(d, bounds=None, eps0=SEG_EPS0):
    """Checkpoint factors g_t = fl32((e_t / d) (1 + eps0 / sqrt(e_t))^2)."""
    d1, d2 = bounds if bounds is not None else rbq1_seg_bounds(d)
    g = np.empty(2, np.float32)
    lib().or_rbq1_seg_factors(int(d), d1, d2, float(eps0), _p(g))
    return g


def rbq1_seg_assign(codes, seg, d, prep, prev=None, bounds=None, g=None):
    """Checkpoint-pruned assignment (seg = rbq1_seg_encode output, prep =
    rbq1_seg_centroid output, g = the two checkpoint factors, default
    ADSampling's with eps0 = 2.1; g = (1, 1) is the exact test).  Returns
    (assign int32[n], D3 f32[n])."""
    if g is None:
        g = rbq1_seg_factors(d, bounds)
    codes = _c(codes, np.uint32)
    nx2, F, pc = (_c(v, t) for v, t in zip(seg, (np.float32, np.float32, np.int32)))
    ybar, b, s, sumy, ny2 = prep
    n = codes.shape[0]
    k = ybar.shape[0]
    d1, d2 = bounds if bounds is not None else rbq1_seg_bounds(d)
    a = np.empty(n, np.int32)
    est = np.empty(n, np.float32)
    pv = _c(prev, np.int32) if prev is not None else None
    lib().or_rbq1_seg_assign(_p(codes), _p(nx2), _p(F), _p(pc), n, d, d1, d2, _p(_c(ybar, np.uint8)),
                             _p(_c(b, np.float32)), _p(_c(s, np.float32)), _p(_c(sumy, np.int32)),
                             _p(_c(ny2, np.float32)), k, _p(pv), _p(_c(g, np.float32)), _p(a), _p(est))
    return a, est


def rbq1_seg_partials(codes, seg, d, prep, bounds=None):
    """Every pair's partial estimates (D1, D2, D3): f32[n, k, 3]."""
    codes = _c(codes, np.uint32)
    nx2, F, pc = (_c(v, t) for v, t in zip(seg, (np.float32, np.float32, np.int32)))
    ybar, b, s, sumy, ny2 = prep
    n, k = codes.shape[0], ybar.shape[0]
    d1, d2 = bounds if bounds is not None else rbq1_seg_bounds(d)
    D = np.empty((n, k, 3), np.float32)
    lib().or_rbq1_seg_partials(_p(codes), _p(nx2), _p(F), _p(pc), n, d, d1, d2, _p(_c(ybar, np.uint8)),
                               _p(_c(b, np.float32)), _p(_c(s, np.float32)), _p(_c(sumy, np.int32)),
                               _p(_c(ny2, np.float32)), k, _p(D))
    return D
