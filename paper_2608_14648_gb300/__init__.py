"""Python binding of libskm, the GB300 Lloyd k-means hot path (C ABI in
include/skm.h).

Argument marshalling only: torch tensors provide device memory and streams,
every step of the path runs in the CUDA kernels of libskm.so.  There is no
fallback: if the library is missing, importing the binding's entry points
raises.  Function names match the C entry points.
"""
from __future__ import annotations

import ctypes
import os

import torch

__all__ = [
    "REPR_F32", "REPR_SQ8", "REPR_RBQ1", "REPR_BF16", "REPR_LVQ4", "SkmError", "lib", "lib_path", "Data",
    "skm_version", "skm_kernel_launches", "skm_workspace_size", "skm_project", "skm_project_hadamard",
    "skm_make_rotation", "skm_pca_fit",
    "skm_quantize", "skm_rbq1_exponent", "skm_lvq4_exponent", "skm_assign", "skm_update", "skm_merge_partials",
    "skm_update_finalize", "skm_fit", "skm_split_empty", "skm_objective", "skm_sq8_decode", "EXPORTED_SYMBOLS",
    "EMPTY_KEEP", "EMPTY_SPLIT",
    "skm_assign_prune_stats",
]

REPR_F32, REPR_SQ8, REPR_RBQ1, REPR_BF16, REPR_LVQ4 = 0, 1, 2, 3, 4
FLAG_PRUNE, FLAG_SYMMETRIC, FLAG_WARM, FLAG_PRUNE_CUDA_CORES = 1, 2, 4, 8
DTYPE_F32, DTYPE_BF16 = 0, 1
EMPTY_KEEP, EMPTY_SPLIT = 0, 1
OP_ASSIGN, OP_UPDATE, OP_FIT, OP_QUANTIZE, OP_PCA, OP_ASSIGN_SEG = 0, 1, 2, 3, 4, 5

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB_PATH = os.path.join(_HERE, "_build", "libskm.so")
_lib = None

# Every entry point declared in include/skm.h.
EXPORTED_SYMBOLS = [
    "skm_last_error", "skm_version", "skm_kernel_launches", "skm_workspace_size", "skm_screen_bytes",
    "skm_screen_prep", "skm_project", "skm_project_hadamard", "skm_unproject", "skm_copy_from_host",
    "skm_make_rotation",
    "skm_pca_fit", "skm_quantize", "skm_rbq1_exponent", "skm_lvq4_exponent", "skm_assign",
    "skm_assign_prune_stats", "skm_assign_rbq1_noalloc", "skm_kernel_timer", "skm_kernel_timer_ms",
    "skm_assign_segmented",
    "skm_update",
    "skm_merge_partials", "skm_update_finalize", "skm_fit", "skm_split_empty", "skm_hier_workspace_size",
    "skm_fit_hierarchical", "skm_objective", "skm_sq8_decode", "skm_step_host_workspace_size",
    "skm_lloyd_step_host", "skm_inject_fault", "skm_fault_armed", "skm_forgy_indices", "skm_column_absmax",
    "skm_mean_scale", "skm_column_sums_fixed", "skm_mean_from_sums", "skm_rbq1_segment_bounds",
    "skm_rbq1_segments",
]


class SkmError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__(f"libskm error {code}: {msg}")
        self.code = code


class Data(ctypes.Structure):
    """skm_data (include/skm.h)."""

    _fields_ = [
        ("repr", ctypes.c_int32), ("d", ctypes.c_int32), ("n", ctypes.c_int64),
        ("x", ctypes.c_void_p), ("nx2", ctypes.c_void_p), ("F", ctypes.c_void_p),
        ("popx", ctypes.c_void_p), ("m", ctypes.c_void_p), ("rbq1_exp", ctypes.c_int32),
        ("flags", ctypes.c_int32), ("screen", ctypes.c_void_p), ("lvq", ctypes.c_void_p),
        ("seg_nx2", ctypes.c_void_p), ("seg_F", ctypes.c_void_p), ("seg_popx", ctypes.c_void_p),
    ]


class QuantParams(ctypes.Structure):
    _fields_ = [
        ("fit", ctypes.c_int32), ("bits", ctypes.c_int32), ("b", ctypes.c_void_p),
        ("s", ctypes.c_void_p), ("m", ctypes.c_void_p), ("nx2", ctypes.c_void_p),
        ("F", ctypes.c_void_p), ("popx", ctypes.c_void_p), ("lvq", ctypes.c_void_p),
    ]


class Stats(ctypes.Structure):
    _fields_ = [("rescored_rows", ctypes.c_int64), ("fallback_rows", ctypes.c_int64),
                ("empty_clusters", ctypes.c_int64), ("prune_first_block", ctypes.c_int64),
                ("prune_complete", ctypes.c_int64), ("cluster_size_std", ctypes.c_double),
                ("empty_per_iter", ctypes.c_void_p), ("prune_blocks", ctypes.c_int64),
                ("prune_front_dims", ctypes.c_int64), ("prune_rows_finished", ctypes.c_int64),
                ("prune_rows_full", ctypes.c_int64)]


class HierConfig(ctypes.Structure):
    _fields_ = [("k", ctypes.c_int32), ("m", ctypes.c_int32), ("meso_iters", ctypes.c_int32),
                ("fine_iters", ctypes.c_int32), ("refine", ctypes.c_int32), ("reserved", ctypes.c_int32 * 3)]


class FitConfig(ctypes.Structure):
    _fields_ = [("k", ctypes.c_int32), ("iters", ctypes.c_int32), ("empty_policy", ctypes.c_int32),
                ("reserved0", ctypes.c_int32), ("seed", ctypes.c_uint64), ("reserved", ctypes.c_int32 * 2)]


EXCHANGE_FN = ctypes.CFUNCTYPE(ctypes.c_int, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p)


class StepHostConfig(ctypes.Structure):
    """skm_step_host_config (include/skm.h)."""

    _fields_ = [("k", ctypes.c_int32), ("chunks", ctypes.c_int32), ("copy_stream", ctypes.c_void_p),
                ("partial", ctypes.c_void_p), ("counts", ctypes.c_void_p), ("exchange", EXCHANGE_FN),
                ("user", ctypes.c_void_p), ("warm", ctypes.c_int32), ("prune", ctypes.c_int32),
                ("reserved", ctypes.c_int32 * 2)]


def lib_path() -> str:
    return _LIB_PATH


def lib():
    """The loaded libskm.so; raises if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(_LIB_PATH):
            raise ImportError(f"libskm.so not found at {_LIB_PATH}: run `python -c 'import __graft_entry__ as g; g.build()'`")
        L = ctypes.CDLL(_LIB_PATH)
        vp, i32, i64, u64, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_uint64, ctypes.c_size_t
        sig = {
            "skm_last_error": ([], ctypes.c_char_p),
            "skm_version": ([], i32),
            "skm_kernel_launches": ([], ctypes.c_uint64),
            "skm_workspace_size": ([i32, vp, i32], sz),
            "skm_screen_bytes": ([vp], sz),
            "skm_screen_prep": ([vp, vp, sz, vp], i32),
            "skm_project": ([vp, i64, i32, vp, vp, i32, i32, vp, vp, sz, vp], i32),
            "skm_make_rotation": ([u64, i32, vp], i32),
            "skm_forgy_indices": ([u64, i64, i32, vp], i32),
            "skm_project_hadamard": ([vp, i64, i32, vp, vp, i32, i32, vp, vp], i32),
            "skm_unproject": ([vp, i64, i32, vp, vp, i32, vp, vp], i32),
            "skm_copy_from_host": ([vp, vp, sz, vp], i32),
            "skm_pca_fit": ([vp, i64, i32, i32, vp, vp, vp, vp, sz, vp], i32),
            "skm_quantize": ([i32, vp, i64, i32, vp, vp, vp, sz, vp], i32),
            "skm_rbq1_exponent": ([vp, i64, vp, vp, sz, vp], i32),
            "skm_lvq4_exponent": ([vp, i64, vp, vp, sz, vp], i32),
            "skm_assign": ([vp, vp, i32, vp, vp, vp, vp, sz, vp], i32),
            "skm_assign_prune_stats": ([vp, sz, vp, vp], i32),
            "skm_kernel_timer": ([i32], i32),
            "skm_kernel_timer_ms": ([vp], i32),
            "skm_assign_rbq1_noalloc": ([vp, vp, i32, vp, vp, vp], i32),
            "skm_assign_segmented": ([vp, vp, i32, vp, vp, i32, vp, vp, vp, sz, vp], i32),
            "skm_update": ([vp, vp, i32, vp, vp, vp, vp, sz, vp], i32),
            "skm_merge_partials": ([vp, vp, i64, i32, vp], i32),
            "skm_update_finalize": ([vp, vp, vp, i32, vp, vp], i32),
            "skm_fit": ([vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp], i32),
            "skm_split_empty": ([vp, vp, vp, i32, vp, sz, vp], i32),
            "skm_hier_workspace_size": ([vp, vp], sz),
            "skm_fit_hierarchical": ([vp, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp], i32),
            "skm_objective": ([vp, i32, i64, i32, vp, i32, vp, vp, vp, sz, vp], i32),
            "skm_sq8_decode": ([vp, i64, i32, vp, vp, vp, vp], i32),
            "skm_inject_fault": ([i32, i32], i32),
            "skm_column_absmax": ([vp, i64, i32, vp, vp, sz, vp], i32),
            "skm_rbq1_segment_bounds": ([i32, vp, vp], i32),
            "skm_rbq1_segments": ([vp, i64, i32, vp, vp, vp, vp, vp], i32),
            "skm_mean_scale": ([ctypes.c_float, i64], i32),
            "skm_column_sums_fixed": ([vp, i64, i32, i32, vp, vp], i32),
            "skm_mean_from_sums": ([vp, i64, i32, i32, vp, vp], i32),
            "skm_fault_armed": ([i32], i32),
            "skm_step_host_workspace_size": ([vp, vp], sz),
            "skm_lloyd_step_host": ([vp, vp, vp, vp, vp, vp, vp, vp, sz, vp], i32),
        }
        for name, (args, res) in sig.items():
            fn = getattr(L, name)
            fn.argtypes = args
            fn.restype = res
        _lib = L
    return _lib


def _check(rc):
    if rc != 0:
        raise SkmError(rc, lib().skm_last_error().decode())


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _ws(nbytes, device, zero=False):
    nbytes = max(int(nbytes), 256)
    # 256-byte alignment: the caching allocator returns 512-byte aligned blocks;
    # zero: a workspace that carries state between calls (SKM_FLAG_WARM) starts
    # with no stamp, whatever the recycled memory held
    return (torch.zeros if zero else torch.empty)(nbytes, dtype=torch.uint8, device=device)


def _dev(t):
    return t.device if t is not None else torch.device("cuda")


class Points:
    """Keeps the tensors of one skm_data alive; `.ref` is the ctypes struct."""

    def __init__(self, repr_, x, d, nx2=None, F=None, popx=None, m=None, rbq1_exp=0, screen=None, flags=0,
                 lvq=None, seg=None):
        assert x.is_contiguous()
        self.repr, self.x, self.d = repr_, x, int(d)
        self.nx2, self.F, self.popx, self.m = nx2, F, popx, m
        self.lvq = lvq
        self.seg = seg  # RBQ1 segment factors (nx2s, Fs, popxs), skm_rbq1_segments
        self.n = x.shape[0]
        self.rbq1_exp = int(rbq1_exp)
        self.screen = screen
        self.flags = int(flags)
        sg = seg if seg is not None else (None, None, None)
        self.ref = Data(repr_, self.d, self.n, x.data_ptr(), _ptr(nx2), _ptr(F), _ptr(popx), _ptr(m),
                        self.rbq1_exp, self.flags, _ptr(screen), _ptr(lvq), _ptr(sg[0]), _ptr(sg[1]), _ptr(sg[2]))

    def with_flags(self, flags):
        return Points(self.repr, self.x, self.d, self.nx2, self.F, self.popx, self.m, self.rbq1_exp, self.screen,
                      flags, self.lvq, self.seg)

    def with_segments(self, seg):
        """The same points with RabitQ segment factors attached (SKM_FLAG_PRUNE on RBQ1)."""
        return Points(self.repr, self.x, self.d, self.nx2, self.F, self.popx, self.m, self.rbq1_exp, self.screen,
                      self.flags, self.lvq, seg)

    def with_screen(self, stream=None):
        """Builds the screening copy once (skm_screen_prep) and attaches it."""
        nbytes = lib().skm_screen_bytes(ctypes.byref(self.ref))
        if nbytes == 0:
            return self
        buf = _ws(nbytes, self.device)
        _check(lib().skm_screen_prep(ctypes.byref(self.ref), _ptr(buf), buf.numel(), _stream(stream)))
        return Points(self.repr, self.x, self.d, self.nx2, self.F, self.popx, self.m, self.rbq1_exp, buf,
                      self.flags, self.lvq, self.seg)

    @property
    def device(self):
        return self.x.device


def skm_version() -> int:
    return lib().skm_version()


def skm_kernel_launches() -> int:
    return int(lib().skm_kernel_launches())


def skm_workspace_size(op, pts: Points, k) -> int:
    n = lib().skm_workspace_size(op, ctypes.byref(pts.ref), int(k))
    if n == 0:
        raise SkmError(1, lib().skm_last_error().decode())
    return n


OP_PROJECT, OP_PROJECT_MIN = 6, 7


def skm_project(X, P, mean=None, out_dtype=DTYPE_F32, stream=None, ws=None, max_ws_bytes=None, cuda_cores=False):
    """Y = (X - mean) P.  Tensor cores (fp32 accuracy from bf16 parts) with a
    workspace of up to max_ws_bytes (default: one pass over all rows);
    cuda_cores=True selects the fp32 CUDA-core kernel (no workspace)."""
    n, d = X.shape
    d_out = P.shape[1]
    Y = torch.empty(n, d_out, device=X.device, dtype=torch.float32 if out_dtype == DTYPE_F32 else torch.bfloat16)
    if cuda_cores:
        ws = None
    elif ws is None:
        probe = Data(REPR_F32, d, n, 0, None, None, None, None, 0, 0)
        full = lib().skm_workspace_size(OP_PROJECT, ctypes.byref(probe), d_out)
        need = full if max_ws_bytes is None else max(min(full, int(max_ws_bytes)),
                                                      lib().skm_workspace_size(OP_PROJECT_MIN, ctypes.byref(probe),
                                                                               d_out))
        ws = _ws(need, X.device)
    _check(lib().skm_project(_ptr(X), n, d, _ptr(mean), _ptr(P), d_out, out_dtype, _ptr(Y), _ptr(ws),
                             0 if ws is None else ws.numel(), _stream(stream)))
    return Y


def skm_project_hadamard(X, sigma, mean=None, out_dtype=DTYPE_F32, stream=None):
    """Randomized Hadamard rotation; sigma: device float32 [D] of +-1 (D a power of two >= d)."""
    n, d = X.shape
    D = sigma.numel()
    Y = torch.empty(n, D, device=X.device, dtype=torch.float32 if out_dtype == DTYPE_F32 else torch.bfloat16)
    _check(lib().skm_project_hadamard(_ptr(X), n, d, _ptr(mean), _ptr(sigma), int(D), out_dtype, _ptr(Y),
                                      _stream(stream)))
    return Y


def skm_copy_from_host(dst, src, stream=None):
    """dst (contiguous device tensor) <- src (contiguous pinned host tensor of
    the same number of bytes), copied by thread blocks over the host link."""
    nb = src.numel() * src.element_size()
    if not dst.is_contiguous() or not src.is_contiguous() or dst.numel() * dst.element_size() != nb:
        raise ValueError("skm_copy_from_host: contiguous tensors of equal byte size")
    _check(lib().skm_copy_from_host(_ptr(dst), _ptr(src), nb, _stream(stream)))
    return dst


def skm_unproject(Y, P, mean=None, stream=None):
    """X = Y P^T + mean (P: the d x d_out projection matrix)."""
    n, d_out = Y.shape
    d = P.shape[0]
    X = torch.empty(n, d, device=Y.device, dtype=torch.float32)
    _check(lib().skm_unproject(_ptr(Y), n, d_out, _ptr(P), _ptr(mean), d, _ptr(X), _stream(stream)))
    return X


def skm_make_rotation(seed, d):
    out = torch.empty(d, d, dtype=torch.float32)
    _check(lib().skm_make_rotation(int(seed), int(d), ctypes.c_void_p(out.data_ptr())))
    return out


def skm_pca_fit(X, d_out, stream=None):
    n, d = X.shape
    dummy = Points(REPR_F32, X, d)
    ws = _ws(skm_workspace_size(OP_PCA, dummy, 1), X.device)
    mean = torch.empty(d, device=X.device, dtype=torch.float32)
    P = torch.empty(d, d_out, device=X.device, dtype=torch.float32)
    w = torch.empty(d_out, device=X.device, dtype=torch.float32)
    _check(lib().skm_pca_fit(_ptr(X), n, d, d_out, _ptr(mean), _ptr(P), _ptr(w), _ptr(ws), ws.numel(),
                             _stream(stream)))
    return mean, P, w


def skm_quantize(repr_, X, fit=True, b=None, s=None, m=None, stream=None, out=None, ws=None, bits=8):
    """SQ8 -> dict(codes, b, s) (bits=4: SQ4 codes 0..15, one per byte);
    RBQ1 -> dict(codes, m, nx2, F, popx).
    `out` may supply preallocated (contiguous) output tensors by those names."""
    n, d = X.shape
    dev = X.device
    out = out or {}
    if ws is None:
        dummy = Points(REPR_F32, X, d)
        ws = _ws(skm_workspace_size(OP_QUANTIZE, dummy, 1), dev)
    if repr_ == REPR_SQ8:
        b = b if b is not None else torch.empty(d, device=dev, dtype=torch.float32)
        s = s if s is not None else torch.empty(d, device=dev, dtype=torch.float32)
        codes = out.get("codes")
        codes = codes if codes is not None else torch.empty(n, d, device=dev, dtype=torch.uint8)
        qp = QuantParams(int(fit), int(bits), b.data_ptr(), s.data_ptr(), None, None, None, None, None)
        _check(lib().skm_quantize(repr_, _ptr(X), n, d, ctypes.byref(qp), _ptr(codes), _ptr(ws), ws.numel(),
                                  _stream(stream)))
        return {"codes": codes, "b": b, "s": s}
    if repr_ == REPR_RBQ1:
        W = (d + 31) // 32
        m = m if m is not None else torch.empty(d, device=dev, dtype=torch.float32)
        def _o(name, shape, dt):
            t = out.get(name)
            if t is None:
                return torch.empty(*shape, device=dev, dtype=dt)
            if not t.is_contiguous() or tuple(t.shape) != tuple(shape) or t.dtype != dt:
                raise ValueError(f"out[{name!r}] must be a contiguous {dt} tensor of shape {shape}")
            return t
        codes = _o("codes", (n, W), torch.int32)
        nx2 = _o("nx2", (n,), torch.float32)
        F = _o("F", (n,), torch.float32)
        popx = _o("popx", (n,), torch.int32)
        qp = QuantParams(int(fit), 0, None, None, m.data_ptr(), nx2.data_ptr(), F.data_ptr(), popx.data_ptr(), None)
        _check(lib().skm_quantize(repr_, _ptr(X), n, d, ctypes.byref(qp), _ptr(codes), _ptr(ws), ws.numel(),
                                  _stream(stream)))
        return {"codes": codes, "m": m, "nx2": nx2, "F": F, "popx": popx}
    if repr_ == REPR_LVQ4:
        W = (d + 7) // 8
        codes = out.get("codes")
        codes = codes if codes is not None else torch.empty(n, W, device=dev, dtype=torch.int32)
        lvq = out.get("lvq")
        lvq = lvq if lvq is not None else torch.empty(n, 4, device=dev, dtype=torch.float32)
        if tuple(codes.shape) != (n, W) or tuple(lvq.shape) != (n, 4) or not codes.is_contiguous() \
                or not lvq.is_contiguous():
            raise ValueError("LVQ4 outputs: codes int32 [n, ceil(d/8)], lvq float32 [n, 4], contiguous")
        qp = QuantParams(0, 0, None, None, None, None, None, None, lvq.data_ptr())
        _check(lib().skm_quantize(repr_, _ptr(X), n, d, ctypes.byref(qp), _ptr(codes), _ptr(ws), ws.numel(),
                                  _stream(stream)))
        return {"codes": codes, "lvq": lvq}
    raise ValueError("repr must be REPR_SQ8, REPR_RBQ1 or REPR_LVQ4")


def skm_lvq4_exponent(lvq, stream=None):
    ws = _ws(1024, lvq.device)
    e = ctypes.c_int(0)
    _check(lib().skm_lvq4_exponent(_ptr(lvq), lvq.shape[0], ctypes.byref(e), _ptr(ws), ws.numel(), _stream(stream)))
    return e.value


def lvq4_points(q, d, e=None):
    """Points for the LVQ4 representation from skm_quantize's outputs."""
    if e is None:
        e = skm_lvq4_exponent(q["lvq"])
    return Points(REPR_LVQ4, q["codes"], d, rbq1_exp=e, lvq=q["lvq"])


def skm_rbq1_exponent(F, stream=None):
    ws = _ws(1024, F.device)
    e = ctypes.c_int(0)
    _check(lib().skm_rbq1_exponent(_ptr(F), F.numel(), ctypes.byref(e), _ptr(ws), ws.numel(), _stream(stream)))
    return e.value


def workspace(op, pts: Points, k):
    """A device workspace tensor sized for op (OP_ASSIGN, OP_UPDATE, OP_FIT),
    zero-filled (a workspace that carries bounds between calls must start
    without a stamp)."""
    return _ws(skm_workspace_size(op, pts, k), pts.device, zero=True)


def rbq1_points(q, d, e=None):
    """Points for the RBQ1 representation from skm_quantize's outputs."""
    if e is None:
        e = skm_rbq1_exponent(q["F"])
    return Points(REPR_RBQ1, q["codes"], d, q["nx2"], q["F"], q["popx"], q["m"], e)


def skm_assign(pts: Points, C, k=None, prev_assign=None, want_dist=True, ws=None, stream=None, out=None,
               dist_out=None):
    k = C.shape[0] if k is None else k
    dev = pts.device
    if ws is None:
        ws = _ws(skm_workspace_size(OP_ASSIGN, pts, k), dev)
    assign = out if out is not None else torch.empty(pts.n, device=dev, dtype=torch.int32)
    dist = None
    if want_dist:
        dist = dist_out if dist_out is not None else torch.empty(pts.n, device=dev, dtype=torch.float32)
    _check(lib().skm_assign(ctypes.byref(pts.ref), _ptr(C), int(k), _ptr(prev_assign), _ptr(assign), _ptr(dist),
                            _ptr(ws), ws.numel(), _stream(stream)))
    return assign, dist


def skm_kernel_timer(on):
    """Enables (True) or disables the events around each tensor-core kernel launch."""
    _check(lib().skm_kernel_timer(int(bool(on))))


def skm_kernel_timer_ms():
    """Duration (ms) of the last tensor-core kernel launch timed (waits for it)."""
    ms = ctypes.c_float(0.0)
    _check(lib().skm_kernel_timer_ms(ctypes.byref(ms)))
    return float(ms.value)


def skm_assign_prune_stats(ws, stream=None):
    """Pruning counters of the last pruned skm_assign on workspace `ws`
    (synchronises the stream): first-block / complete survivors and the
    block partial sums evaluated after the first block."""
    st = Stats()
    _check(lib().skm_assign_prune_stats(_ptr(ws), ws.numel(), ctypes.byref(st), _stream(stream)))
    return {"prune_first_block": st.prune_first_block, "prune_complete": st.prune_complete,
            "prune_blocks": st.prune_blocks, "prune_front_dims": st.prune_front_dims,
            "prune_rows_finished": st.prune_rows_finished, "prune_rows_full": st.prune_rows_full}


def skm_assign_rbq1_noalloc(pts: Points, C, out, dist_out=None, stream=None):
    """RBQ1 assignment that allocates nothing in the library (fixed device
    scratch); `out` (int32[n]) and `dist_out` (float[n] or None) are caller
    tensors."""
    _check(lib().skm_assign_rbq1_noalloc(ctypes.byref(pts.ref), _ptr(C), C.shape[0], _ptr(out), _ptr(dist_out),
                                         _stream(stream)))
    return out, dist_out


def skm_assign_segmented(pts: Points, C, group, base, want_dist=True, ws=None, stream=None, out=None):
    """Rows sorted by group; row r takes the nearest of C[base[g]:base[g+1]], g = group[r]."""
    k = C.shape[0]
    dev = pts.device
    if ws is None:
        ws = _ws(skm_workspace_size(OP_ASSIGN_SEG, pts, k), dev)
    assign = out if out is not None else torch.empty(pts.n, device=dev, dtype=torch.int32)
    dist = torch.empty(pts.n, device=dev, dtype=torch.float32) if want_dist else None
    _check(lib().skm_assign_segmented(ctypes.byref(pts.ref), _ptr(C), int(k), _ptr(group), _ptr(base),
                                      int(base.numel() - 1), _ptr(assign), _ptr(dist), _ptr(ws), ws.numel(),
                                      _stream(stream)))
    return assign, dist


def skm_update(pts: Points, assign, C_inout, counts=None, partial=None, ws=None, stream=None):
    k = C_inout.shape[0] if C_inout is not None else counts.shape[0]
    dev = pts.device
    if ws is None:
        ws = _ws(skm_workspace_size(OP_UPDATE, pts, k), dev)
    if counts is None:
        counts = torch.zeros(k, device=dev, dtype=torch.int64)
    _check(lib().skm_update(ctypes.byref(pts.ref), _ptr(assign), int(k), _ptr(C_inout), _ptr(counts), _ptr(partial),
                            _ptr(ws), ws.numel(), _stream(stream)))
    return C_inout, counts


def skm_merge_partials(dst, src, stream=None):
    et = 0 if dst.dtype == torch.float64 else 1
    _check(lib().skm_merge_partials(_ptr(dst), _ptr(src), dst.numel(), et, _stream(stream)))
    return dst


def skm_update_finalize(pts: Points, partial, counts, C_inout, stream=None):
    _check(lib().skm_update_finalize(ctypes.byref(pts.ref), _ptr(partial), _ptr(counts), C_inout.shape[0],
                                     _ptr(C_inout), _stream(stream)))
    return C_inout


def skm_split_empty(pts: Points, C_inout, counts, stream=None):
    k = C_inout.shape[0]
    ws = _ws(8 * k + 512, pts.device)
    _check(lib().skm_split_empty(ctypes.byref(pts.ref), _ptr(C_inout), _ptr(counts), int(k), _ptr(ws), ws.numel(),
                                 _stream(stream)))
    return C_inout


def skm_forgy_indices(seed, n, k):
    """Seeded Forgy indices (int64 CPU tensor [k]); see include/skm.h."""
    out = torch.empty(int(k), dtype=torch.int64)
    _check(lib().skm_forgy_indices(int(seed) & (2**64 - 1), int(n), int(k), ctypes.c_void_p(out.data_ptr())))
    return out


def skm_fit(pts: Points, k, iters, C_init=None, init_idx=None, want_objective=True, want_dist=True,
            ws=None, stream=None, empty_policy=EMPTY_KEEP, seed=0):
    """Returns (C, assign, dist or None, objective list or None, stats dict).
    With neither C_init nor init_idx the library draws Forgy indices from `seed`."""
    dev = pts.device
    if ws is None:
        ws = _ws(skm_workspace_size(OP_FIT, pts, k), dev)
    if pts.repr == REPR_SQ8:
        C = torch.empty(k, pts.d, device=dev, dtype=torch.uint8)
    else:
        C = torch.empty(k, pts.d, device=dev, dtype=torch.float32)
    assign = torch.empty(pts.n, device=dev, dtype=torch.int32)
    dist = torch.empty(pts.n, device=dev, dtype=torch.float32) if want_dist else None
    obj = (ctypes.c_double * (iters + 1))() if want_objective else None
    st = Stats()
    empties = (ctypes.c_int64 * max(1, min(iters, 4096)))()
    st.empty_per_iter = ctypes.cast(empties, ctypes.c_void_p)
    cfg = FitConfig(int(k), int(iters), int(empty_policy), 0, int(seed) & (2**64 - 1))
    _check(lib().skm_fit(ctypes.byref(cfg), ctypes.byref(pts.ref), _ptr(C_init), _ptr(init_idx), _ptr(C),
                         _ptr(assign), _ptr(dist), obj, ctypes.byref(st), _ptr(ws), ws.numel(), _stream(stream)))
    stats = {"rescored_rows": st.rescored_rows, "fallback_rows": st.fallback_rows,
             "empty_clusters": st.empty_clusters, "prune_first_block": st.prune_first_block,
             "prune_complete": st.prune_complete, "prune_blocks": st.prune_blocks,
             "prune_front_dims": st.prune_front_dims, "prune_rows_finished": st.prune_rows_finished,
             "prune_rows_full": st.prune_rows_full, "cluster_size_std": st.cluster_size_std,
             "empty_per_iter": list(empties)[:min(iters, 4096)]}
    return C, assign, dist, (list(obj) if obj is not None else None), stats


def skm_fit_hierarchical(pts: Points, k, m, meso_init_idx, meso_iters, fine_iters, refine=False, ws=None,
                         stream=None):
    """Returns (C [k], assign [n], meso assign [n], fine counts per meso cluster (list), stats dict)."""
    dev = pts.device
    cfg = HierConfig(int(k), int(m), int(meso_iters), int(fine_iters), int(bool(refine)))
    if ws is None:
        nbytes = lib().skm_hier_workspace_size(ctypes.byref(cfg), ctypes.byref(pts.ref))
        if nbytes == 0:
            raise SkmError(1, lib().skm_last_error().decode())
        ws = _ws(nbytes, dev)
    if pts.repr == REPR_SQ8:
        C = torch.empty(k, pts.d, device=dev, dtype=torch.uint8)
    else:
        C = torch.empty(k, pts.d, device=dev, dtype=torch.float32)
    assign = torch.empty(pts.n, device=dev, dtype=torch.int32)
    meso = torch.empty(pts.n, device=dev, dtype=torch.int32)
    kf = (ctypes.c_int32 * m)()
    st = Stats()
    _check(lib().skm_fit_hierarchical(ctypes.byref(cfg), ctypes.byref(pts.ref), _ptr(meso_init_idx), _ptr(C),
                                      _ptr(assign), _ptr(meso), kf, ctypes.byref(st), _ptr(ws), ws.numel(),
                                      _stream(stream)))
    stats = {"rescored_rows": st.rescored_rows, "fallback_rows": st.fallback_rows}
    return C, assign, meso, list(kf), stats


def skm_objective(X, C, assign, stream=None):
    n, d = X.shape
    is_bf16 = 1 if X.dtype in (torch.bfloat16, torch.int16, torch.uint16) else 0
    ws = _ws(8192, X.device)
    out = ctypes.c_double(0.0)
    _check(lib().skm_objective(_ptr(X), is_bf16, n, d, _ptr(C), C.shape[0], _ptr(assign), ctypes.byref(out),
                               _ptr(ws), ws.numel(), _stream(stream)))
    return out.value


def skm_sq8_decode(codes, b, s, stream=None):
    n, d = codes.shape
    Y = torch.empty(n, d, device=codes.device, dtype=torch.float32)
    _check(lib().skm_sq8_decode(_ptr(codes), n, d, _ptr(b), _ptr(s), _ptr(Y), _stream(stream)))
    return Y


def _host_data(repr_, X_host, d):
    if X_host.device.type != "cpu" or not X_host.is_contiguous():
        raise ValueError("points: a contiguous host tensor")
    return Data(repr_, int(d), X_host.shape[0], X_host.data_ptr(), None, None, None, None, 0, 0, None, None)


class LloydStepHost:
    """skm_lloyd_step_host with its workspace: one Lloyd iteration of points
    held in (pinned) host memory per call.  `exchange` (optional) is a
    callable run between the partial sums and the finalisation; it must
    enqueue its work on the step's stream and then reads/writes the tensors
    `self.partial` and `self.counts`.  warm=True: the host points do not
    change between calls, so each row range's screen starts from the bounds
    its previous call left (one assignment workspace per range).
    prune=True (BF16, with warm): exact pruned assignments seeded with the
    assignments in the assign_host array passed to the call (the previous
    call's, passed back unchanged)."""

    def __init__(self, repr_, X_host, d, k, chunks=16, device=None, copy_stream=None, exchange=None, warm=False,
                 prune=False):
        self.device = torch.device("cuda") if device is None else torch.device(device)
        self.repr, self.k, self.d = repr_, int(k), int(d)
        self.X_host = X_host
        self.ref = _host_data(repr_, X_host, d)
        pdt = torch.int64 if repr_ == REPR_SQ8 else torch.float64
        self.partial = torch.zeros(self.k, self.d, dtype=pdt, device=self.device)
        self.counts = torch.zeros(self.k, dtype=torch.int64, device=self.device)
        self.copy_stream = copy_stream if copy_stream is not None else torch.cuda.Stream(self.device)
        self._user_exchange = exchange
        self._cb = EXCHANGE_FN(self._exchange) if exchange is not None else EXCHANGE_FN()
        self.cfg = StepHostConfig(self.k, int(chunks), ctypes.c_void_p(self.copy_stream.cuda_stream),
                                  self.partial.data_ptr(), self.counts.data_ptr(), self._cb, None, int(bool(warm)),
                                  int(bool(prune)))
        nbytes = lib().skm_step_host_workspace_size(ctypes.byref(self.cfg), ctypes.byref(self.ref))
        if nbytes == 0:
            raise SkmError(1, lib().skm_last_error().decode())
        self.ws = _ws(nbytes, self.device, zero=True)

    def _exchange(self, partial, counts, user, stream):
        # the hook's work goes on the stream this step was called with (the
        # library passes that stream's handle; a handle of 0 is the default
        # stream, which torch.cuda.ExternalStream(0) would not give back)
        try:
            with torch.cuda.stream(self._call_stream):
                self._user_exchange()
            return 0
        except Exception:  # reported to the library as a failed exchange
            return 1

    def __call__(self, C_host, C_host_out=None, assign_host=None, counts_host=None, want_objective=False,
                 stream=None):
        """Returns (C_host_out, assign_host, counts_host or None, objective or None)."""
        n = self.X_host.shape[0]
        C_host_out = C_host if C_host_out is None else C_host_out
        if assign_host is None:
            assign_host = torch.empty(n, dtype=torch.int32, pin_memory=True)
        obj = ctypes.c_double(0.0) if want_objective else None
        self._call_stream = stream if stream is not None else torch.cuda.current_stream(self.device)
        _check(lib().skm_lloyd_step_host(ctypes.byref(self.cfg), ctypes.byref(self.ref), _ptr(C_host),
                                         _ptr(C_host_out), _ptr(assign_host), _ptr(counts_host),
                                         ctypes.byref(obj) if obj is not None else None, _ptr(self.ws),
                                         self.ws.numel(), _stream(self._call_stream)))
        return C_host_out, assign_host, counts_host, (obj.value if obj is not None else None)


FAULT_WORKSPACE, FAULT_LAUNCH, FAULT_STATUS, FAULT_WAIT = 1, 2, 3, 4


def skm_inject_fault(kind, count=1):
    """Arms `count` occurrences of an SKM_FAULT_* (0 disarms); see include/skm.h."""
    _check(lib().skm_inject_fault(int(kind), int(count)))


def skm_fault_armed(kind) -> int:
    return int(lib().skm_fault_armed(int(kind)))


def skm_column_absmax(X, stream=None) -> float:
    """max |x| over a device float32 [n, d] tensor (synchronises)."""
    n, d = X.shape
    ws = _ws(256, X.device)
    out = ctypes.c_float(0.0)
    _check(lib().skm_column_absmax(_ptr(X), n, d, ctypes.byref(out), _ptr(ws), ws.numel(), _stream(stream)))
    return float(out.value)


def skm_mean_scale(amax, n_total) -> int:
    return int(lib().skm_mean_scale(float(amax), int(n_total)))


def skm_column_sums_fixed(X, s, sums, stream=None):
    """sums (device int64 [d]) += per column, the sum of rint(x 2^s) over X's rows."""
    n, d = X.shape
    _check(lib().skm_column_sums_fixed(_ptr(X), n, d, int(s), _ptr(sums), _stream(stream)))
    return sums


def skm_mean_from_sums(sums, n_total, s, stream=None):
    m = torch.empty(sums.numel(), device=sums.device, dtype=torch.float32)
    _check(lib().skm_mean_from_sums(_ptr(sums), int(n_total), sums.numel(), int(s), _ptr(m), _stream(stream)))
    return m


def skm_rbq1_segment_bounds(d):
    a, b = ctypes.c_int(0), ctypes.c_int(0)
    _check(lib().skm_rbq1_segment_bounds(int(d), ctypes.byref(a), ctypes.byref(b)))
    return a.value, b.value


def skm_rbq1_segments(X, m, stream=None):
    """RabitQ segment factors of the points X (device float32 [n, d]) for the
    mean m: (nx2s float32 [n, 3], Fs float32 [n, 3], popxs int32 [n, 3])."""
    n, d = X.shape
    nx2 = torch.empty(n, 3, device=X.device, dtype=torch.float32)
    F = torch.empty(n, 3, device=X.device, dtype=torch.float32)
    pc = torch.empty(n, 3, device=X.device, dtype=torch.int32)
    _check(lib().skm_rbq1_segments(_ptr(X), n, d, _ptr(m), _ptr(nx2), _ptr(F), _ptr(pc), _stream(stream)))
    return nx2, F, pc
