"""Host-side checks of the C ABI that need no GPU: the library loads, exports
every symbol include/skm.h declares, and rejects invalid arguments before
any launch (so fake device pointers are never dereferenced)."""
import ctypes
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def skm():
    from paper_2608_14648_gb300 import build as b

    b.build()
    import paper_2608_14648_gb300 as skm

    return skm


def _declared_symbols():
    src = open(os.path.join(ROOT, "include", "skm.h")).read()
    return sorted(set(re.findall(r"\b(skm_[a-z0-9_]+)\s*\(", src)))


def test_library_exports_every_declared_symbol(skm):
    declared = _declared_symbols()
    assert set(declared) == set(skm.EXPORTED_SYMBOLS)
    L = ctypes.CDLL(skm.lib_path())
    for name in declared:
        assert hasattr(L, name), name
    assert skm.skm_version() >= 100


def _data(skm, repr_=0, n=100, d=16):
    return skm.Data(repr_, d, n, 0x1000, None, None, None, None, 0, 0)


FAKE = ctypes.c_void_p(0x1000)


def test_invalid_arguments_are_rejected_before_launch(skm):
    L = skm.lib()
    x = _data(skm)
    # k > n: allowed for a plain assignment, rejected by fit (Forgy needs k points)
    cfg = skm.FitConfig(101, 3)
    rc = L.skm_fit(ctypes.byref(cfg), ctypes.byref(x), None, FAKE, FAKE, FAKE, None, None, None, FAKE, 1 << 30, None)
    assert rc == 1 and b"exceeds" in L.skm_last_error()
    # k = 0
    assert L.skm_assign(ctypes.byref(x), FAKE, 0, None, FAKE, None, FAKE, 1 << 20, None) == 1
    # d out of range
    bad = _data(skm, d=0)
    assert L.skm_assign(ctypes.byref(bad), FAKE, 4, None, FAKE, None, FAKE, 1 << 20, None) == 1
    big = _data(skm, d=5000)
    assert L.skm_assign(ctypes.byref(big), FAKE, 4, None, FAKE, None, FAKE, 1 << 20, None) == 2
    # unknown repr
    assert L.skm_assign(ctypes.byref(_data(skm, repr_=9)), FAKE, 4, None, FAKE, None, FAKE, 1 << 20, None) == 1
    # NULL centroids / assign
    assert L.skm_assign(ctypes.byref(x), None, 4, None, FAKE, None, FAKE, 1 << 20, None) == 1
    # RBQ1 without its factors
    r = _data(skm, repr_=2)
    assert L.skm_assign(ctypes.byref(r), FAKE, 4, None, FAKE, None, FAKE, 1 << 20, None) == 1
    # workspace too small
    need = L.skm_workspace_size(0, ctypes.byref(_data(skm, repr_=1)), 4)
    assert need > 0
    rc = L.skm_assign(ctypes.byref(_data(skm, repr_=1)), FAKE, 4, None, FAKE, None, FAKE, need - 1, None)
    assert rc == 4
    # misaligned workspace
    rc = L.skm_assign(ctypes.byref(_data(skm, repr_=1)), FAKE, 4, None, FAKE, None, ctypes.c_void_p(0x1010), need,
                      None)
    assert rc == 1
    # BF16 fit without fp32 initial centroids (seeded Forgy cannot build them)
    cfg = skm.FitConfig(4, 3)
    xb = _data(skm, repr_=3)
    rc = L.skm_fit(ctypes.byref(cfg), ctypes.byref(xb), None, None, FAKE, FAKE, None, None, None, FAKE, 1 << 30, None)
    assert rc == 1 and b"C_init" in L.skm_last_error()
    # projection to more dims than the input
    assert L.skm_project(FAKE, 10, 8, None, FAKE, 9, 0, FAKE, None, 0, None) == 1
    # misaligned projection workspace
    assert L.skm_project(FAKE, 10, 8, None, FAKE, 4, 0, FAKE, ctypes.c_void_p(0x1010), 1 << 20, None) == 1
    # projection workspace sizes: one pass >= the chunked minimum
    x8 = _data(skm, n=100000, d=64)
    assert L.skm_workspace_size(6, ctypes.byref(x8), 32) >= L.skm_workspace_size(7, ctypes.byref(x8), 32) > 0
    # unknown workspace op
    assert L.skm_workspace_size(9, ctypes.byref(x), 4) == 0
    # pruning counters: no workspace, no output, a workspace too small for them
    st = skm.Stats()
    assert L.skm_assign_prune_stats(None, 1 << 20, ctypes.byref(st), None) == 1
    assert L.skm_assign_prune_stats(FAKE, 1 << 20, None, None) == 1
    assert L.skm_assign_prune_stats(FAKE, 8, ctypes.byref(st), None) == 1
    # unknown empty-cluster policy
    cfg = skm.FitConfig(4, 3, 7)
    rc = L.skm_fit(ctypes.byref(cfg), ctypes.byref(x), FAKE, None, FAKE, FAKE, None, None, None, FAKE, 1 << 30, None)
    assert rc == 1 and b"empty_policy" in L.skm_last_error()
    # split: k = 0, NULL counts, workspace too small for k int64
    assert L.skm_split_empty(ctypes.byref(x), FAKE, FAKE, 0, FAKE, 1 << 20, None) == 1
    assert L.skm_split_empty(ctypes.byref(x), FAKE, None, 4, FAKE, 1 << 20, None) == 1
    assert L.skm_split_empty(ctypes.byref(x), FAKE, FAKE, 1000, FAKE, 100, None) == 4


def test_workspace_sizes_grow_with_problem(skm):
    L = skm.lib()
    small = L.skm_workspace_size(2, ctypes.byref(_data(skm, n=1000, d=64)), 10)
    large = L.skm_workspace_size(2, ctypes.byref(_data(skm, n=100000, d=64)), 10)
    assert 0 < small < large


def test_make_rotation_is_orthogonal_and_seeded(skm):
    P = skm.skm_make_rotation(7, 48).numpy().astype(np.float64)
    np.testing.assert_allclose(P.T @ P, np.eye(48), atol=2e-6)
    P2 = skm.skm_make_rotation(7, 48).numpy()
    np.testing.assert_array_equal(P.astype(np.float32), P2)
    P3 = skm.skm_make_rotation(8, 48).numpy()
    assert not np.allclose(P2, P3)


def test_lvq4_arguments_are_rejected_before_launch(skm):
    L = skm.lib()

    def lvq_data(n=100, d=16, lvq=0x2000):
        x = skm.Data(skm.REPR_LVQ4, d, n, 0x1000, None, None, None, None, 0, 0)
        x.lvq = lvq
        return x

    # the per-point terms are required and must be 16-byte aligned
    assert L.skm_assign(ctypes.byref(lvq_data(lvq=None)), FAKE, 4, None, FAKE, None, FAKE, 1 << 30, None) == 1
    assert L.skm_assign(ctypes.byref(lvq_data(lvq=0x2004)), FAKE, 4, None, FAKE, None, FAKE, 1 << 30, None) == 1
    # more points than the fixed-point sums allow
    assert L.skm_assign(ctypes.byref(lvq_data(n=(1 << 26) + 1)), FAKE, 4, None, FAKE, None, FAKE, 1 << 40,
                        None) == 2
    # workspace sizes exist for assign / update / fit (tensor path and the d > 1024 path)
    for d in (16, 768, 2048):
        for op in (0, 1, 2):
            assert L.skm_workspace_size(op, ctypes.byref(lvq_data(d=d)), 4) > 0
    # quantize: NULL or misaligned outputs
    qp = skm.QuantParams(0, 0, None, None, None, None, None, None, None)
    assert L.skm_quantize(skm.REPR_LVQ4, FAKE, 10, 16, ctypes.byref(qp), FAKE, FAKE, 1 << 20, None) == 1
    qp.lvq = 0x2008
    assert L.skm_quantize(skm.REPR_LVQ4, FAKE, 10, 16, ctypes.byref(qp), FAKE, FAKE, 1 << 20, None) == 1
    # exponent: misaligned terms
    e = ctypes.c_int(0)
    assert L.skm_lvq4_exponent(ctypes.c_void_p(0x2004), 10, ctypes.byref(e), FAKE, 1 << 20, None) == 1
    # hierarchical fit needs d <= 1024
    cfg = skm.HierConfig(8, 2, 1, 1, 0)
    assert L.skm_hier_workspace_size(ctypes.byref(cfg), ctypes.byref(lvq_data(d=2048))) == 0


def test_symmetric_flag_is_validated(skm):
    L = skm.lib()
    x = _data(skm, repr_=1)  # SQ8
    x.flags = skm.FLAG_SYMMETRIC
    assert L.skm_assign(ctypes.byref(x), FAKE, 4, None, FAKE, None, FAKE, 1 << 30, None) == 1
    r = skm.Data(skm.REPR_RBQ1, 16, 100, 0x1000, FAKE, FAKE, FAKE, FAKE, 0, skm.FLAG_SYMMETRIC)
    assert L.skm_assign_rbq1_noalloc(ctypes.byref(r), FAKE, 4, FAKE, None, None) == 2
    assert L.skm_workspace_size(0, ctypes.byref(r), 4) > 0


def test_kernel_timer_arguments(skm):
    L = skm.lib()
    assert L.skm_kernel_timer_ms(None) == 1  # NULL output: rejected before any CUDA call
    assert L.skm_kernel_timer(0) == 0  # disabling needs no device


def test_copy_from_host_arguments(skm):
    L = skm.lib()
    FAKE = ctypes.c_void_p(0x1000)
    # zero bytes: a no-op that touches nothing
    assert L.skm_copy_from_host(None, None, 0, None) == 0
    # NULL destination or source with bytes to copy: rejected before any CUDA call
    assert L.skm_copy_from_host(None, FAKE, 16, None) == 1
    assert L.skm_copy_from_host(FAKE, None, 16, None) == 1
    assert "NULL" in L.skm_last_error().decode()


def test_step_host_arguments_are_rejected_before_any_work(skm):
    """skm_lloyd_step_host / skm_step_host_workspace_size: bad configurations
    return their status (and size 0) before any CUDA call."""
    L = skm.lib()
    X = np.zeros((100, 16), np.float32)
    x = skm.Data(0, 16, 100, X.ctypes.data, None, None, None, None, 0, 0)

    def cfg(k=10, chunks=4):
        return skm.StepHostConfig(k, chunks, None, None, None, skm.EXCHANGE_FN(), None)

    assert L.skm_step_host_workspace_size(ctypes.byref(cfg()), ctypes.byref(x)) > 0
    # warm: one assignment workspace per range for F32/BF16, nothing extra for SQ8
    warm = cfg()
    warm.warm = 1
    assert L.skm_step_host_workspace_size(ctypes.byref(warm), ctypes.byref(x)) > \
        L.skm_step_host_workspace_size(ctypes.byref(cfg()), ctypes.byref(x))
    x8 = skm.Data(1, 16, 100, X.ctypes.data, None, None, None, None, 0, 0)
    assert L.skm_step_host_workspace_size(ctypes.byref(warm), ctypes.byref(x8)) == \
        L.skm_step_host_workspace_size(ctypes.byref(cfg()), ctypes.byref(x8))
    # prune: BF16 with warm only; the ranges' workspaces then hold survivor lists
    Xb = np.zeros((1000, 256), np.uint16)
    xb = skm.Data(skm.REPR_BF16, 256, 1000, Xb.ctypes.data, None, None, None, None, 0, 0)
    pr = cfg()
    pr.warm, pr.prune = 1, 1
    wb = cfg()
    wb.warm = 1
    assert L.skm_step_host_workspace_size(ctypes.byref(pr), ctypes.byref(xb)) >= \
        L.skm_step_host_workspace_size(ctypes.byref(wb), ctypes.byref(xb)) + 1000 * 256
    cold_prune = cfg()
    cold_prune.prune = 1
    for c, xx in ((cold_prune, xb), (pr, x)):  # without warm; F32 points
        assert L.skm_step_host_workspace_size(ctypes.byref(c), ctypes.byref(xx)) == 0
        assert L.skm_lloyd_step_host(ctypes.byref(c), ctypes.byref(xx), FAKE, FAKE, FAKE, None, None, FAKE,
                                     1 << 30, None) == 2
        assert b"prune" in L.skm_last_error()
    for c, code, what in [(cfg(k=101), 1, b"k = 101"), (cfg(k=0), 1, b"k = 0"), (cfg(chunks=0), 1, b"chunks"),
                          (cfg(chunks=257), 1, b"chunks")]:
        assert L.skm_step_host_workspace_size(ctypes.byref(c), ctypes.byref(x)) == 0
        rc = L.skm_lloyd_step_host(ctypes.byref(c), ctypes.byref(x), FAKE, FAKE, FAKE, None, None, FAKE, 1 << 30,
                                   None)
        assert rc == code and what in L.skm_last_error()
    for repr_ in (2, 4):  # RBQ1 / LVQ4: factors would need copying too
        xr = skm.Data(repr_, 16, 100, X.ctypes.data, None, None, None, None, 0, 0)
        assert L.skm_lloyd_step_host(ctypes.byref(cfg()), ctypes.byref(xr), FAKE, FAKE, FAKE, None, None, FAKE,
                                     1 << 30, None) == 2
    xf = skm.Data(0, 16, 100, X.ctypes.data, None, None, None, None, 0, 1)  # a flag
    assert L.skm_lloyd_step_host(ctypes.byref(cfg()), ctypes.byref(xf), FAKE, FAKE, FAKE, None, None, FAKE,
                                 1 << 30, None) == 2
    # missing outputs / workspace
    assert L.skm_lloyd_step_host(ctypes.byref(cfg()), ctypes.byref(x), FAKE, FAKE, None, None, None, FAKE,
                                 1 << 30, None) == 1
    assert L.skm_lloyd_step_host(ctypes.byref(cfg()), ctypes.byref(x), FAKE, FAKE, FAKE, None, None, None,
                                 1 << 30, None) == 1
    # too small a workspace
    assert L.skm_lloyd_step_host(ctypes.byref(cfg()), ctypes.byref(x), FAKE, FAKE, FAKE, None, None,
                                 ctypes.c_void_p(0x100000), 1024, None) == 4


def test_fault_injection_switch(skm):
    """skm_inject_fault arms occurrences that the first checks use up: an
    armed workspace fault makes a valid call return SKM_ERR_NO_MEMORY before
    anything is enqueued (so the fake pointers are never touched)."""
    L = skm.lib()
    assert L.skm_inject_fault(9, 1) == 1 and L.skm_inject_fault(1, -1) == 1
    assert L.skm_fault_armed(9) == 0
    x = _data(skm)
    try:
        assert L.skm_inject_fault(1, 2) == 0 and L.skm_fault_armed(1) == 2
        for left in (1, 0):
            rc = L.skm_assign(ctypes.byref(x), FAKE, 4, None, FAKE, None, FAKE, 1 << 30, None)
            assert rc == 4 and b"injected" in L.skm_last_error()
            assert L.skm_fault_armed(1) == left
        assert L.skm_inject_fault(2, 5) == 0 and L.skm_inject_fault(2, 0) == 0 and L.skm_fault_armed(2) == 0
    finally:
        for kind in (1, 2, 3, 4):
            L.skm_inject_fault(kind, 0)


def test_fault_injection_from_environment(skm):
    """SKM_FAULT=workspace arms one occurrence when the library first checks."""
    import subprocess
    import sys

    code = (
        "import ctypes, paper_2608_14648_gb300 as skm\n"
        "L = skm.lib()\n"
        "x = skm.Data(0, 16, 100, 0x1000, None, None, None, None, 0, 0)\n"
        "F = ctypes.c_void_p(0x1000)\n"
        "assert L.skm_fault_armed(1) == 1\n"
        "assert L.skm_assign(ctypes.byref(x), F, 4, None, F, None, F, 1 << 30, None) == 4\n"
        "assert L.skm_fault_armed(1) == 0\n"
        "print('ok')\n")
    env = dict(os.environ, SKM_FAULT="workspace")
    r = subprocess.run([sys.executable, "-c", code], cwd=ROOT, env=env, capture_output=True, text=True, timeout=120)
    assert r.returncode == 0 and r.stdout.strip() == "ok", r.stderr


def test_forgy_indices_match_the_oracle(skm):
    """The library's seeded Forgy draw (hash-map Fisher-Yates) equals the
    oracle's (full-array Fisher-Yates) for the same seed: bit-exact."""
    import oracle

    L = skm.lib()
    for seed, n, k in [(0, 10, 10), (1, 1, 1), (7, 1000, 999), (2**40 + 3, 20_000, 100),
                       (0, 10_000_000, 10_000), (2**64 - 1, 1_000_000, 1000)]:
        got = skm.skm_forgy_indices(seed, n, k).numpy()
        np.testing.assert_array_equal(got, oracle.forgy_indices(seed, n, k))
    out = np.empty(4, np.int64)
    assert L.skm_forgy_indices(0, 3, 4, out.ctypes.data) == 1  # k > n
    assert L.skm_forgy_indices(0, 3, 0, out.ctypes.data) == 1
    assert L.skm_forgy_indices(0, 3, 2, None) == 1


def test_rbq1_packed_reading_needs_no_screen_workspace(skm):
    """1-bit rows of a multiple of 16 bytes at a 16-byte aligned address are
    read packed when no e4m3 screening copy is given, so the assignment
    workspace holds per-CTA expansion slots instead of a copy of all points;
    the copy stays available (skm_screen_bytes) for callers who want it."""
    L = skm.lib()

    def data(d, ptr, n):
        return skm.Data(2, d, n, ptr, FAKE, FAKE, FAKE, FAKE, 0, 0)

    n = 1_000_000
    for d in (768, 1024, 100):
        assert L.skm_screen_bytes(ctypes.byref(data(d, 0x1000, n))) >= n * d
        packed = L.skm_workspace_size(0, ctypes.byref(data(d, 0x1000, n)), 1000)
        copied = L.skm_workspace_size(0, ctypes.byref(data(d, 0x1004, n)), 1000)  # misaligned rows
        assert packed < n * d // 4 and copied >= n * d
    # 3 words a row: the copy
    assert L.skm_workspace_size(0, ctypes.byref(data(96, 0x1000, n)), 1000) >= n * 96


def test_lvq4_packed_reading_needs_no_screen_workspace(skm):
    """LVQ4 nibble rows of a multiple of 16 bytes at a 16-byte aligned address
    are read packed when no e4m3 copy is given (per-CTA expansion slots in
    the workspace instead of a copy of all points)."""
    L = skm.lib()

    def data(d, ptr, n):
        return skm.Data(4, d, n, ptr, None, None, None, None, 0, 0, None, FAKE)

    n = 1_000_000
    for d in (768, 1024, 992):
        packed = L.skm_workspace_size(0, ctypes.byref(data(d, 0x1000, n)), 1000)
        copied = L.skm_workspace_size(0, ctypes.byref(data(d, 0x1004, n)), 1000)
        assert packed < n * d // 4 and copied >= n * d
    assert L.skm_workspace_size(0, ctypes.byref(data(1000, 0x1000, n)), 1000) >= n * 1000  # 125 words


def test_prune_front_workspace_holds_survivor_lists(skm):
    """bf16 points with SKM_FLAG_PRUNE, 256 <= d <= 1024, d % 8 == 0 and a
    16-byte aligned base can take the tensor-core front: the workspace then
    holds the per-row survivor lists (64 int32) and thresholds; other
    shapes prune on CUDA cores only and need no per-row buffers."""
    L = skm.lib()

    def data(d, ptr, n):
        x = skm.Data(skm.REPR_BF16, d, n, ptr, None, None, None, None, 0, 0)
        x.flags = skm.FLAG_PRUNE
        return x

    n, k = 100_000, 1000
    for d in (256, 512, 1024):
        ws = L.skm_workspace_size(0, ctypes.byref(data(d, 0x1000, n)), k)
        assert ws >= n * (64 + 5) * 4
    for d, ptr in ((128, 0x1000), (1032, 0x1000), (260, 0x1000), (256, 0x1008)):
        assert L.skm_workspace_size(0, ctypes.byref(data(d, ptr, n)), k) < n * 4
