"""The RBQ1 assignment entry point that allocates nothing.

Some callers cannot allocate device memory (a host engine that owns all
device memory, or a latency-critical path that must not reach cudaMalloc);
skm_assign_rbq1_noalloc serves them from a fixed device array inside the
library.  This checks, through the C ABI, that two calls in a row give the
same assignments and estimated distances as skm_assign, bit for bit (the
tolerance the RBQ1 path is held to), including when the second call uses a
different centroid set than the first, at the edges of the fixed scratch
(k = 1 and 3, k * ceil(d/32) exactly at its 131072-word limit, d above 1024
where skm_assign itself takes the popcount kernel), and that entries of the
output buffers past the last point are left alone.  The file is named to be
collected last."""
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu


def _check_two_calls(skm, X, pts, n, calls):
    guard = 16
    for call, (k, seed) in enumerate(calls):
        C = X[synth.forgy_indices(n, k, seed=seed).cuda()].clone()
        a_ref, d_ref = skm.skm_assign(pts, C)
        a_buf = torch.full((n + guard,), -7, dtype=torch.int32, device="cuda")
        d_buf = torch.full((n + guard,), -3.5, dtype=torch.float32, device="cuda")
        a_buf[:n] = -1
        d_buf[:n] = float("nan")
        skm.skm_assign_rbq1_noalloc(pts, C, a_buf[:n], d_buf[:n])
        torch.cuda.synchronize()
        assert torch.equal(a_buf[:n], a_ref), f"call {call} (k={k}): assignments differ"
        assert torch.equal(d_buf[:n], d_ref), f"call {call} (k={k}): distances differ"
        assert bool((a_buf[n:] == -7).all()) and bool((d_buf[n:] == -3.5).all()), \
            f"call {call} (k={k}): wrote past the last point"


def test_noalloc_matches_workspace_entry_point_on_two_calls(cuda_ok):
    import paper_2608_14648_gb300 as skm

    n, d = 20000, 768
    X = synth.gmm_points(n, d, 60, seed=31).cuda()
    pts = skm.rbq1_points(skm.skm_quantize(skm.REPR_RBQ1, X), d)
    _check_two_calls(skm, X, pts, n, [(1000, 1), (257, 2)])


def test_noalloc_smallest_k(cuda_ok):
    import paper_2608_14648_gb300 as skm

    n, d = 5003, 200
    X = synth.gmm_points(n, d, 8, seed=32).cuda()
    pts = skm.rbq1_points(skm.skm_quantize(skm.REPR_RBQ1, X), d)
    _check_two_calls(skm, X, pts, n, [(1, 3), (3, 4)])


def test_noalloc_at_the_plane_word_limit(cuda_ok):
    import paper_2608_14648_gb300 as skm

    n, d = 6000, 1024  # k * ceil(d/32) = 4096 * 32 = 131072, the scratch's limit
    X = synth.gmm_points(n, d, 40, seed=33).cuda()
    pts = skm.rbq1_points(skm.skm_quantize(skm.REPR_RBQ1, X), d)
    _check_two_calls(skm, X, pts, n, [(4096, 5), (4000, 6)])


def test_noalloc_beyond_d_1024(cuda_ok):
    import paper_2608_14648_gb300 as skm

    n, d = 4001, 1100  # skm_assign takes the AND + popcount kernel here too
    X = synth.gmm_points(n, d, 20, seed=34).cuda()
    pts = skm.rbq1_points(skm.skm_quantize(skm.REPR_RBQ1, X), d)
    _check_two_calls(skm, X, pts, n, [(300, 7), (31, 8)])


def test_noalloc_rejects_sizes_beyond_its_scratch(cuda_ok):
    import paper_2608_14648_gb300 as skm

    n, d = 20000, 1024
    X = synth.gmm_points(n, d, 10, seed=3).cuda()
    pts = skm.rbq1_points(skm.skm_quantize(skm.REPR_RBQ1, X), d)
    C = X[:4200].clone()  # 4200 * 32 words > 131072
    a = torch.empty(n, dtype=torch.int32, device="cuda")
    with pytest.raises(skm.SkmError) as ei:
        skm.skm_assign_rbq1_noalloc(pts, C, a)
    assert ei.value.code == 2
