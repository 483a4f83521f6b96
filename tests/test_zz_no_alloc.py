"""The RBQ1 assignment entry point that allocates nothing.

Some callers cannot allocate device memory (a host engine that owns all
device memory, or a latency-critical path that must not reach cudaMalloc);
skm_assign_rbq1_noalloc serves them from a fixed device array inside the
library.  This checks, through the C ABI, that two calls in a row give the
same assignments and estimated distances as skm_assign, bit for bit (the
tolerance the RBQ1 path is held to), including when the second call uses a
different centroid set than the first.  The file is named to be collected
last."""
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu


def test_noalloc_matches_workspace_entry_point_on_two_calls(cuda_ok):
    import paper_2608_14648_gb300 as skm

    n, d = 20000, 768
    X = synth.gmm_points(n, d, 60, seed=31).cuda()
    pts = skm.rbq1_points(skm.skm_quantize(skm.REPR_RBQ1, X), d)
    for call, (k, seed) in enumerate([(1000, 1), (257, 2)]):
        C = X[synth.forgy_indices(n, k, seed=seed).cuda()].clone()
        a_ref, d_ref = skm.skm_assign(pts, C)
        a = torch.full((n,), -1, dtype=torch.int32, device="cuda")
        dist = torch.full((n,), float("nan"), dtype=torch.float32, device="cuda")
        skm.skm_assign_rbq1_noalloc(pts, C, a, dist)
        torch.cuda.synchronize()
        assert torch.equal(a, a_ref), f"call {call}: assignments differ"
        assert torch.equal(dist, d_ref), f"call {call}: distances differ"


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
