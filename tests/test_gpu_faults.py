"""Error paths, made to run by host-side fault injection (skm_inject_fault),
without faulting the GPU: a bounded device wait on a barrier that nothing
arrives on gives up (SKM_ERR_TIMEOUT), a launch is reported failed
(SKM_ERR_CUDA), skm_fit's device status word is set (SKM_ERR_DEVICE_CHECK),
a workspace check fails (SKM_ERR_NO_MEMORY).  After each, the next call on
the same stream succeeds and gives the same result as before the fault."""
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu

WORKSPACE, LAUNCH, STATUS, WAIT = 1, 2, 3, 4


@pytest.fixture(scope="module")
def skm(cuda_ok):
    import paper_2608_14648_gb300 as skm

    skm.lib()
    yield skm
    for kind in (WORKSPACE, LAUNCH, STATUS, WAIT):
        skm.skm_inject_fault(kind, 0)


def _sq8_points(skm, n=6000, d=96):
    X = synth.gmm_points(n, d, 20, seed=61).cuda()
    q = skm.skm_quantize(skm.REPR_SQ8, X)
    return skm.Points(skm.REPR_SQ8, q["codes"], d), X


def _fit(skm, pts, k, idx):
    C, a, _, _, _ = skm.skm_fit(pts, k, 3, init_idx=idx, want_objective=False, want_dist=False)
    torch.cuda.synchronize()
    return C, a


@pytest.mark.parametrize("kind,code", [(WAIT, 5), (STATUS, 6), (LAUNCH, 3), (WORKSPACE, 4)])
def test_injected_fault_then_clean_fit(skm, kind, code):
    pts, _ = _sq8_points(skm)
    k = 40
    idx = synth.forgy_indices(pts.n, k, seed=1).cuda()
    C0, a0 = _fit(skm, pts, k, idx)
    skm.skm_inject_fault(kind, 1)
    with pytest.raises(skm.SkmError) as ei:
        _fit(skm, pts, k, idx)
    torch.cuda.synchronize()
    assert ei.value.code == code, str(ei.value)
    assert skm.skm_fault_armed(kind) == 0
    C1, a1 = _fit(skm, pts, k, idx)  # same stream, nothing left behind
    assert torch.equal(C1, C0) and torch.equal(a1, a0)


@pytest.mark.parametrize("repr_name", ["f32", "rbq1"])
def test_injected_wait_in_each_tensor_core_mode(skm, repr_name):
    """The injected wait gives up before any load in the fp32 screen and the
    e4m3 1-bit kernels too; skm_fit reports the timeout and the next fit is
    unaffected."""
    n, d, k = 5000, 128, 30
    X = synth.gmm_points(n, d, 20, seed=62).cuda()
    idx = synth.forgy_indices(n, k, seed=2).cuda()
    if repr_name == "f32":
        pts = skm.Points(skm.REPR_F32, X, d)
    else:
        pts = skm.rbq1_points(skm.skm_quantize(skm.REPR_RBQ1, X), d)
    _, a0 = _fit(skm, pts, k, idx)
    skm.skm_inject_fault(WAIT, 2)
    with pytest.raises(skm.SkmError) as ei:
        _fit(skm, pts, k, idx)
    assert ei.value.code == 5
    assert skm.skm_fault_armed(WAIT) == 0
    _, a1 = _fit(skm, pts, k, idx)
    assert torch.equal(a1, a0)


def test_injected_launch_fault_in_assign(skm):
    pts, _ = _sq8_points(skm, n=3000, d=64)
    C = pts.x[:25].clone()
    a0, d0 = skm.skm_assign(pts, C)
    skm.skm_inject_fault(LAUNCH, 1)
    with pytest.raises(skm.SkmError) as ei:
        skm.skm_assign(pts, C)
    torch.cuda.synchronize()
    assert ei.value.code == 3
    a1, d1 = skm.skm_assign(pts, C)
    assert torch.equal(a1, a0) and torch.equal(d1, d0)
