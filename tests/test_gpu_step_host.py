"""skm_lloyd_step_host (one Lloyd iteration of points in pinned host memory,
the copy overlapped with the work) against the device-resident calls on the
same points: skm_assign, then skm_update with partial sums and
skm_update_finalize.  Assignments and counts equal; centroids equal (SQ8,
exact integers) or within 1e-6 relative L2 per centroid (F32/BF16: the
update sums runs of member rows in fp32 before adding them into the fp64
partial sums, and the runs start at other rows when the points arrive in
ranges); the objective equals the fp64 sum of the assignment's distances."""
import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def skm(cuda_ok):
    import paper_2608_14648_gb300 as skm

    skm.lib()
    return skm


def _close_l2(C, C_ref, tol=1e-6):
    c, r = C.double().numpy(), C_ref.double().numpy()
    rel = np.linalg.norm(c - r, axis=1) / np.maximum(np.linalg.norm(r, axis=1), 1e-30)
    assert rel.max() <= tol, f"centroid relative L2 {rel.max()}"


def _reference(skm, pts, C):
    k = C.shape[0]
    a, dist = skm.skm_assign(pts, C)
    pdt = torch.int64 if pts.repr == skm.REPR_SQ8 else torch.float64
    part = torch.zeros(k, pts.d, dtype=pdt, device="cuda")
    cnt = torch.zeros(k, dtype=torch.int64, device="cuda")
    skm.skm_update(pts, a, None, counts=cnt, partial=part)
    C2 = C.clone()
    skm.skm_update_finalize(pts, part, cnt, C2)
    torch.cuda.synchronize()
    return a.cpu(), dist.double().sum().item(), C2.cpu(), cnt.cpu()


def _inputs(skm, kind, n, d, k, seed):
    X = synth.gmm_points(n, d, 30, seed=seed)
    idx = synth.forgy_indices(n, k, seed=seed)
    if kind == "f32":
        return skm.REPR_F32, X.contiguous(), X[idx].clone()
    if kind == "bf16":
        Xb = X.to(torch.bfloat16).view(torch.int16).contiguous()
        C = (Xb[idx].to(torch.int32) << 16).view(torch.float32).contiguous()
        return skm.REPR_BF16, Xb, C
    q = skm.skm_quantize(skm.REPR_SQ8, X.cuda())
    codes = q["codes"].cpu().contiguous()
    return skm.REPR_SQ8, codes, codes[idx].clone()


@pytest.mark.parametrize("kind,n,d,k,chunks", [("f32", 20011, 96, 37, 7), ("bf16", 30000, 256, 300, 16),
                                               ("sq8", 20011, 128, 64, 5), ("f32", 5000, 33, 9, 1),
                                               ("bf16", 4099, 64, 17, 2), ("sq8", 7, 16, 3, 8)])
def test_step_host_matches_device_calls(skm, kind, n, d, k, chunks):
    repr_, Xh, C0 = _inputs(skm, kind, n, d, k, seed=n + d)
    Xp = Xh.pin_memory()
    pts = skm.Points(repr_, Xh.cuda(), d)
    a_ref, obj_ref, C_ref, cnt_ref = _reference(skm, pts, C0.cuda())
    step = skm.LloydStepHost(repr_, Xp, d, k, chunks=chunks)
    C_in = C0.clone().pin_memory()
    C_out = torch.empty_like(C_in).pin_memory()
    cnt = torch.empty(k, dtype=torch.int64)
    for _ in range(2):  # the same inputs twice: the call leaves no state behind
        _, a, _, obj = step(C_in, C_out, counts_host=cnt, want_objective=True)
        assert torch.equal(a, a_ref)
        assert torch.equal(cnt, cnt_ref)
        if repr_ == skm.REPR_SQ8:
            assert torch.equal(C_out, C_ref)
        else:
            _close_l2(C_out, C_ref)
        assert abs(obj - obj_ref) <= 1e-9 * abs(obj_ref)
    assert torch.equal(C_in, C0)  # the input centroids are left alone


def test_step_host_exchange_hook(skm):
    """The hook sees the summed partials: doubling them (two identical ranks
    all-reduced) leaves the means unchanged and doubles the counts; a hook
    that fails ends the call with SKM_ERR_EXCHANGE."""
    repr_, Xh, C0 = _inputs(skm, "f32", 9000, 64, 20, seed=5)
    Xp = Xh.pin_memory()
    pts = skm.Points(repr_, Xh.cuda(), 64)
    a_ref, _, C_ref, cnt_ref = _reference(skm, pts, C0.cuda())
    holder = {}

    def double():
        s = holder["step"]
        s.partial.mul_(2)
        s.counts.mul_(2)

    step = skm.LloydStepHost(repr_, Xp, 64, 20, chunks=4, exchange=double)
    holder["step"] = step
    cnt = torch.empty(20, dtype=torch.int64)
    C_out, a, _, _ = step(C0.clone().pin_memory(), counts_host=cnt)
    assert torch.equal(a, a_ref) and torch.equal(cnt, 2 * cnt_ref)
    _close_l2(C_out, C_ref)

    def broken():
        raise RuntimeError("peer lost")

    bad = skm.LloydStepHost(repr_, Xp, 64, 20, chunks=4, exchange=broken)
    with pytest.raises(skm.SkmError) as ei:
        bad(C0.clone().pin_memory())
    assert ei.value.code == 7
    # the stream and library stay usable after the failed step
    C_out, a, _, _ = step(C0.clone().pin_memory())
    assert torch.equal(a, a_ref)


def test_step_host_rejects_pageable_points(skm):
    repr_, Xh, C0 = _inputs(skm, "f32", 1000, 16, 4, seed=9)
    step = skm.LloydStepHost(repr_, Xh, 16, 4, chunks=2)  # Xh is pageable
    with pytest.raises(skm.SkmError) as ei:
        step(C0.clone())
    assert ei.value.code == 1


@pytest.mark.parametrize("kind,chunks", [("bf16", 16), ("f32", 5)])
def test_step_host_warm_ranges_match_cold(skm, kind, chunks):
    """warm=1: each row range keeps its own assignment workspace and starts
    its screen from the bounds its previous call left.  Over Lloyd
    iterations (each call's output centroids fed to the next) the warm steps
    give the cold steps' assignments (near-ties aside) and centroids."""
    n, d, k = 30011, 128, 200
    repr_, Xh, C0 = _inputs(skm, kind, n, d, k, seed=41)
    Xp = Xh.pin_memory()
    cold = skm.LloydStepHost(repr_, Xp, d, k, chunks=chunks)
    warm = skm.LloydStepHost(repr_, Xp, d, k, chunks=chunks, warm=True)
    assert warm.ws.numel() > cold.ws.numel()
    Cc, Cw = C0.clone().pin_memory(), C0.clone().pin_memory()
    for it in range(4):
        _, a_c, _, _ = cold(Cc, Cc)
        _, a_w, _, _ = warm(Cw, Cw)
        agree = (a_c == a_w).float().mean().item()
        assert agree >= 0.9999, f"iteration {it}: agreement {agree}"
        if agree == 1.0:
            _close_l2(Cw, Cc)


def test_step_host_pruned_ranges_match_device_pruning(skm):
    """prune=1 (BF16, warm): each range's assignment is the exact pruned one
    (tensor-core front seeded with the assignments passed in assign_host,
    bounds kept per range); over Lloyd iterations it equals the device-side
    pruned assignment bit for bit, and the centroids follow."""
    n, d, k, chunks = 30000, 256, 300, 4
    repr_, Xh, C0 = _inputs(skm, "bf16", n, d, k, seed=43)
    Xp = Xh.pin_memory()
    Xd = Xh.cuda()
    pc = skm.Points(skm.REPR_BF16, Xd, d, flags=skm.FLAG_PRUNE)
    dense = skm.Points(skm.REPR_BF16, Xd, d)
    hstep = skm.LloydStepHost(repr_, Xp, d, k, chunks=chunks, warm=True, prune=True)
    warm_only = skm.LloydStepHost(repr_, Xp, d, k, chunks=chunks, warm=True)
    assert hstep.ws.numel() > warm_only.ws.numel()
    a0, _ = skm.skm_assign(dense, C0.cuda())  # the first call's seeds
    a_host = a0.cpu().pin_memory()
    C = C0.clone().pin_memory()
    for it in range(4):
        a_ref, _ = skm.skm_assign(pc, C.cuda())
        part = torch.zeros(k, d, dtype=torch.float64, device="cuda")
        cnt = torch.zeros(k, dtype=torch.int64, device="cuda")
        skm.skm_update(pc, a_ref, None, counts=cnt, partial=part)
        C_ref = C.cuda().clone()
        skm.skm_update_finalize(pc, part, cnt, C_ref)
        torch.cuda.synchronize()
        C_out = torch.empty_like(C).pin_memory()
        hstep(C, C_out, a_host)
        assert torch.equal(a_host, a_ref.cpu()), f"iteration {it}"
        _close_l2(C_out, C_ref.cpu())
        C = C_out


def test_step_host_pruned_shared_centroid_prep_uneven_ranges(skm):
    """prune=1 over 5 uneven ranges: the ranges after the first take the
    tensor-core front's centroid side from the first range's call (each
    checking its own kept bounds against the generation of the shared
    previous centroids).  Steps that want the objective (exact seed distances
    in every range) alternate with steps that use the kept bounds; every
    step's assignment equals the device-side pruned assignment bit for bit,
    the objective equals the fp64 sum of its distances, and the centroids
    follow."""
    n, d, k, chunks = 23457, 256, 257, 5
    repr_, Xh, C0 = _inputs(skm, "bf16", n, d, k, seed=47)
    Xp = Xh.pin_memory()
    Xd = Xh.cuda()
    pc = skm.Points(skm.REPR_BF16, Xd, d, flags=skm.FLAG_PRUNE)
    dense = skm.Points(skm.REPR_BF16, Xd, d)
    hstep = skm.LloydStepHost(repr_, Xp, d, k, chunks=chunks, warm=True, prune=True)
    a0, _ = skm.skm_assign(dense, C0.cuda())
    a_host = a0.cpu().pin_memory()
    C = C0.clone().pin_memory()
    for it in range(5):
        a_ref, d_ref = skm.skm_assign(pc, C.cuda())
        part = torch.zeros(k, d, dtype=torch.float64, device="cuda")
        cnt = torch.zeros(k, dtype=torch.int64, device="cuda")
        skm.skm_update(pc, a_ref, None, counts=cnt, partial=part)
        C_ref = C.cuda().clone()
        skm.skm_update_finalize(pc, part, cnt, C_ref)
        torch.cuda.synchronize()
        C_out = torch.empty_like(C).pin_memory()
        want = it % 2 == 1
        _, _, _, obj = hstep(C, C_out, a_host, want_objective=want)
        assert torch.equal(a_host, a_ref.cpu()), f"iteration {it}"
        if want:
            assert obj == pytest.approx(d_ref.double().sum().item(), rel=1e-12)
        _close_l2(C_out, C_ref.cpu())
        C = C_out
