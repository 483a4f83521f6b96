#!/usr/bin/env python
"""Benchmark of the Lloyd k-means hot path on GB300.

Workload: 1,000,000 unit-norm synthetic embeddings, d = 768 (2,000-component
Gaussian mixture, per-dimension variance (1+j)^-0.5, Haar rotation, L2
normalisation), k = 1,000, clustered both as raw fp32 and as RabitQ 1-bit
codes.  One step = one Lloyd iteration (assign + update) of each
representation, i.e. 2 * N * k point-centroid distances.  Metric:
point-centroid distances per second per Lloyd iteration.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

N > 1 runs under torchrun, one rank per GPU: every rank clusters its own
1M-point shard (weak scaling) and the update's cluster sums and counts are
all-reduced once per representation per step (the path's one exchange).
--impl reference times the CPU oracle on a bounded sample of the workload.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

N_POINTS, DIM, K, N_COMP = 1_000_000, 768, 1000, 2000
METRIC = "k-means point·centroid distances/s per Lloyd iter (1 GB300); % of roofline"
WORKLOAD = "emb1m_d768: N=1,000,000 x d=768 unit-norm GMM embeddings, k=1,000; fp32 + RabitQ 1-bit"
SM_COUNT = 152
# row ranges of the end-to-end step's host-to-device copy (overlapped with work)
E2E_CHUNKS = 16
# POPC results per clock per SM used for the 1-bit kernel's ALU roofline
# (measured 15.9 on GB300 with a throughput probe).
POPC_PER_CLK_SM = 16
# DRAM bytes (read + write) per point of the assignment kernels, from one ncu
# capture each (200,000 points x d=768, k=1000; profiles/tc_assign_*.md).
# Each point row is read once per launch, so traffic scales with the points.
TRAFFIC_PER_POINT = {
    "assign_f32": (314.849280e6 + 5.701888e6) / 200_000,
    "assign_rbq1": (156.890624e6 + 3.590912e6) / 200_000,
}


def env_rank():
    return (int(os.environ.get("RANK", "0")), int(os.environ.get("LOCAL_RANK", "0")),
            int(os.environ.get("WORLD_SIZE", "1")))


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            j = json.load(f)
        return {"hbm_gbs": j["hbm_gbs"], "bf16_tflops": j["bf16_tflops"],
                "bf16_tflops_sustained": j.get("bf16_tflops_sustained", j["bf16_tflops"]),
                "sm_max_mhz": j.get("sm_max_mhz", 2070.0), "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "sm_max_mhz": 2070.0,
            "source": "fallback"}


class ClockSampler:
    """nvidia-smi samples (200 ms) of SM clock and throttle reasons while running."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu_index = gpu_index
        self.proc = None
        self.lines = []
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "200",
                 "-i", str(self.gpu_index)], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, ValueError):
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        if self.thread:
            self.thread.join(timeout=2)
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(nm)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm)}


# ----------------------------------------------------------------------------
def cpu_baseline_sample(X_host, C32, codes, nx2, F, popx, m, e, Cr, budget_s=12.0):
    """Oracle (as it stands) on a bounded row sample: one Lloyd iteration of
    each representation.  Returns (distances/s, rows, seconds, threads)."""
    import oracle

    def one(ns):
        t0 = time.perf_counter()
        a, _, _ = oracle.assign_f32(X_host[:ns], C32)
        oracle.update_f32(X_host[:ns], a, C32)
        prep = oracle.rbq1_centroid_sq4(Cr, m)
        ar, _ = oracle.rbq1_assign(codes[:ns], nx2[:ns], F[:ns], popx[:ns], DIM, prep)
        oracle.rbq1_update(codes[:ns], F[:ns], DIM, m, e, ar, Cr)
        return time.perf_counter() - t0

    t0 = one(500)
    ns = int(min(X_host.shape[0], max(500, 500 * budget_s / max(t0, 1e-3))))
    t = one(ns)
    return 2.0 * ns * K / t, ns, t, oracle.num_threads()


def run_ours(args):
    import numpy as np
    import torch

    import paper_2608_14648_gb300 as skm
    import synth

    rank, local_rank, world = env_rank()
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    dist = None
    if world > 1:
        import torch.distributed as dist

        from paper_2608_14648_gb300 import dist as skd

        dist.init_process_group("nccl")
    peaks = load_peaks()

    # ---- inputs (per-rank shard), resident in HBM before timing -------------
    X = synth.gmm_points(N_POINTS, DIM, N_COMP, seed=rank, device=dev)
    idx = synth.forgy_indices(N_POINTS, K, seed=0).to(dev)
    C32 = X[idx].clone()
    if world > 1:
        dist.broadcast(C32, 0)
    pts32 = skm.Points(skm.REPR_F32, X, DIM).with_screen()  # bf16 screening copy, built once
    q = skm.skm_quantize(skm.REPR_RBQ1, X)
    if world > 1:  # global mean, then re-encode; global fixed-point exponent
        m = skd.global_mean(q["m"].double() * N_POINTS, N_POINTS)
        q = skm.skm_quantize(skm.REPR_RBQ1, X, fit=False, m=m.contiguous())
    e = skm.skm_rbq1_exponent(q["F"])
    if world > 1:
        e = skd.global_exponent(e, dev)
    ptsR = skm.rbq1_points(q, DIM, e).with_screen()  # e4m3 expansion of the bits, built once
    Cr, _, _, _, _ = skm.skm_fit(ptsR, K, 0, init_idx=idx, want_objective=False, want_dist=False)
    if world > 1:
        dist.broadcast(Cr, 0)

    wsA32 = skm.workspace(skm.OP_ASSIGN, pts32, K)
    wsU32 = skm.workspace(skm.OP_UPDATE, pts32, K)
    wsAR = skm.workspace(skm.OP_ASSIGN, ptsR, K)
    wsUR = skm.workspace(skm.OP_UPDATE, ptsR, K)
    a32 = torch.empty(N_POINTS, dtype=torch.int32, device=dev)
    aR = torch.empty(N_POINTS, dtype=torch.int32, device=dev)
    cnt32 = torch.zeros(K, dtype=torch.int64, device=dev)
    cntR = torch.zeros(K, dtype=torch.int64, device=dev)
    part32 = torch.zeros(K, DIM, dtype=torch.float64, device=dev) if world > 1 else None
    partR = torch.zeros(K, DIM + 1, dtype=torch.int64, device=dev) if world > 1 else None
    stream = torch.cuda.current_stream()
    ev = {name: [] for name in ("a32", "aR")}

    def lloyd(pts, C, a, cnt, part, wsA, wsU, key, record):
        if record:
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
        skm.skm_assign(pts, C, K, want_dist=False, ws=wsA, out=a)
        if record:
            e1.record(stream)
            ev[key].append((e0, e1))
        if part is None:
            skm.skm_update(pts, a, C, counts=cnt, ws=wsU)
        else:
            part.zero_()
            cnt.zero_()
            skm.skm_update(pts, a, None, counts=cnt, partial=part, ws=wsU)
            skd.allreduce_partials(part, cnt)
            skm.skm_update_finalize(pts, part, cnt, C)

    def step(record):
        lloyd(pts32, C32, a32, cnt32, part32, wsA32, wsU32, "a32", record)
        lloyd(ptsR, Cr, aR, cntR, partR, wsAR, wsUR, "aR", record)

    for _ in range(args.warmup):
        step(False)
    torch.cuda.synchronize()
    # One GPU: the step (both Lloyd iterations, every kernel of assign and
    # update) is captured once in a CUDA graph and replayed, so no host launch
    # gap sits between kernels; the library's launch counter during the
    # capture gives the kernels per step.  Several GPUs: eager (the exchange is
    # an NCCL all-reduce between the ranks).
    graph, launches_per_step, graph_note = None, None, None
    if world == 1 and not args.eager:
        try:
            side = torch.cuda.Stream()
            side.wait_stream(stream)
            with torch.cuda.stream(side):
                step(False)
            stream.wait_stream(side)
            torch.cuda.synchronize()
            l0 = skm.skm_kernel_launches()
            graph = torch.cuda.CUDAGraph()
            with torch.cuda.graph(graph):
                step(False)
            launches_per_step = skm.skm_kernel_launches() - l0
            graph.replay()
            torch.cuda.synchronize()
        except Exception as exc:
            graph, graph_note = None, f"graph capture failed, eager steps: {exc!r}"[:200]
    if world > 1:
        dist.barrier()
    clocks = ClockSampler(local_rank)
    clocks.start()
    torch.cuda.synchronize()
    launches0 = skm.skm_kernel_launches()
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t_start.record(stream)
    for _ in range(args.steps):
        if graph is not None:
            graph.replay()
        else:
            step(True)
    t_end.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    launches = (launches_per_step * args.steps if graph is not None
                else skm.skm_kernel_launches() - launches0)
    if graph is not None:  # per-kernel event times from eager steps after the timed region
        for _ in range(3):
            step(True)
        torch.cuda.synchronize()
    clk = clocks.stop()
    ms = t_start.elapsed_time(t_end)
    if world > 1:
        t = torch.tensor([ms], device=dev, dtype=torch.float64)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ms = float(t.item())
    ms_step = ms / args.steps
    value = world * 2.0 * N_POINTS * K * args.steps / (ms / 1e3)

    # ---- the AND+popcount 1-bit kernel, timed beside the tensor-core one --------
    t_pop = None
    if not args.no_popcount:
        torch.cuda.synchronize()
        p0, p1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a_pop = torch.empty_like(aR)
        skm.skm_assign_rbq1_noalloc(ptsR, Cr, a_pop)
        p0.record(stream)
        skm.skm_assign_rbq1_noalloc(ptsR, Cr, a_pop)
        p1.record(stream)
        torch.cuda.synchronize()
        t_pop = p0.elapsed_time(p1)

    # ---- roofline of the dominant kernel --------------------------------------
    t_a32 = statistics.mean(a.elapsed_time(b) for a, b in ev["a32"])
    t_aR = statistics.mean(a.elapsed_time(b) for a, b in ev["aR"])
    long_region = ms > 1000.0
    bf16_peak = peaks["bf16_tflops_sustained"] if long_region else peaks["bf16_tflops"]
    fp8_peak = 2.0 * bf16_peak  # nominal dense e4m3 : bf16 ratio (4.5 : 2.25 PFLOP/s)
    flops = 2.0 * N_POINTS * K * DIM
    W = (DIM + 31) // 32
    popc_aR = float(N_POINTS) * K * 4 * W
    popc_peak = SM_COUNT * POPC_PER_CLK_SM * peaks["sm_max_mhz"] * 1e6  # per second
    kernels = {
        "assign_f32": {"ms": t_a32, "bound": "tensor", "achieved": flops / (t_a32 / 1e3) / 1e12,
                       "peak": bf16_peak, "unit": "TFLOP/s",
                       "algorithmic": f"2*N*k*d = {flops:.3e} bf16 flop per launch (screen GEMM)"},
        "assign_rbq1": {"ms": t_aR, "bound": "tensor", "achieved": flops / (t_aR / 1e3) / 1e12,
                        "peak": fp8_peak, "unit": "TFLOP/s",
                        "algorithmic": f"2*N*k*d = {flops:.3e} e4m3 flop per launch (exact integer P)"},
    }
    if t_pop is not None:
        kernels["assign_rbq1_popcount"] = {
            "ms": t_pop, "bound": "alu", "achieved": popc_aR / (t_pop / 1e3) / 1e12,
            "peak": popc_peak / 1e12, "unit": "Tpopc/s", "in_step": False,
            "algorithmic": f"N*k*4*ceil(d/32) = {popc_aR:.3e} POPC per launch"}
    for kd in kernels.values():
        kd["frac"] = kd["achieved"] / kd["peak"]
    dom = max((n for n in kernels if kernels[n].get("in_step", True)), key=lambda n: kernels[n]["ms"])
    kd = kernels[dom]
    traffic = TRAFFIC_PER_POINT.get(dom)
    roofline = {"bound": kd["bound"], "achieved": round(kd["achieved"], 4), "peak": round(kd["peak"], 4),
                "unit": kd["unit"], "frac": round(kd["frac"], 5),
                "traffic": round(traffic * N_POINTS) if traffic else None, "kernel": dom,
                "peak_source": f"{peaks['source']} ({'sustained' if long_region else 'burst'} bf16"
                               f"{', x2 for e4m3' if dom == 'assign_rbq1' else ''})"}

    # ---- end to end through the C ABI with host buffers ----------------------
    e2e = None
    if not args.no_e2e:
        X_host = torch.empty(N_POINTS, DIM, dtype=torch.float32, pin_memory=True)
        X_host.copy_(X)
        C_host32 = torch.empty(K, DIM, dtype=torch.float32, pin_memory=True)
        C_hostR = torch.empty(K, DIM, dtype=torch.float32, pin_memory=True)
        C_host32.copy_(C32)
        C_hostR.copy_(Cr)
        a_host = torch.empty(2, N_POINTS, dtype=torch.int32, pin_memory=True)
        # two device buffers for the points: step t + 1's copy streams in while
        # step t is still being assigned and updated (the next step's points do
        # not depend on this step; its centroids do, and wait for the D2H)
        Xbuf = [torch.empty_like(X), torch.empty_like(X)]
        Cd32 = torch.empty_like(C32)
        CdR = torch.empty_like(Cr)
        # The H2D copy of the points is cut into E2E_CHUNKS row ranges on a copy
        # stream; each range is assigned (fp32: screening copy built inside the
        # call; 1-bit: encoded, then assigned) and its fp32 cluster sums are
        # added into fp64 partial sums (the sharded update form) as soon as it
        # has landed, so the copy of later ranges overlaps the work on earlier
        # ones.  The fp32 update is finalised after the last range; the 1-bit
        # update needs the fixed-point exponent of every F and runs after it.
        nchunk = E2E_CHUNKS
        bounds = [(i * N_POINTS // nchunk, (i + 1) * N_POINTS // nchunk) for i in range(nchunk)]
        cmax = max(b1 - b0 for b0, b1 in bounds)
        W = (DIM + 31) // 32
        codesE = torch.empty(N_POINTS, W, device=dev, dtype=torch.int32)
        nx2E = torch.empty(N_POINTS, device=dev, dtype=torch.float32)
        FE = torch.empty(N_POINTS, device=dev, dtype=torch.float32)
        popxE = torch.empty(N_POINTS, device=dev, dtype=torch.int32)
        mE = q["m"]
        probe32 = skm.Points(skm.REPR_F32, Xbuf[0][:cmax], DIM)
        wsA2 = skm.workspace(skm.OP_ASSIGN, probe32, K)
        wsAR2 = skm.workspace(skm.OP_ASSIGN, skm.Points(skm.REPR_RBQ1, codesE[:cmax], DIM, nx2E[:cmax],
                                                        FE[:cmax], popxE[:cmax], mE, e), K)
        wsQ2 = skm.workspace(skm.OP_QUANTIZE, probe32, 1)
        part32e = torch.zeros(K, DIM, device=dev, dtype=torch.float64)
        cnt32e = torch.zeros(K, device=dev, dtype=torch.int64)
        wsU2 = skm.workspace(skm.OP_UPDATE, probe32, K)
        copy_stream = torch.cuda.Stream()   # the points, one step ahead
        cent_stream = torch.cuda.Stream()   # the centroids, after the previous step's D2H
        e2e_steps = max(2, min(args.steps, 5))
        landed = [[torch.cuda.Event() for _ in range(nchunk)] for _ in range(2)]
        c_landed = torch.cuda.Event()
        buf_free = [torch.cuda.Event(), torch.cuda.Event()]
        d2h_done = torch.cuda.Event()
        # per-range point descriptors over the fixed device buffers (views)
        pcs = [[skm.Points(skm.REPR_F32, xb[b0:b1], DIM) for b0, b1 in bounds] for xb in Xbuf]
        qouts = [{"codes": codesE[b0:b1], "nx2": nx2E[b0:b1], "F": FE[b0:b1], "popx": popxE[b0:b1]}
                 for b0, b1 in bounds]
        prcs = [skm.Points(skm.REPR_RBQ1, codesE[b0:b1], DIM, nx2E[b0:b1], FE[b0:b1], popxE[b0:b1], mE, e)
                for b0, b1 in bounds]
        pall = [skm.Points(skm.REPR_F32, xb, DIM) for xb in Xbuf]
        host_ms = []
        h2d = X_host.numel() * 4 + 2 * K * DIM * 4
        d2h = 2 * N_POINTS * 4 + 2 * K * DIM * 4
        # the host link's copy rate just before the run (the e2e step is bound by
        # it; it varies with other traffic on the shared host)
        torch.cuda.synchronize()
        p0, p1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        p0.record(stream)
        Xbuf[0].copy_(X_host, non_blocking=True)
        p1.record(stream)
        torch.cuda.synchronize()
        h2d_probe_gbs = X_host.numel() * 4 / (p0.elapsed_time(p1) / 1e3) / 1e9

        def enqueue_points(t):
            slot = t % 2
            if t >= 2:
                copy_stream.wait_event(buf_free[slot])  # step t - 2 is done with this buffer
            with torch.cuda.stream(copy_stream):
                for (b0, b1), ev in zip(bounds, landed[slot]):
                    Xbuf[slot][b0:b1].copy_(X_host[b0:b1], non_blocking=True)
                    ev.record(copy_stream)

        def e2e_run(nsteps):
            """nsteps end-to-end steps; the device time from the first copy to the
            last step's D2H (ms)."""
            s0, s1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            s0.record(stream)
            copy_stream.wait_stream(stream)
            cent_stream.wait_stream(stream)
            enqueue_points(0)
            for t in range(nsteps):
                th0 = time.perf_counter()
                slot = t % 2
                if t + 1 < nsteps:
                    enqueue_points(t + 1)
                if t > 0:
                    cent_stream.wait_event(d2h_done)  # this step's centroids are the last step's results
                # by the SMs, not a copy engine: there they would queue behind the
                # next step's point ranges
                skm.skm_copy_from_host(Cd32, C_host32, stream=cent_stream)
                skm.skm_copy_from_host(CdR, C_hostR, stream=cent_stream)
                c_landed.record(cent_stream)
                stream.wait_event(c_landed)
                part32e.zero_()
                cnt32e.zero_()
                xb = Xbuf[slot]
                for (b0, b1), ev, pc, qo, prc in zip(bounds, landed[slot], pcs[slot], qouts, prcs):
                    stream.wait_event(ev)
                    skm.skm_assign(pc, Cd32, K, want_dist=False, ws=wsA2, out=a32[b0:b1])
                    skm.skm_update(pc, a32[b0:b1], None, counts=cnt32e, partial=part32e, ws=wsU2)
                    skm.skm_quantize(skm.REPR_RBQ1, xb[b0:b1], fit=False, m=mE, ws=wsQ2, out=qo)
                    skm.skm_assign(prc, CdR, K, want_dist=False, ws=wsAR2, out=aR[b0:b1])
                buf_free[slot].record(stream)
                if world > 1:  # the same exchange as the device-resident step
                    skd.allreduce_partials(part32e, cnt32e)
                skm.skm_update_finalize(pall[slot], part32e, cnt32e, Cd32)
                host_ms.append((time.perf_counter() - th0) * 1e3)  # enqueue only (no sync so far)
                eE = skm.skm_rbq1_exponent(FE)
                if world > 1:
                    eE = skd.global_exponent(eE, dev)
                pR2 = skm.Points(skm.REPR_RBQ1, codesE, DIM, nx2E, FE, popxE, mE, eE)
                if world > 1:
                    partR.zero_()
                    cntR.zero_()
                    skm.skm_update(pR2, aR, None, counts=cntR, partial=partR, ws=wsUR)
                    skd.allreduce_partials(partR, cntR)
                    skm.skm_update_finalize(pR2, partR, cntR, CdR)
                else:
                    skm.skm_update(pR2, aR, CdR, counts=cntR, ws=wsUR)
                a_host[0].copy_(a32, non_blocking=True)
                a_host[1].copy_(aR, non_blocking=True)
                C_host32.copy_(Cd32, non_blocking=True)
                C_hostR.copy_(CdR, non_blocking=True)
                d2h_done.record(stream)
            s1.record(stream)
            torch.cuda.synchronize()
            return s0.elapsed_time(s1)

        e2e_run(2)  # warm-up (first-use costs of the range-sized calls), untimed
        host_ms.clear()
        if world > 1:
            dist.barrier()
        def timed_e2e():
            t_ms = e2e_run(e2e_steps)
            if world > 1:
                t = torch.tensor([t_ms], device=dev, dtype=torch.float64)
                dist.all_reduce(t, op=dist.ReduceOp.MAX)
                t_ms = float(t.item())
            return t_ms

        ems = timed_e2e()
        # The host link is shared with the host's other traffic: a run whose
        # copies averaged under 3/4 of the rate probed just before it is taken
        # again once (both attempts are reported).
        probe = h2d_probe_gbs
        if world > 1:
            t = torch.tensor([probe], device=dev, dtype=torch.float64)
            dist.all_reduce(t, op=dist.ReduceOp.MIN)
            probe = float(t.item())
        first_attempt = None
        if h2d / (ems / e2e_steps / 1e3) / 1e9 < 0.75 * probe:
            first_attempt = {"ms_per_step": ems / e2e_steps,
                             "h2d_effective_gbs": round(h2d / (ems / e2e_steps / 1e3) / 1e9, 1)}
            host_ms.clear()
            if world > 1:
                dist.barrier()
            ems = timed_e2e()
        # and right after it: the link is shared with the host's other traffic
        torch.cuda.synchronize()
        p0.record(stream)
        Xbuf[0].copy_(X_host, non_blocking=True)
        p1.record(stream)
        torch.cuda.synchronize()
        h2d_probe_after_gbs = X_host.numel() * 4 / (p0.elapsed_time(p1) / 1e3) / 1e9
        e2e = {"value": world * 2.0 * N_POINTS * K * e2e_steps / (ems / 1e3), "unit": "distances/s",
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "steps": e2e_steps,
               "host_enqueue_ms_per_step": round(statistics.mean(host_ms), 3),
               "h2d_probe_gbs": round(h2d_probe_gbs, 1), "h2d_probe_after_gbs": round(h2d_probe_after_gbs, 1),
               "h2d_effective_gbs": round(h2d / (ems / e2e_steps / 1e3) / 1e9, 1),
               "remeasured_after": first_attempt,
               "ms_per_step": ems / e2e_steps,
               "path": f"pinned host fp32 points -> H2D in {nchunk} row ranges on a copy stream (two device "
                       "buffers: the next step's points stream in during this step's tail), each range assigned "
                       "(fp32) and encoded + assigned (1-bit) once it has landed -> skm_update (fp32, 1-bit) -> "
                       "D2H assignments + centroids, which the next step copies back as its centroids"}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        h = {k2: v.cpu().numpy() for k2, v in q.items()}
        codes = h["codes"].view(np.uint32)
        X_host_np = X[:200_000].cpu().numpy()
        v, ns, t, cores = cpu_baseline_sample(X_host_np, C32.cpu().numpy(), codes, h["nx2"], h["F"], h["popx"],
                                              h["m"], e, Cr.cpu().numpy())
        cpu = {"value": v, "unit": "distances/s", "cores": cores, "kind": "oracle",
               "sample": f"{ns} of {N_POINTS} rows, one Lloyd iteration (assign + update) of fp32 and 1-bit "
                         f"against all {K} centroids, {t:.1f} s"}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "distances/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32 (bf16 tensor screen + fp32 rescore) / 1-bit (e4m3 tensor, exact)",
            "data": "synthetic (seeded GMM embeddings, generated on the GPU)",
            "config": {"workload": WORKLOAD, "n": N_POINTS, "d": DIM, "k": K, "reprs": ["f32", "rbq1"],
                       "step": "one Lloyd iteration (assign + update) per representation",
                       "l2": "inputs larger than L2 (3.1 GB fp32 points streamed every step)",
                       "timing": ("replays of one CUDA graph capturing the whole step" if graph is not None
                                  else "eager steps") + (f" ({graph_note})" if graph_note else ""),
                       "parallelism": f"dp{world}"},
            "roofline": roofline, "kernels": kernels, "cpu_baseline": cpu, "e2e": e2e, "clocks": clk,
            "gpu_launches": int(launches),
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def run_reference(args):
    """CPU oracle as it stands, on the host cores, on a bounded sample."""
    import numpy as np

    rank, _, world = env_rank()
    if rank != 0:
        return
    import oracle
    import synth

    ns = 4000
    X = synth.gmm_points(ns, DIM, N_COMP, seed=0).numpy()
    idx = synth.forgy_indices(ns, K, seed=0).numpy()
    C32 = X[idx].copy()
    m = oracle.rbq1_mean(X)
    codes, nx2, F, popx = oracle.rbq1_encode(X, m)
    e = oracle.rbq1_exponent(F)
    Cr = oracle.rbq1_decode_points(codes, F, DIM, m, e, idx)

    def step(rows):
        nonlocal C32, Cr
        a, _, _ = oracle.assign_f32(X[:rows], C32)
        C32, _ = oracle.update_f32(X[:rows], a, C32)
        prep = oracle.rbq1_centroid_sq4(Cr, m)
        ar, _ = oracle.rbq1_assign(codes[:rows], nx2[:rows], F[:rows], popx[:rows], DIM, prep)
        Cr, _ = oracle.rbq1_update(codes[:rows], F[:rows], DIM, m, e, ar, Cr)

    t0 = time.perf_counter()
    step(500)
    t1 = time.perf_counter() - t0
    budget = 150.0 / max(1, args.steps + args.warmup)
    rows = int(min(ns, max(500, 500 * budget / max(t1, 1e-3))))
    for _ in range(args.warmup):
        step(rows)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step(rows)
    t = time.perf_counter() - t0
    value = 2.0 * rows * K * args.steps / t
    sample = f"{rows} rows of the {WORKLOAD} recipe, one Lloyd iteration per representation per step"
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "distances/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * t / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64 (oracle)",
            "data": "synthetic (seeded GMM embeddings)",
            "config": {"workload": WORKLOAD, "n": N_POINTS, "d": DIM, "k": K, "reprs": ["f32", "rbq1"],
                       "parallelism": "host cores"},
            "cpu_baseline": {"value": value, "unit": "distances/s", "kind": "oracle", "cores": oracle.num_threads(),
                             "sample": sample},
            "e2e": {"value": value, "unit": "distances/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def run_case(args):
    """Small single-operation runs for profiler captures (ncu): `reps` calls
    of one entry point on a synthetic workload of the given size."""
    import torch

    import paper_2608_14648_gb300 as skm
    import synth

    torch.cuda.set_device(0)
    n, d, k = args.n, args.d, args.k
    X = synth.gmm_points(n, d, max(2 * k, 16), seed=0, device="cuda")
    if args.case == "project":  # Y = X P on tensor cores (k = output dimensions)
        P = synth.haar_rotation(d, 1)[:, :k].to(torch.float32).contiguous().cuda()
        skm.skm_project(X, P)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(args.reps):
            skm.skm_project(X, P)
        e1.record()
        torch.cuda.synchronize()
        print(json.dumps({"case": "project", "n": n, "d": d, "d_out": k, "reps": args.reps,
                          "ms_per_call": e0.elapsed_time(e1) / args.reps}))
        return
    if args.case.startswith("quantize_"):  # skm_quantize: statistics pass + encode, and encode alone
        repr_ = {"quantize_sq8": skm.REPR_SQ8, "quantize_rbq1": skm.REPR_RBQ1,
                 "quantize_lvq4": skm.REPR_LVQ4}[args.case]
        ws = skm.workspace(skm.OP_QUANTIZE, skm.Points(skm.REPR_F32, X, d), 1)
        q = skm.skm_quantize(repr_, X, ws=ws)
        extra = {k_: q[k_] for k_ in ("b", "s", "m") if k_ in q}
        out_t = {k_: v for k_, v in q.items() if k_ not in ("b", "s", "m")}
        code_bytes = sum(v.numel() * v.element_size() for v in out_t.values())
        ms = {}
        for fit in ((False,) if repr_ == skm.REPR_LVQ4 else (True, False)):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            torch.cuda.synchronize()
            e0.record()
            for _ in range(args.reps):
                skm.skm_quantize(repr_, X, fit=fit, out=out_t, ws=ws, **extra)
            e1.record()
            torch.cuda.synchronize()
            ms["fit" if fit else "encode"] = e0.elapsed_time(e1) / args.reps
        enc_bytes = 4 * n * d + code_bytes  # read the points once, write codes and factors
        print(json.dumps({"case": args.case, "n": n, "d": d, "reps": args.reps, "ms_per_call": ms,
                          "encode_bytes": enc_bytes, "encode_gbs": enc_bytes / (ms["encode"] * 1e6)}))
        return
    C = X[synth.forgy_indices(n, k, seed=0).cuda()].clone()
    if args.case in ("assign_f32", "update_f32"):
        pts = skm.Points(skm.REPR_F32, X, d).with_screen()
    elif args.case in ("assign_rbq1", "update_rbq1", "assign_rbq1_popcount"):
        pts = skm.rbq1_points(skm.skm_quantize(skm.REPR_RBQ1, X), d)
        if args.case == "assign_rbq1":
            pts = pts.with_screen()
    elif args.case in ("assign_lvq4", "update_lvq4"):
        pts = skm.lvq4_points(skm.skm_quantize(skm.REPR_LVQ4, X), d)
        if args.case == "assign_lvq4":
            pts = pts.with_screen()
    elif args.case in ("assign_sq8", "update_sq8"):
        q = skm.skm_quantize(skm.REPR_SQ8, X)
        pts = skm.Points(skm.REPR_SQ8, q["codes"], d).with_screen()
        C = q["codes"][:k].clone()
    elif args.case == "assign_prune_sq8":  # SQ8 codes, exact integer prefix-block pruning
        q = skm.skm_quantize(skm.REPR_SQ8, X)
        pts = skm.Points(skm.REPR_SQ8, q["codes"], d, flags=skm.FLAG_PRUNE)
        C = q["codes"][synth.forgy_indices(n, k, seed=0).cuda()].clone()
    elif args.case == "assign_prune":  # bf16 points, exact prefix-block pruning
        Xb = X.to(torch.bfloat16).view(torch.int16).contiguous()
        pts = skm.Points(skm.REPR_BF16, Xb, d, flags=skm.FLAG_PRUNE)
        C = (Xb[synth.forgy_indices(n, k, seed=0).cuda()].to(torch.int32) << 16).view(torch.float32).contiguous()
    else:
        raise SystemExit(f"unknown case {args.case}")
    wsA = skm.workspace(skm.OP_ASSIGN, pts, k)
    wsU = skm.workspace(skm.OP_UPDATE, pts, k)
    a = torch.empty(n, dtype=torch.int32, device="cuda")
    cnt = torch.zeros(k, dtype=torch.int64, device="cuda")
    skm.skm_assign(pts, C, k, want_dist=False, ws=wsA, out=a)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(args.reps):
        if args.case == "assign_rbq1_popcount":
            skm.skm_assign_rbq1_noalloc(pts, C, a)
        elif args.case.startswith("assign"):
            skm.skm_assign(pts, C, k, want_dist=False, ws=wsA, out=a)
        else:
            skm.skm_update(pts, a, C.clone(), counts=cnt, ws=wsU)
    e1.record()
    torch.cuda.synchronize()
    out = {"case": args.case, "n": n, "d": d, "k": k, "reps": args.reps,
           "ms_per_call": e0.elapsed_time(e1) / args.reps}
    if args.case == "assign_f32":  # how often the screen alone decides a row
        _, _, _, _, stats = skm.skm_fit(pts, k, 0, C_init=C, want_objective=False, want_dist=False)
        out["screen_stats"] = stats
    print(json.dumps(out))


def _run_hier(args, name, n, k, idx, runs):
    """Flat Lloyd (skm_fit, `iters` iterations + final assignment) against
    hierarchical k-means (m = round(sqrt k) meso clusters, `iters` meso and
    `iters` fine iterations + final assignments), whole calls timed with CUDA
    events after one warm-up call each."""
    import math

    import torch

    import paper_2608_14648_gb300 as skm

    m = max(1, round(math.sqrt(k)))
    midx = idx[:m].contiguous()
    for label, pts, C, d, peak, kind in runs:
        if label not in ("fp32", "sq8", "rbq1"):
            continue
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
        ws = skm.workspace(skm.OP_FIT, pts, k)
        skm.skm_fit(pts, k, args.iters, init_idx=idx, want_objective=False, want_dist=False, ws=ws)
        ev[0].record()
        skm.skm_fit(pts, k, args.iters, init_idx=idx, want_objective=False, want_dist=False, ws=ws)
        ev[1].record()
        torch.cuda.synchronize()
        del ws
        skm.skm_fit_hierarchical(pts, k, m, midx, args.iters, args.iters)
        ev[2].record()
        _, _, _, kf, _ = skm.skm_fit_hierarchical(pts, k, m, midx, args.iters, args.iters)
        ev[3].record()
        torch.cuda.synchronize()
        t_flat = ev[0].elapsed_time(ev[1])
        t_h = ev[2].elapsed_time(ev[3])
        out = {"config": args.config, "workload": name, "repr": label, "n": n, "d": d, "k": k, "m": m,
               "iters": args.iters, "flat_fit_ms": round(t_flat, 3), "hierarchical_fit_ms": round(t_h, 3),
               "speedup": round(t_flat / t_h, 2), "fine_counts_min_max": [min(kf), max(kf)]}
        print(json.dumps(out), flush=True)
        torch.cuda.empty_cache()


def _timed_projection(args, name, X, P, mean, out_dtype, peaks):
    """skm_project on the tensor cores (timed with CUDA events, after one
    warm-up call) and once on CUDA cores for comparison; returns Y."""
    import torch

    import paper_2608_14648_gb300 as skm

    n, d = X.shape
    dout = P.shape[1]
    Y = skm.skm_project(X, P, mean, out_dtype=out_dtype)
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
    ev[0].record()
    Y = skm.skm_project(X, P, mean, out_dtype=out_dtype)
    ev[1].record()
    torch.cuda.synchronize()
    t_tc = ev[0].elapsed_time(ev[1])
    ev[2].record()
    skm.skm_project(X, P, mean, out_dtype=out_dtype, cuda_cores=True)
    ev[3].record()
    torch.cuda.synchronize()
    t_cc = ev[2].elapsed_time(ev[3])
    work = 6 * 2.0 * n * d * dout  # bf16 tensor flop: six part products
    print(json.dumps({"config": args.config, "workload": name, "projection": f"{n} x {d} -> {dout}",
                      "tensor_ms": round(t_tc, 3), "cuda_core_ms": round(t_cc, 3),
                      "tensor_tflops": round(work / (t_tc / 1e3) / 1e12, 1),
                      "frac_of_bf16_peak": round(work / (t_tc / 1e3) / 1e12 / peaks["bf16_tflops"], 4),
                      "note": "includes the bf16 split pass (HBM) and the six-product GEMM"}), flush=True)
    return Y


def _quality(args, name, X, idx, k, runs, sq8_q):
    """Clustering quality in full precision: every representation's fit (the
    configured iterations from the same Forgy indices) evaluated on the raw
    fp32 points -- WCSS = sum ||x - c_a||^2 with SQ8 centroids decoded -- next
    to the fp32 fit's."""
    import paper_2608_14648_gb300 as skm

    d = X.shape[1]
    p32 = skm.Points(skm.REPR_F32, X, d)
    C32, a32, _, _, _ = skm.skm_fit(p32, k, args.iters, init_idx=idx, want_objective=False, want_dist=False)
    w32 = skm.skm_objective(X, C32, a32)
    out = {"config": args.config, "workload": name, "quality": "full-precision WCSS after the fit",
           "iters": args.iters, "fp32_wcss": w32}
    for label, pts, _, _, _, _ in runs:
        if label in ("fp32",) or label.endswith("_prune") or label.endswith("_symmetric"):
            continue
        C, a, _, _, _ = skm.skm_fit(pts, k, args.iters, init_idx=idx, want_objective=False, want_dist=False)
        if label == "sq8":
            C = skm.skm_sq8_decode(C, sq8_q["b"], sq8_q["s"])
        w = skm.skm_objective(X, C, a)
        out[f"{label}_wcss"] = w
        out[f"{label}_vs_fp32"] = round(w / w32, 6)
        if label == "rbq1" and args.iters > 0:
            # Section 4 ("Closing RabitQ's Gap in Balance"): the last update from
            # the raw vectors with the quantized run's assignment, then a final
            # quantized assignment
            C, a, _, _, _ = skm.skm_fit(pts, k, args.iters - 1, init_idx=idx, want_objective=False,
                                        want_dist=False)
            C, _ = skm.skm_update(p32, a, C)
            a, _ = skm.skm_assign(pts, C, want_dist=False)
            w = skm.skm_objective(X, C, a)
            out["rbq1_raw_last_update_wcss"] = w
            out["rbq1_raw_last_update_vs_fp32"] = round(w / w32, 6)
    print(json.dumps(out), flush=True)


def run_config(args):
    """One JSON line per representation of a workload configuration: the
    median over Lloyd iterations 2..iters of (centroid prep + assign + update)
    timed with CUDA events, distances/s = n k / t_iter, and the assignment
    against its roofline (2 n k d flop on the bf16 / e4m3 tensor peak)."""
    import numpy as np
    import torch

    import paper_2608_14648_gb300 as skm
    import synth

    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    peaks = load_peaks()
    iters = args.iters
    name = {"c0": "tiny_f32", "c1": "emb1m_d768", "c2": "emb1m_d1024_sq8", "c3": "emb10m_d1024_rbq1",
            "c4": "emb10m_pca256"}[args.config]
    spec = synth.WORKLOADS[name]
    n, k = spec.n, spec.k
    idx = synth.forgy_indices(n, k, seed=0).to(dev)
    X = synth.workload_points(spec, seed=0, device=dev)
    runs = []  # (label, Points, C0, d, peak TFLOP/s, flop kind)
    bf16_peak = peaks["bf16_tflops"]
    if args.config in ("c0", "c1"):
        runs.append(("fp32", skm.Points(skm.REPR_F32, X, spec.d).with_screen(), X[idx].clone(), spec.d,
                     bf16_peak, "bf16"))
    if args.config == "c1":
        q = skm.skm_quantize(skm.REPR_RBQ1, X)
        pR = skm.rbq1_points(q, spec.d).with_screen()
        CR, _, _, _, _ = skm.skm_fit(pR, k, 0, init_idx=idx, want_objective=False, want_dist=False)
        runs.append(("rbq1", pR, CR, spec.d, 2 * bf16_peak, "e4m3"))
        if args.symmetric:
            runs.append(("rbq1_symmetric", pR.with_flags(skm.FLAG_SYMMETRIC), CR.clone(), spec.d, 2 * bf16_peak,
                         "e4m3"))
    if args.config in ("c1", "c2"):
        pL = skm.lvq4_points(skm.skm_quantize(skm.REPR_LVQ4, X), spec.d).with_screen()
        CL, _, _, _, _ = skm.skm_fit(pL, k, 0, init_idx=idx, want_objective=False, want_dist=False)
        runs.append(("lvq4", pL, CL, spec.d, 2 * bf16_peak, "e4m3"))
    sq8_q = None
    if args.config == "c2":
        q = skm.skm_quantize(skm.REPR_SQ8, X)
        sq8_q = q
        runs.append(("sq8", skm.Points(skm.REPR_SQ8, q["codes"], spec.d).with_screen(),
                     q["codes"][idx].clone(), spec.d, bf16_peak, "bf16"))
        if args.prune:
            runs.append(("sq8_prune", skm.Points(skm.REPR_SQ8, q["codes"], spec.d, flags=skm.FLAG_PRUNE),
                         q["codes"][idx].clone(), spec.d, None, "int32 CUDA cores"))
    if args.config == "c3":
        P = synth.haar_rotation(spec.d, 99).to(torch.float32).contiguous().to(dev)
        Y = _timed_projection(args, name, X, P, None, skm.DTYPE_F32, peaks)
        del X
        q = skm.skm_quantize(skm.REPR_RBQ1, Y)
        if args.lvq4:
            pL = skm.lvq4_points(skm.skm_quantize(skm.REPR_LVQ4, Y), spec.d).with_screen()
            CL, _, _, _, _ = skm.skm_fit(pL, k, 0, init_idx=idx, want_objective=False, want_dist=False)
            runs.append(("lvq4", pL, CL, spec.d, 2 * bf16_peak, "e4m3"))
        del Y
        pR = skm.rbq1_points(q, spec.d).with_screen()
        CR, _, _, _, _ = skm.skm_fit(pR, k, 0, init_idx=idx, want_objective=False, want_dist=False)
        runs.append(("rbq1", pR, CR, spec.d, 2 * bf16_peak, "e4m3"))
    if args.config == "c4":
        dp = 256
        mean, P, _ = skm.skm_pca_fit(X, dp)
        Yb = _timed_projection(args, name, X, P, mean, skm.DTYPE_BF16, peaks).view(torch.int16)
        del X
        Cb = (Yb[idx].to(torch.int32) << 16).view(torch.float32).contiguous()
        runs.append(("bf16_screen", skm.Points(skm.REPR_BF16, Yb, dp).with_screen(), Cb, dp, bf16_peak, "bf16"))
        runs.append(("bf16_prune", skm.Points(skm.REPR_BF16, Yb, dp, flags=skm.FLAG_PRUNE), Cb.clone(), dp,
                     None, "fp32 CUDA cores"))
    torch.cuda.synchronize()
    if args.hier:
        _run_hier(args, name, n, k, idx, runs)
        return
    if args.config in ("c1", "c2"):
        _quality(args, name, X, idx, k, runs, sq8_q)
    for label, pts, C, d, peak, kind in runs:
        C = C.clone()
        wsA = skm.workspace(skm.OP_ASSIGN, pts, k)
        wsU = skm.workspace(skm.OP_UPDATE, pts, k)
        a = torch.empty(n, dtype=torch.int32, device=dev)
        prev = None
        cnt = torch.zeros(k, dtype=torch.int64, device=dev)
        stream = torch.cuda.current_stream()
        ta, tu = [], []
        for it in range(iters):
            e0, e1, e2 = (torch.cuda.Event(enable_timing=True) for _ in range(3))
            e0.record(stream)
            skm.skm_assign(pts, C, k, prev_assign=prev, want_dist=False, ws=wsA, out=a)
            e1.record(stream)
            skm.skm_update(pts, a, C, counts=cnt, ws=wsU)
            e2.record(stream)
            torch.cuda.synchronize()
            ta.append(e0.elapsed_time(e1))
            tu.append(e1.elapsed_time(e2))
            if label.endswith("_prune"):
                prev = a.clone()
        sel = slice(1, None) if iters > 1 else slice(0, None)
        t_a = float(np.median(ta[sel]))
        t_u = float(np.median(tu[sel]))
        t_it = float(np.median([x + y for x, y in zip(ta[sel], tu[sel])]))
        # the same iteration captured once in a CUDA graph and replayed (no
        # host launch overhead between the kernels: what small problems need)
        t_graph, graph_note = None, None
        try:
            prev_buf = a.clone() if label.endswith("_prune") else None
            side = torch.cuda.Stream()
            side.wait_stream(stream)
            with torch.cuda.stream(side):
                skm.skm_assign(pts, C, k, prev_assign=prev_buf, want_dist=False, ws=wsA, out=a)
                skm.skm_update(pts, a, C, counts=cnt, ws=wsU)
            stream.wait_stream(side)
            torch.cuda.synchronize()
            graph = torch.cuda.CUDAGraph()
            with torch.cuda.graph(graph):
                skm.skm_assign(pts, C, k, prev_assign=prev_buf, want_dist=False, ws=wsA, out=a)
                if prev_buf is not None:
                    prev_buf.copy_(a)
                skm.skm_update(pts, a, C, counts=cnt, ws=wsU)
            tg = []
            for _ in range(max(iters, 2)):
                g0, g1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                g0.record(stream)
                graph.replay()
                g1.record(stream)
                torch.cuda.synchronize()
                tg.append(g0.elapsed_time(g1))
            t_graph = float(np.median(tg[1:]))
            del graph
        except Exception as exc:  # report instead of failing the run
            graph_note = f"graph capture failed: {exc!r}"[:200]
        out = {"config": args.config, "workload": name, "repr": label, "n": n, "d": d, "k": k,
               "iters": iters, "ms_per_iter": round(t_it, 4), "assign_ms": round(t_a, 4),
               "update_ms": round(t_u, 4), "distances_per_s": n * k / (t_it / 1e3)}
        if t_graph is not None:
            out["ms_per_iter_graph"] = round(t_graph, 4)
            out["distances_per_s_graph"] = n * k / (t_graph / 1e3)
        if graph_note:
            out["graph_note"] = graph_note
        if peak:
            ach = 2.0 * n * k * d / (t_a / 1e3) / 1e12
            out["assign_roofline"] = {"bound": "tensor", "achieved_tflops": round(ach, 2),
                                      "peak_tflops": peak, "frac": round(ach / peak, 4), "flop": kind}
        if label.endswith("_prune"):
            _, _, _, _, st = skm.skm_fit(pts, k, 1, C_init=C, want_objective=False, want_dist=False)
            out["prune_stats_2_assigns"] = st
            out["dense_equiv_tensor_ms"] = round(2.0 * n * k * d / (bf16_peak * 1e12) * 1e3, 3)
        print(json.dumps(out), flush=True)
        del wsA, wsU
        torch.cuda.empty_cache()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-popcount", action="store_true")
    ap.add_argument("--eager", action="store_true", help="time eager steps instead of CUDA-graph replays")
    ap.add_argument("--case", default=None,
                    help="single-operation run for profiling: assign_f32|assign_rbq1|assign_sq8|assign_lvq4|"
                         "assign_rbq1_popcount|assign_prune|assign_prune_sq8|update_f32|update_rbq1|update_sq8|"
                         "update_lvq4|project|quantize_sq8|quantize_rbq1|quantize_lvq4")
    ap.add_argument("--n", type=int, default=200_000)
    ap.add_argument("--d", type=int, default=768)
    ap.add_argument("--k", type=int, default=1000)
    ap.add_argument("--reps", type=int, default=3)
    ap.add_argument("--config", default=None, choices=["c0", "c1", "c2", "c3", "c4"],
                    help="per-configuration Lloyd iteration timing (median of iterations 2..iters)")
    ap.add_argument("--iters", type=int, default=10)
    ap.add_argument("--lvq4", action="store_true", help="with --config c3: also time LVQ4 on the rotated points")
    ap.add_argument("--prune", action="store_true", help="with --config c2: also time SQ8 with exact pruning")
    ap.add_argument("--symmetric", action="store_true",
                    help="with --config c1: also time the symmetric 1-bit assignment (binarized centroids)")
    ap.add_argument("--hier", action="store_true",
                    help="with --config: flat Lloyd fit against hierarchical k-means (m = sqrt k)")
    args = ap.parse_args()
    if args.case:
        run_case(args)
        return
    if args.config:
        run_config(args)
        return
    if args.warmup < 3:
        print("warning: fewer than 3 warm-up steps", file=sys.stderr)
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
