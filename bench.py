#!/usr/bin/env python
"""Benchmark of the Lloyd k-means hot path on GB300.

Headline workload (emb10m_pca256): 10,000,000 unit-norm synthetic embeddings,
D = 1024 (10,000-component Gaussian mixture, per-dimension variance
(1+j)^-0.5, Haar rotation, L2 normalisation), PCA-projected to d' = 256 (fp32
projection, bf16 storage), k = 10,000.  One step = one Lloyd iteration (STEP 2
assignment + STEP 3 update) over all points, i.e. N * k point-centroid
distances.  Metric: point-centroid distances per second per Lloyd iteration.
Beside it the line reports the 1M x 768 (fp32 and 1-bit) and 10M x 1024
(1-bit, k = 3,162) iterations, the pruned assignment of the headline
workload, and the end-to-end step from pinned host memory.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

N > 1 runs under torchrun, one rank per GPU: every rank clusters its own
10M-point shard (weak scaling); the PCA basis and the initial centroids come
from rank 0, and the update's cluster sums and counts are all-reduced once per
step (the path's one exchange).  --impl reference times the CPU oracle on a
bounded sample of the headline workload.
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

HEAD = "emb10m_pca256"
D_PCA = 256
METRIC = "k-means point·centroid distances/s per Lloyd iter (1 GB300); % of roofline"
WORKLOAD = ("emb10m_pca256: N=10,000,000 unit-norm GMM embeddings, D=1024 -> PCA d'=256 (fp32 projection, "
            "bf16 storage), k=10,000")
SM_COUNT = 152
# dense-screen Lloyd iterations run as setup before the timed (pruned) steps
DENSE_SETUP = 4
# row ranges of the end-to-end step's host-to-device copy (overlapped with work)
E2E_CHUNKS = 8
# POPC results per clock per SM used for the 1-bit kernel's ALU roofline
# (measured 15.9 on GB300 with a throughput probe).
POPC_PER_CLK_SM = 16
# DRAM bytes (read + write) per point of the assignment kernels, each from
# one ncu capture of a smaller case of the same kernel (every point row is
# read once per launch, so traffic scales with the points): the bf16 screen
# at 400,000 x 256 with k = 10,000; the tensor-core pruning front at
# 1,000,000 x 256 with k = 10,000 (the headline recipe at that size); the fp32
# screen and the 1-bit kernel (packed codes, tiles expanded in an
# L2-resident scratch) at 200,000 x 768 with k = 1,000.
TRAFFIC_PER_POINT = {
    "assign_bf16_prune_front": (390.669312e6 + 38.499072e6) / 1_000_000,
    "assign_bf16_screen": (213.449216e6 + 4.711680e6) / 400_000,
    "assign_f32": (314.849280e6 + 5.701888e6) / 200_000,
    "assign_rbq1": (22.462464e6 + 23.388416e6) / 200_000,
}


def prune_roofline(pairs, later_blocks, nb, ms, peaks):
    """Executed-work roofline of a pruned assignment: every (point, centroid)
    pair's first 32-dimension block plus the later blocks the bounds did not
    skip, each 32 fp32 subtractions and 32 fmas on the CUDA cores, against
    SM_COUNT SMs x 128 fp32 lanes at the maximum SM clock."""
    blocks = pairs + float(later_blocks)
    achieved = blocks * 64.0 / (ms / 1e3) / 1e12
    peak = SM_COUNT * 128 * peaks["sm_max_mhz"] * 1e6 / 1e12
    return {"bound": "alu", "unit": "T fp32 lane-instructions/s", "executed_blocks": blocks,
            "executed_fraction_of_dense": blocks / (pairs * nb), "achieved": achieved, "peak": peak,
            "frac": achieved / peak}


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
def _graph_of(step, stream):
    """Captures step() once in a CUDA graph (after one run on a side stream);
    returns (graph, library launches per step) or (None, note)."""
    import torch

    import paper_2608_14648_gb300 as skm

    try:
        side = torch.cuda.Stream()
        side.wait_stream(stream)
        with torch.cuda.stream(side):
            step()
        stream.wait_stream(side)
        torch.cuda.synchronize()
        l0 = skm.skm_kernel_launches()
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            step()
        launches = skm.skm_kernel_launches() - l0
        graph.replay()
        torch.cuda.synchronize()
        return graph, launches
    except Exception as exc:  # eager steps instead, reported
        return None, f"graph capture failed, eager steps: {exc!r}"[:200]


def _timed_steps(step, stream, steps, warmup, world, dist, local_rank, use_graph):
    """warmup eager steps, then `steps` steps (CUDA-graph replays on one GPU)
    bracketed by a barrier and synchronisation; returns (ms max over ranks,
    launches, timing note, clocks)."""
    import torch

    import paper_2608_14648_gb300 as skm

    for _ in range(warmup):
        step()
    torch.cuda.synchronize()
    graph, lps, note = None, None, None
    if use_graph:
        graph, lps = _graph_of(step, stream)
        if graph is None:
            note, lps = lps, None
    if world > 1:
        dist.barrier()
    clocks = ClockSampler(local_rank)
    clocks.start()
    torch.cuda.synchronize()
    l0 = skm.skm_kernel_launches()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for _ in range(steps):
        if graph is not None:
            graph.replay()
        else:
            step()
    t1.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clk = clocks.stop()
    ms = t0.elapsed_time(t1)
    if world > 1:
        t = torch.tensor([ms], device="cuda", dtype=torch.float64)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ms = float(t.item())
    launches = lps * steps if graph is not None else skm.skm_kernel_launches() - l0
    timing = ("replays of one CUDA graph capturing the whole step" if graph is not None else "eager steps") + \
        (f" ({note})" if note else "")
    return ms, int(launches), timing, clk


def _event_ms(fn, reps, stream):
    """Mean CUDA-event time of fn() over reps calls, each bracketed alone."""
    import torch

    ts = []
    for _ in range(reps):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        fn()
        e1.record(stream)
        torch.cuda.synchronize()
        ts.append(e0.elapsed_time(e1))
    return statistics.mean(ts)


def _kernel_ms(fn, reps):
    """Mean duration of the tensor-core kernel launched by fn() (the library's
    events around the launch, on its stream), over reps calls."""
    import paper_2608_14648_gb300 as skm

    skm.skm_kernel_timer(True)
    try:
        ts = []
        for _ in range(reps):
            fn()
            ts.append(skm.skm_kernel_timer_ms())
    finally:
        skm.skm_kernel_timer(False)
    return statistics.mean(ts)


def _split_ms(fns, reps, stream):
    """Mean CUDA-event time of each of fns over reps rounds of calling them in
    order (each bracketed alone)."""
    import torch

    ts = [[] for _ in fns]
    for _ in range(reps):
        for i, fn in enumerate(fns):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            fn()
            e1.record(stream)
            torch.cuda.synchronize()
            ts[i].append(e0.elapsed_time(e1))
    return [statistics.mean(t) for t in ts]


def cpu_baseline_c4(Yb_host, C_host, K, budget_s=15.0):
    """Oracle (as it stands) on a bounded row sample of the headline
    workload: one Lloyd iteration (assignment against all k centroids in fp64,
    update) of the first rows.  Returns (distances/s, rows, seconds, threads)."""
    import oracle

    def one(ns):
        t0 = time.perf_counter()
        a, _, _ = oracle.assign_bf16(Yb_host[:ns], C_host)
        oracle.update_bf16(Yb_host[:ns], a, C_host)
        return time.perf_counter() - t0

    one(200)  # thread pool start-up
    t0 = one(2000)
    ns = int(min(Yb_host.shape[0], max(2000, 2000 * budget_s / max(t0, 1e-3))))
    t = one(ns)
    return ns * K / t, ns, t, oracle.num_threads()


def setup_head(dev, rank, world, dist, peaks):
    """The headline workload resident in HBM: generated points, PCA basis
    (rank 0's, broadcast), bf16 projection, Forgy centroids (rank 0's)."""
    import torch

    import paper_2608_14648_gb300 as skm
    import synth

    spec = synth.WORKLOADS[HEAD]
    N, K = spec.n, spec.k
    X = synth.workload_points(spec, seed=rank, device=dev)
    mean = torch.empty(spec.d, device=dev, dtype=torch.float32)
    P = torch.empty(spec.d, D_PCA, device=dev, dtype=torch.float32)
    if rank == 0:
        mean, P, _ = skm.skm_pca_fit(X, D_PCA)
    if world > 1:
        dist.broadcast(mean, 0)
        dist.broadcast(P, 0)
    skm.skm_project(X[:1024], P, mean, out_dtype=skm.DTYPE_BF16, max_ws_bytes=8 << 30)  # first-use costs
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    Y = skm.skm_project(X, P, mean, out_dtype=skm.DTYPE_BF16, max_ws_bytes=8 << 30)
    e1.record()
    torch.cuda.synchronize()
    t_proj = e0.elapsed_time(e1)
    del X
    torch.cuda.empty_cache()
    Yb = Y.view(torch.int16)
    idx = synth.forgy_indices(N, K, seed=0).to(dev)
    C = (Yb[idx].to(torch.int32) << 16).view(torch.float32).contiguous()
    if world > 1:
        dist.broadcast(C, 0)
    flops = 6 * 2.0 * N * spec.d * D_PCA
    proj = {"ms": t_proj, "bound": "tensor", "achieved": flops / (t_proj / 1e3) / 1e12, "peak": peaks["bf16_tflops"],
            "unit": "TFLOP/s", "in_step": False,
            "algorithmic": f"6 bf16 part products x 2*N*D*d' = {flops:.3e} flop (fp32-accurate projection, "
                           "one-time preparation; includes the split pass)"}
    proj["frac"] = proj["achieved"] / proj["peak"]
    return Yb, C, idx, proj


def run_extra_configs(args, dev, peaks, stream, local_rank):
    """The 1M x 768 (fp32 and 1-bit) and 10M x 1024 (1-bit, k = 3,162)
    iterations, each timed like the headline (graph replays), with clocks."""
    import torch

    import paper_2608_14648_gb300 as skm
    import synth

    out = {}

    def timed(name, pts, C, k, n, d, flop_peak, kind, copy_pts=None):
        wsA = skm.workspace(skm.OP_ASSIGN, pts, k)
        wsU = skm.workspace(skm.OP_UPDATE, pts, k)
        a = torch.empty(n, dtype=torch.int32, device=dev)
        cnt = torch.zeros(k, dtype=torch.int64, device=dev)

        def step():
            skm.skm_assign(pts, C, k, want_dist=False, ws=wsA, out=a)
            skm.skm_update(pts, a, C, counts=cnt, ws=wsU)

        steps = max(5, min(args.steps, 20))
        ms, launches, timing, clk = _timed_steps(step, stream, steps, 3, 1, None, local_rank, not args.eager)
        t_a, t_u = _split_ms([lambda: skm.skm_assign(pts, C, k, want_dist=False, ws=wsA, out=a),
                              lambda: skm.skm_update(pts, a, C, counts=cnt, ws=wsU)], 3, stream)
        flops = 2.0 * n * k * d
        ach = flops / (t_a / 1e3) / 1e12
        out[name] = {"n": n, "d": d, "k": k, "ms_per_iter": ms / steps, "distances_per_s": n * k * steps / (ms / 1e3),
                     "assign_ms": t_a, "update_ms": t_u, "assign_achieved_tflops": ach, "assign_peak_tflops": flop_peak,
                     "assign_frac": ach / flop_peak, "flop": kind, "steps": steps, "timing": timing, "clocks": clk,
                     "gpu_launches": launches}
        if copy_pts is not None:  # 1-bit: the points stay packed; the e4m3 copy for comparison
            wsC = skm.workspace(skm.OP_ASSIGN, copy_pts, k)
            t_c = _event_ms(lambda: skm.skm_assign(copy_pts, C, k, want_dist=False, ws=wsC, out=a), 3, stream)
            out[name]["points_in_hbm"] = f"packed 1-bit codes, {4 * ((d + 31) // 32)} B a point"
            out[name]["assign_ms_from_e4m3_copy"] = t_c
            out[name]["e4m3_copy_bytes"] = n * (d + 15) // 16 * 16
            del wsC
        del wsA, wsU

    bf16 = peaks["bf16_tflops"]
    spec = synth.WORKLOADS["emb1m_d768"]
    X = synth.workload_points(spec, seed=0, device=dev)
    idx = synth.forgy_indices(spec.n, spec.k, seed=0).to(dev)
    timed("emb1m_d768_f32", skm.Points(skm.REPR_F32, X, spec.d, flags=skm.FLAG_WARM).with_screen(), X[idx].clone(),
          spec.k, spec.n, spec.d, bf16, "bf16")
    pR = skm.rbq1_points(skm.skm_quantize(skm.REPR_RBQ1, X), spec.d)
    CR, _, _, _, _ = skm.skm_fit(pR, spec.k, 0, init_idx=idx, want_objective=False, want_dist=False)
    timed("emb1m_d768_rbq1", pR, CR, spec.k, spec.n, spec.d, 2 * bf16, "e4m3", copy_pts=pR.with_screen())
    # the AND + popcount 1-bit kernel on the same codes (no allocation entry point)
    a_pop = torch.empty(spec.n, dtype=torch.int32, device=dev)
    skm.skm_assign_rbq1_noalloc(pR, CR, a_pop)
    t_pop = _event_ms(lambda: skm.skm_assign_rbq1_noalloc(pR, CR, a_pop), 2, stream)
    popc = float(spec.n) * spec.k * 4 * ((spec.d + 31) // 32)
    popc_peak = SM_COUNT * POPC_PER_CLK_SM * peaks["sm_max_mhz"] * 1e6
    out["emb1m_d768_rbq1_popcount"] = {"assign_ms": t_pop, "bound": "alu", "achieved_tpopc": popc / (t_pop / 1e3) / 1e12,
                                       "peak_tpopc": popc_peak / 1e12, "frac": popc / (t_pop / 1e3) / popc_peak,
                                       "algorithmic": f"N*k*4*ceil(d/32) = {popc:.3e} POPC per launch"}
    del X, pR, CR, a_pop
    torch.cuda.empty_cache()

    spec = synth.WORKLOADS["emb10m_d1024_rbq1"]
    X = synth.workload_points(spec, seed=0, device=dev)
    P = synth.haar_rotation(spec.d, 99).to(torch.float32).contiguous().to(dev)
    Y = skm.skm_project(X, P, max_ws_bytes=8 << 30)
    del X
    q = skm.skm_quantize(skm.REPR_RBQ1, Y)
    del Y
    torch.cuda.empty_cache()
    idx = synth.forgy_indices(spec.n, spec.k, seed=0).to(dev)
    pR = skm.rbq1_points(q, spec.d)
    CR, _, _, _, _ = skm.skm_fit(pR, spec.k, 0, init_idx=idx, want_objective=False, want_dist=False)
    timed("emb10m_d1024_rbq1", pR, CR, spec.k, spec.n, spec.d, 2 * bf16, "e4m3", copy_pts=pR.with_screen())
    del pR, CR, q
    torch.cuda.empty_cache()
    return out


def run_ours(args):
    import numpy as np
    import torch

    import paper_2608_14648_gb300 as skm

    rank, local_rank, world = env_rank()
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    dist = None
    if world > 1:
        import torch.distributed as dist

        dist.init_process_group("nccl")
    peaks = load_peaks()
    stream = torch.cuda.current_stream()

    # ---- inputs (per-rank shard), resident in HBM before timing -------------
    Yb, C, idx, proj = setup_head(dev, rank, world, dist, peaks)
    N, K = Yb.shape[0], C.shape[0]
    warm = 0 if args.cold_screen else skm.FLAG_WARM
    # the dense bf16 screen (per-point norms built once; FLAG_WARM: each screen
    # starts from the previous call's bounds): the first step's seeds, and the
    # comparison step (--dense)
    pts_d = skm.Points(skm.REPR_BF16, Yb, D_PCA, flags=warm).with_screen()
    wsD = skm.workspace(skm.OP_ASSIGN, pts_d, K)
    # the step's assignment: exact dimension pruning (Section 3.1
    # "SuperKMeans") with the first 128 dimensions on tensor cores, seeded with
    # the previous step's assignment; FLAG_WARM: each row's bound carried over
    pts_p = skm.Points(skm.REPR_BF16, Yb, D_PCA, flags=skm.FLAG_PRUNE | warm)
    pts = pts_d if args.dense else pts_p
    wsA = wsD if args.dense else skm.workspace(skm.OP_ASSIGN, pts_p, K)
    wsU = skm.workspace(skm.OP_UPDATE, pts_d, K)
    a = torch.empty(N, dtype=torch.int32, device=dev)
    cnt = torch.zeros(K, dtype=torch.int64, device=dev)
    part = torch.zeros(K, D_PCA, dtype=torch.float64, device=dev) if world > 1 else None
    C_step = C.clone()
    # setup (untimed): DENSE_SETUP Lloyd iterations with the dense screen from
    # the Forgy centroids.  Prefix pruning pays once the centroids have
    # settled (at the Forgy centroids the front keeps ~2,300 of 10,000
    # centroids a row; from about the sixth iteration ~1.3), which is also
    # when skm_fit switches to it; the timed steps are later iterations.
    for _ in range(DENSE_SETUP):
        skm.skm_assign(pts_d, C_step, K, want_dist=False, ws=wsD, out=a)
        if part is None:
            skm.skm_update(pts_d, a, C_step, counts=cnt, ws=wsU)
        else:
            part.zero_()
            cnt.zero_()
            skm.skm_update(pts_d, a, None, counts=cnt, partial=part, ws=wsU)
            dist.all_reduce(part)
            dist.all_reduce(cnt)
            skm.skm_update_finalize(pts_d, part, cnt, C_step)
    skm.skm_assign(pts_d, C_step, K, want_dist=False, ws=wsD, out=a)  # the first pruned step's seeds
    prev = None if args.dense else a

    def step():
        skm.skm_assign(pts, C_step, K, prev_assign=prev, want_dist=False, ws=wsA, out=a)
        if part is None:
            skm.skm_update(pts, a, C_step, counts=cnt, ws=wsU)
        else:  # the one exchange: cluster sums and counts, all-reduced
            part.zero_()
            cnt.zero_()
            skm.skm_update(pts, a, None, counts=cnt, partial=part, ws=wsU)
            dist.all_reduce(part)
            dist.all_reduce(cnt)
            skm.skm_update_finalize(pts, part, cnt, C_step)

    ms, launches, timing, clk = _timed_steps(step, stream, args.steps, args.warmup, world, dist, local_rank,
                                             world == 1 and not args.eager)
    ms_step = ms / args.steps
    value = world * float(N) * K * args.steps / (ms / 1e3)

    # ---- per-kernel times (eager calls after the timed region) ----------------
    # assignment and update each timed inside eager steps (every assignment
    # after an update, as in the timed region)
    t_assign, t_update = _split_ms([lambda: skm.skm_assign(pts, C_step, K, prev_assign=prev, want_dist=False,
                                                           ws=wsA, out=a),
                                    lambda: skm.skm_update(pts, a, C_step, counts=cnt, ws=wsU)], 3, stream)
    long_region = ms > 1000.0
    bf16_peak = peaks["bf16_tflops_sustained"] if long_region else peaks["bf16_tflops"]
    flops = 2.0 * N * K * D_PCA
    upd_bytes = N * D_PCA * 2 + N * 4 * 3  # rows read once; assignments, sorted order, cluster ids
    kernels = {}
    # the assignment's tensor-core kernel alone (events around its launch), in
    # further eager steps' assignments
    k_assign = _kernel_ms(lambda: skm.skm_assign(pts, C_step, K, prev_assign=prev, want_dist=False, ws=wsA, out=a),
                          3)
    if not args.dense:
        st = skm.skm_assign_prune_stats(wsA, stream)  # the last call's (a Lloyd step's)
        F = st["prune_front_dims"]
        fflops = 2.0 * N * K * F
        kernels["assign_bf16_prune_front"] = {
            "ms": k_assign, "call_ms": t_assign, "bound": "tensor", "achieved": fflops / (k_assign / 1e3) / 1e12,
            "peak": bf16_peak, "unit": "TFLOP/s",
            "call_achieved": fflops / (t_assign / 1e3) / 1e12,
            "algorithmic": f"2*N*k*F = {fflops:.3e} bf16 flop per launch (F = {F} front dimensions on tensor cores, "
                           "the measured executed work) over the front kernel's own duration; the call (call_ms) "
                           "also sorts the centroids, forms the rows' thresholds from their kept bounds and "
                           "finishes the survivors on CUDA cores",
            "front_dims": F, "survivors_per_row": st["prune_first_block"] / N,
            "rows_finished_cuda_cores": st["prune_rows_finished"], "rows_pruned_over_all_k": st["prune_rows_full"],
            "cuda_core_block_sums": st["prune_blocks"], "complete_pairs": st["prune_complete"],
            "dense_equivalent_tflops": flops / (t_assign / 1e3) / 1e12,
            "note": "exact: the same assignments and distances as the CUDA-core prefix pruning, bit for bit"}
        # the dense screen on the same centroids (warm from its own previous call)
        a_d = torch.empty_like(a)
        skm.skm_assign(pts_d, C_step, K, want_dist=False, ws=wsD, out=a_d)
        t_dense = _event_ms(lambda: skm.skm_assign(pts_d, C_step, K, want_dist=False, ws=wsD, out=a_d), 3, stream)
        k_dense = _kernel_ms(lambda: skm.skm_assign(pts_d, C_step, K, want_dist=False, ws=wsD, out=a_d), 3)
        kernels["assign_bf16_prune_front"]["agreement_with_dense_screen"] = float((a_d == a).float().mean())
        del a_d
    else:
        t_dense, k_dense = t_assign, k_assign
    kernels["assign_bf16_screen"] = {
        "ms": k_dense, "call_ms": t_dense, "bound": "tensor", "achieved": flops / (k_dense / 1e3) / 1e12,
        "peak": bf16_peak, "unit": "TFLOP/s", "in_step": bool(args.dense),
        "call_achieved": flops / (t_dense / 1e3) / 1e12,
        "algorithmic": f"2*N*k*d' = {flops:.3e} bf16 flop per launch (dense tensor-core screen) over the kernel's "
                       "own duration; the call (call_ms) also prepares the centroids and rescores undecided rows "
                       "in fp32"}
    kernels.update({
        "update_bf16": {
            "ms": t_update, "bound": "hbm", "achieved": upd_bytes / (t_update / 1e3) / 1e9, "peak": peaks["hbm_gbs"],
            "unit": "GB/s", "algorithmic": f"N*d'*2 + 12*N = {upd_bytes:.3e} bytes per launch (bf16 rows read once, "
                                           "assignments, sorted order and cluster ids)"},
        "project_pca": proj,
    })

    # ---- the pruned assignment of the same workload (exact, SKM_FLAG_PRUNE) on a row subset
    if not args.no_prune and world == 1:
        ns = min(N, 1_000_000)
        pp = skm.Points(skm.REPR_BF16, Yb[:ns], D_PCA, flags=skm.FLAG_PRUNE | skm.FLAG_PRUNE_CUDA_CORES)
        ap = torch.empty(ns, dtype=torch.int32, device=dev)
        prev = a[:ns].clone()  # bound seeded with the previous assignment's centroid
        wsP = skm.workspace(skm.OP_ASSIGN, pp, K)
        skm.skm_assign(pp, C_step, K, prev_assign=prev, want_dist=False, ws=wsP, out=ap)
        t_prune = _event_ms(lambda: skm.skm_assign(pp, C_step, K, prev_assign=prev, want_dist=False, ws=wsP,
                                                   out=ap), 2, stream)
        st = skm.skm_assign_prune_stats(wsP, stream)  # counters of the last timed call
        # the dense screen's assignment of the same rows for the same centroids
        a_ref, _ = skm.skm_assign(skm.Points(skm.REPR_BF16, Yb[:ns], D_PCA).with_screen(), C_step, K, want_dist=False)
        same = float((ap == a_ref).float().mean())
        pairs = float(ns) * K
        dense_ms = t_assign * ns / N
        kernels["assign_bf16_prune"] = {
            "ms": t_prune, "rows": ns, "in_step": False,
            "first_block_survivors": st["prune_first_block"] / pairs, "complete_survivors": st["prune_complete"] / pairs,
            "dense_screen_ms_same_rows": dense_ms, "speedup_vs_dense": dense_ms / t_prune,
            "agreement_with_dense": same,
            "note": "exact 32-dimension prefix-block pruning, bound seeded with the previous assignment",
            **prune_roofline(pairs, st["prune_blocks"], D_PCA // 32, t_prune, peaks)}
        del pp, ap, prev, wsP
    for kd in kernels.values():
        if "achieved" in kd:
            kd["frac"] = kd["achieved"] / kd["peak"]
    head_kernel = "assign_bf16_screen" if args.dense else "assign_bf16_prune_front"
    kd = kernels[head_kernel]
    traffic = TRAFFIC_PER_POINT.get(head_kernel)
    roofline = {"bound": kd["bound"], "achieved": round(kd["achieved"], 4), "peak": round(kd["peak"], 4),
                "unit": kd["unit"], "frac": round(kd["frac"], 5),
                "traffic": round(traffic * N) if traffic else None, "kernel": head_kernel,
                "peak_source": f"{peaks['source']} ({'sustained' if long_region else 'burst'} bf16)"}

    # ---- end to end through the C ABI with host buffers ----------------------
    e2e = None
    if not args.no_e2e:
        Y_host = torch.empty(N, D_PCA, dtype=torch.int16, pin_memory=True)
        Y_host.copy_(Yb)
        # the Lloyd run continues from the device steps' centroids and
        # assignments (the seeds of the first call; each call then leaves its
        # assignments there)
        C_host = torch.empty(K, D_PCA, dtype=torch.float32, pin_memory=True)
        C_host.copy_(C_step)
        a_host = torch.empty(N, dtype=torch.int32, pin_memory=True)
        a_host.copy_(a)
        holder = {}

        def exchange():
            s = holder["step"]
            dist.all_reduce(s.partial)
            dist.all_reduce(s.counts)

        prune_e2e = not (args.dense or args.cold_screen)
        hstep = skm.LloydStepHost(skm.REPR_BF16, Y_host, D_PCA, K, chunks=args.e2e_chunks, device=dev,
                                  exchange=exchange if world > 1 else None, warm=not args.cold_screen,
                                  prune=prune_e2e)
        holder["step"] = hstep
        for _ in range(2):  # untimed warm-up (first-use costs of the range-sized calls)
            hstep(C_host, C_host, a_host)
        e2e_steps = max(2, min(args.steps, 5))
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for _ in range(e2e_steps):
            hstep(C_host, C_host, a_host)  # synchronous: results are in host memory on return
        ems = (time.perf_counter() - t0) * 1e3
        if world > 1:
            t = torch.tensor([ems], device=dev, dtype=torch.float64)
            dist.all_reduce(t, op=dist.ReduceOp.MAX)
            ems = float(t.item())
        # the host link's copy rate right after (the step's bound when the work is shorter)
        p0, p1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        p0.record(stream)
        Yb.copy_(Y_host, non_blocking=True)
        p1.record(stream)
        torch.cuda.synchronize()
        h2d_probe_gbs = Y_host.numel() * 2 / (p0.elapsed_time(p1) / 1e3) / 1e9
        # points and centroids in; pruned, also the seeds (the previous assignments)
        h2d = Y_host.numel() * 2 + C_host.numel() * 4 + (a_host.numel() * 4 if prune_e2e else 0)
        d2h = a_host.numel() * 4 + C_host.numel() * 4
        e2e = {"value": world * float(N) * K * e2e_steps / (ems / 1e3), "unit": "distances/s",
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "steps": e2e_steps,
               "ms_per_step": ems / e2e_steps, "h2d_probe_gbs": round(h2d_probe_gbs, 1),
               "h2d_effective_gbs": round(h2d / (ems / e2e_steps / 1e3) / 1e9, 1),
               "path": f"skm_lloyd_step_host: pinned host bf16 points (and, pruned, the previous assignments as "
                       f"seeds) -> {args.e2e_chunks} row ranges copied on a copy stream into three device range buffers "
                       "while earlier ranges are assigned (each range from the bounds its previous call left) and "
                       "summed -> finalised centroids and assignments back in host memory on return (host wall "
                       "clock per call)"}
        del hstep, Y_host

    # ---- the other configurations (one GPU) -------------------------------------
    extra = None
    if world == 1 and not args.no_extra:
        del wsA, wsU, pts, pts_d, pts_p, wsD
        torch.cuda.empty_cache()
        extra = run_extra_configs(args, dev, peaks, stream, local_rank)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        Yh = Yb[:200_000].cpu().numpy().view(np.uint16)
        v, ns, t, cores = cpu_baseline_c4(Yh, C.cpu().numpy(), K)
        cpu = {"value": v, "unit": "distances/s", "cores": cores, "kind": "oracle",
               "sample": f"{ns} of {N} rows of the headline workload, one Lloyd iteration (fp64 assignment "
                         f"against all {K} centroids + update), {t:.1f} s"}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "distances/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None,
            "dtype": ("bf16 points, fp32 centroids (bf16 tensor-core screen + fp32 rescore: the exact fp32 argmin)"
                      if args.dense else
                      "bf16 points, fp32 centroids (exact prefix pruning: bf16 tensor-core front over 128 dims "
                      "with a rigorous bound, survivors finished in fp32 block sums: the exact fp32 argmin)"),
            "data": "synthetic (seeded GMM embeddings, generated on the GPU; PCA fitted on them)",
            "config": {"workload": WORKLOAD, "n": N, "D": 1024, "d": D_PCA, "k": K, "repr": "bf16 (PCA-256)",
                       "step": ("one Lloyd iteration (assign + update) over all points" + (
                           "" if args.dense else "; assignment: exact dimension pruning seeded with the previous "
                                                 "step's assignment, bounds carried between steps") +
                           f"; the Lloyd run starts from seeded Forgy centroids, {DENSE_SETUP} dense-screen "
                           f"iterations and the {args.warmup} warm-up steps precede the timed ones"),
                       "l2": "inputs larger than L2 (5.1 GB of bf16 points streamed every step)",
                       "timing": timing, "parallelism": f"dp{world}"},
            "roofline": roofline, "kernels": kernels, "configs": extra, "cpu_baseline": cpu, "e2e": e2e,
            "clocks": clk, "gpu_launches": launches,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def run_reference(args):
    """CPU oracle as it stands, on the host cores, on a bounded sample of the
    headline workload's recipe (PCA fitted on the sample)."""
    rank, _, world = env_rank()
    if rank != 0:
        return
    import oracle
    import synth

    spec = synth.WORKLOADS[HEAD]
    ns = 20_000
    X = synth.gmm_points(ns, spec.d, spec.n_comp, seed=0, decay=spec.decay, std=spec.std).numpy()
    mu, P, _ = oracle.pca_fit(X, D_PCA)
    Yb = oracle.round_bf16(oracle.project(X, P, mu))
    del X
    K = spec.k
    idx = synth.forgy_indices(ns, K, seed=0).numpy()
    C = oracle.bf16_to_f32(Yb[idx]).copy()

    def step(rows):
        nonlocal C
        a, _, _ = oracle.assign_bf16(Yb[:rows], C)
        C, _ = oracle.update_bf16(Yb[:rows], a, C)

    t0 = time.perf_counter()
    step(200)
    t1 = time.perf_counter() - t0
    budget = 150.0 / max(1, args.steps + args.warmup)
    rows = int(min(ns, max(200, 200 * budget / max(t1, 1e-3))))
    for _ in range(args.warmup):
        step(rows)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step(rows)
    t = time.perf_counter() - t0
    value = float(rows) * K * args.steps / t
    sample = (f"{rows} rows of the {HEAD} recipe (PCA fitted on a {ns}-row sample), one Lloyd iteration against "
              f"all {K} centroids per step")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "distances/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * t / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64 (oracle)",
            "data": "synthetic (seeded GMM embeddings)",
            "config": {"workload": WORKLOAD, "n": spec.n, "D": spec.d, "d": D_PCA, "k": K, "repr": "bf16 (PCA-256)",
                       "step": "one Lloyd iteration (assign + update) over the sampled points",
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
        if args.case == "assign_rbq1" and args.e4m3_copy:  # the e4m3 screening copy instead of packed codes
            pts = pts.with_screen()
    elif args.case == "assign_rbq1_skm":  # SuperKMeans checkpoints on RabitQ codes (CUDA cores)
        q = skm.skm_quantize(skm.REPR_RBQ1, X)
        pts = skm.rbq1_points(q, d).with_segments(skm.skm_rbq1_segments(X, q["m"])).with_flags(skm.FLAG_PRUNE)
    elif args.case in ("assign_lvq4", "update_lvq4"):
        pts = skm.lvq4_points(skm.skm_quantize(skm.REPR_LVQ4, X), d)
        if args.case == "assign_lvq4" and args.e4m3_copy:  # the e4m3 screening copy instead of packed codes
            pts = pts.with_screen()
    elif args.case in ("assign_sq8", "update_sq8"):
        q = skm.skm_quantize(skm.REPR_SQ8, X)
        pts = skm.Points(skm.REPR_SQ8, q["codes"], d).with_screen()
        C = q["codes"][:k].clone()
    elif args.case == "assign_prune_sq8":  # SQ8 codes, exact integer prefix-block pruning
        q = skm.skm_quantize(skm.REPR_SQ8, X)
        pts = skm.Points(skm.REPR_SQ8, q["codes"], d, flags=skm.FLAG_PRUNE)
        C = q["codes"][synth.forgy_indices(n, k, seed=0).cuda()].clone()
    elif args.case == "assign_bf16":  # bf16 points, tensor-core screen (the headline's kernel)
        Xb = X.to(torch.bfloat16).view(torch.int16).contiguous()
        pts = skm.Points(skm.REPR_BF16, Xb, d).with_screen()
        C = (Xb[synth.forgy_indices(n, k, seed=0).cuda()].to(torch.int32) << 16).view(torch.float32).contiguous()
    elif args.case in ("assign_prune", "assign_prune_front"):  # bf16 points, exact prefix-block pruning
        if args.case == "assign_prune_front":
            # the 10M PCA-256 recipe at n points and k = n_comp centroids: 1024
            # dimensions projected to d with the sample's own PCA, in bf16
            import dataclasses

            spec = dataclasses.replace(synth.WORKLOADS[HEAD], n=n, k=k, n_comp=k)
            del X
            X = synth.workload_points(spec, seed=0, device="cuda")
            mean, P, _ = skm.skm_pca_fit(X, d)
            X = skm.skm_project(X, P, mean, out_dtype=skm.DTYPE_BF16).view(torch.int16).contiguous()
            Xb = X
        else:
            Xb = X.to(torch.bfloat16).view(torch.int16).contiguous()
        pts = skm.Points(skm.REPR_BF16, Xb, d, flags=skm.FLAG_PRUNE)
        C = (Xb[synth.forgy_indices(n, k, seed=0).cuda()].to(torch.int32) << 16).view(torch.float32).contiguous()
    else:
        raise SystemExit(f"unknown case {args.case}")
    wsA = skm.workspace(skm.OP_ASSIGN, pts, k)
    wsU = skm.workspace(skm.OP_UPDATE, pts, k)
    a = torch.empty(n, dtype=torch.int32, device="cuda")
    cnt = torch.zeros(k, dtype=torch.int64, device="cuda")
    prev = None
    if args.case == "assign_rbq1_skm":  # the bound from a previous assignment, as in a later Lloyd iteration
        Cr, _, _, _, _ = skm.skm_fit(pts.with_flags(0), k, 0, init_idx=synth.forgy_indices(n, k, seed=0).cuda(),
                                     want_objective=False, want_dist=False)
        C = Cr
        prev, _ = skm.skm_assign(pts.with_flags(0), C, k, want_dist=False)
        tp = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        tp[0].record()
        skm.skm_assign(pts.with_flags(0), C, k, want_dist=False)
        tp[1].record()
    if args.case == "assign_prune_front":
        # a later Lloyd iteration: centroids after three dense steps, the bound
        # seeded with the dense assignment (the tensor-core front runs)
        dense = pts.with_flags(0).with_screen()
        C, _, _, _, _ = skm.skm_fit(dense, k, 3, C_init=C, want_objective=False, want_dist=False)
        prev, _ = skm.skm_assign(dense, C, k, want_dist=False)
        tp = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        tp[0].record()
        skm.skm_assign(dense, C, k, want_dist=False)
        tp[1].record()
    skm.skm_assign(pts, C, k, prev_assign=prev, want_dist=False, ws=wsA, out=a)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(args.reps):
        if args.case == "assign_rbq1_popcount":
            skm.skm_assign_rbq1_noalloc(pts, C, a)
        elif args.case.startswith("assign"):
            skm.skm_assign(pts, C, k, prev_assign=prev, want_dist=False, ws=wsA, out=a)
        else:
            skm.skm_update(pts, a, C.clone(), counts=cnt, ws=wsU)
    e1.record()
    torch.cuda.synchronize()
    out = {"case": args.case, "n": n, "d": d, "k": k, "reps": args.reps,
           "ms_per_call": e0.elapsed_time(e1) / args.reps}
    if args.case in ("assign_prune", "assign_prune_sq8", "assign_prune_front"):  # the work the bounds left
        st = skm.skm_assign_prune_stats(wsA)
        pairs = float(n) * k
        out["first_block_survivors"] = st["prune_first_block"] / pairs
        out["complete_survivors"] = st["prune_complete"] / pairs
        out["later_blocks_per_pair"] = st["prune_blocks"] / pairs
        if args.case == "assign_prune_front":
            out["prune_stats"] = st
            out["dense_screen_ms"] = tp[0].elapsed_time(tp[1])
    if args.case == "assign_f32":  # how often the screen alone decides a row
        _, _, _, _, stats = skm.skm_fit(pts, k, 0, C_init=C, want_objective=False, want_dist=False)
        out["screen_stats"] = stats
    if args.case == "assign_rbq1_skm":  # survivors per checkpoint, against the dense tensor-core call
        torch.cuda.synchronize()
        out["dense_tensor_ms"] = tp[0].elapsed_time(tp[1])
        _, _, _, _, stats = skm.skm_fit(pts, k, 1, C_init=C, want_objective=False, want_dist=False)
        pairs = 2.0 * n * k
        out["after_checkpoint_1"] = stats["prune_first_block"] / pairs
        out["after_checkpoint_2"] = stats["prune_complete"] / pairs
        out["same_assignment_as_dense_fraction"] = float((a == prev).float().mean())
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
    ap.add_argument("--e2e-chunks", type=int, default=E2E_CHUNKS, help="row ranges of the host-memory step")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-prune", action="store_true", help="skip the pruned assignment of the headline workload")
    ap.add_argument("--no-extra", action="store_true", help="skip the 1M x 768 and 10M x 1024 1-bit iterations")
    ap.add_argument("--eager", action="store_true", help="time eager steps instead of CUDA-graph replays")
    ap.add_argument("--case", default=None,
                    help="single-operation run for profiling: assign_f32|assign_bf16|assign_rbq1|assign_rbq1_skm|assign_sq8|"
                         "assign_lvq4|"
                         "assign_rbq1_popcount|assign_prune|assign_prune_sq8|update_f32|update_rbq1|update_sq8|"
                         "update_lvq4|project|quantize_sq8|quantize_rbq1|quantize_lvq4")
    ap.add_argument("--n", type=int, default=200_000)
    ap.add_argument("--cold-screen", action="store_true",
                    help="headline step without SKM_FLAG_WARM (every call starts with no carried bound)")
    ap.add_argument("--dense", action="store_true",
                    help="headline step with the dense bf16 screen instead of the pruned assignment")
    ap.add_argument("--e4m3-copy", action="store_true",
                    help="--case assign_rbq1 / assign_lvq4: read the points from their e4m3 copy instead of packed")
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
