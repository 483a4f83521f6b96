// extern "C" entry points of libskm (declared in include/skm.h): argument
// validation on the host, workspace carving, and the launch sequences of the
// Lloyd k-means hot path (Section 2.3) for each representation.
#include <stdarg.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <mutex>
#include <vector>

#include "skm_internal.cuh"
#include "skm_tc.cuh"

namespace skm {

static thread_local char g_err[512] = "";
static std::atomic<unsigned long long> g_launches{0};

// ---- fault injection (host side; SKM_FAULT_* kinds 1..4)
static std::atomic<int> g_fault[5];
static std::once_flag g_fault_env;

static void fault_from_env() {
    const char *v = getenv("SKM_FAULT");
    if (!v) return;
    const char *names[5] = {"", "workspace", "launch", "status", "wait"};
    for (int kind = 1; kind <= 4; ++kind)
        if (strcmp(v, names[kind]) == 0) g_fault[kind].store(1);
}

bool fault_take(int kind) {
    std::call_once(g_fault_env, fault_from_env);
    if (kind < 1 || kind > 4) return false;
    int c = g_fault[kind].load();
    while (c > 0)
        if (g_fault[kind].compare_exchange_weak(c, c - 1)) return true;
    return false;
}

// ---- timer of the tensor-core kernel launches (profiling callers)
static std::mutex g_timer_mu;
static std::atomic<int> g_timer_on{0};
static cudaEvent_t g_timer_ev[2] = {nullptr, nullptr};

void tc_timer_mark(cudaStream_t st, int which) {
    if (!g_timer_on.load(std::memory_order_relaxed)) return;
    std::lock_guard<std::mutex> lock(g_timer_mu);
    if (g_timer_ev[which]) cudaEventRecord(g_timer_ev[which], st);
}

cudaError_t launched(int count) {
    g_launches.fetch_add((unsigned long long)count, std::memory_order_relaxed);
    const cudaError_t e = cudaGetLastError();
    if (e == cudaSuccess && fault_take(SKM_FAULT_LAUNCH)) return cudaErrorLaunchFailure;
    return e;
}

int set_error(int code, const char *fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof(g_err), fmt, ap);
    va_end(ap);
    return code;
}

static inline cudaStream_t S(void *s) { return static_cast<cudaStream_t>(s); }

constexpr int MAX_D = 4096;
constexpr int MAX_K = 65536;
constexpr int64_t MAX_N = (int64_t(1) << 31) - 1;
constexpr int64_t MAX_N_RBQ1 = int64_t(1) << 24;
constexpr int64_t MAX_N_LVQ4 = int64_t(1) << 26;
constexpr int RED_BLOCKS = 304;
constexpr int PRUNE_MAX_D = 1024;  // 2 x 152 SMs for column / objective reductions
constexpr int EMPTY_LOG = 4096;    // iterations whose empty-cluster counts skm_fit records

static int check_data(const skm_data *x, bool need_codes = true) {
    if (!x) return set_error(SKM_ERR_INVALID_ARG, "skm_data is NULL");
    if (x->repr < SKM_REPR_F32 || x->repr > SKM_REPR_LVQ4)
        return set_error(SKM_ERR_INVALID_ARG, "unknown repr %d", x->repr);
    if (x->d < 1 || x->d > MAX_D)
        return set_error(x->d < 1 ? SKM_ERR_INVALID_ARG : SKM_ERR_UNSUPPORTED,
                         "d = %d outside [1, %d]", x->d, MAX_D);
    if (x->n < 1 || x->n > MAX_N)
        return set_error(x->n < 1 ? SKM_ERR_INVALID_ARG : SKM_ERR_UNSUPPORTED,
                         "n = %lld outside [1, 2^31)", (long long)x->n);
    if (need_codes && !x->x) return set_error(SKM_ERR_INVALID_ARG, "x->x is NULL");
    if ((x->flags & SKM_FLAG_PRUNE) &&
        (x->repr == SKM_REPR_F32 || x->repr == SKM_REPR_BF16 || x->repr == SKM_REPR_SQ8) && x->d > PRUNE_MAX_D)
        return set_error(SKM_ERR_UNSUPPORTED, "SKM_FLAG_PRUNE supports d <= %d", PRUNE_MAX_D);
    if (x->repr == SKM_REPR_RBQ1) {
        if (x->n > MAX_N_RBQ1)
            return set_error(SKM_ERR_UNSUPPORTED, "RBQ1 supports n <= 2^24 (got %lld)",
                             (long long)x->n);
        if (!x->nx2 || !x->F || !x->popx || !x->m)
            return set_error(SKM_ERR_INVALID_ARG, "RBQ1 needs nx2, F, popx and m");
    }
    if ((x->flags & SKM_FLAG_SYMMETRIC) && x->repr != SKM_REPR_RBQ1)
        return set_error(SKM_ERR_INVALID_ARG, "SKM_FLAG_SYMMETRIC applies to RBQ1 only");
    if ((x->flags & SKM_FLAG_PRUNE) && x->repr == SKM_REPR_RBQ1) {
        int d1, d2;
        rbq1_seg_bounds(x->d, &d1, &d2);
        if (x->d > 1024 || d2 >= x->d)
            return set_error(SKM_ERR_UNSUPPORTED, "RBQ1 pruning needs 2 d1 < d <= 1024 (d = %d)", x->d);
        if (x->flags & SKM_FLAG_SYMMETRIC)
            return set_error(SKM_ERR_UNSUPPORTED, "RBQ1 pruning uses the asymmetric estimate");
        if (need_codes && (!x->seg_nx2 || !x->seg_F || !x->seg_popx))
            return set_error(SKM_ERR_INVALID_ARG, "RBQ1 pruning needs the segment factors seg_nx2, seg_F, seg_popx");
    }
    if (x->repr == SKM_REPR_LVQ4) {
        if (x->n > MAX_N_LVQ4)
            return set_error(SKM_ERR_UNSUPPORTED, "LVQ4 supports n <= 2^26 (got %lld)", (long long)x->n);
        if (!x->lvq) return set_error(SKM_ERR_INVALID_ARG, "LVQ4 needs the per-point terms lvq");
        if (((uintptr_t)x->lvq & 15) != 0)
            return set_error(SKM_ERR_INVALID_ARG, "LVQ4 terms lvq must be 16-byte aligned");
    }
    return SKM_OK;
}

static int check_k(const skm_data *x, int k, bool k_le_n = false) {
    if (k < 1 || k > MAX_K)
        return set_error(k < 1 ? SKM_ERR_INVALID_ARG : SKM_ERR_UNSUPPORTED,
                         "k = %d outside [1, %d]", k, MAX_K);
    if (k_le_n && (int64_t)k > x->n)
        return set_error(SKM_ERR_INVALID_ARG, "k = %d exceeds n = %lld", k, (long long)x->n);
    return SKM_OK;
}

// ------------------------------------------------------------ workspace plans
static bool use_prune(const skm_data *x) {
    return (x->flags & SKM_FLAG_PRUNE) && (x->repr == SKM_REPR_F32 || x->repr == SKM_REPR_BF16 ||
                                          x->repr == SKM_REPR_SQ8 || x->repr == SKM_REPR_RBQ1);
}

// Pruning counters, the first buffer of every assignment workspace: [0] pairs
// alive after the first block (or after the tensor-core front), [1]
// complete, [2] blocks evaluated after the first (the front's finish: every
// block it evaluated), [3] front dimensions (0: CUDA cores only), [4] rows the
// front listed for the CUDA-core finish, [5] rows pruned over all k after a
// list overflow, [6..8] that pruning's own [0..2], [9] k.
constexpr int PRUNE_CTRS = 10;

static void prune_stats_from(const unsigned long long (&h)[PRUNE_CTRS], skm_stats *out) {
    out->prune_first_block = (int64_t)h[0];
    out->prune_complete = (int64_t)(h[1] + h[7]);
    out->prune_blocks = (int64_t)(h[2] + h[8] + h[5] * h[9]);
    out->prune_front_dims = (int64_t)h[3];
    out->prune_rows_finished = (int64_t)h[4];
    out->prune_rows_full = (int64_t)h[5];
}

struct AssignBufs {
    unsigned long long *prune = nullptr;    // PRUNE_CTRS counters
    int32_t *nx = nullptr, *nc = nullptr;  // SQ8 with d > 1024 (__dp4a path)
    uint4 *planes = nullptr;                // RBQ1 with d > 1024 (AND + popcount path)
    Rbq1CInfo *info = nullptr;
    uint32_t *yw = nullptr;                 // LVQ4 with d > 1024 (__dp4a path): centroid nibbles
    float4 *linfo = nullptr;
    TcAssignBufs tc;                        // tensor-core paths (F32, BF16, SQ8, RBQ1)
    Rbq1SegInfo *seginfo = nullptr;         // RBQ1 with SKM_FLAG_PRUNE (planes above)
};

static void plan_assign(const skm_data *x, int k, Carver &cv, AssignBufs &b) {
    const int64_t n = x->n;
    const int d = x->d;
    b.prune = cv.take<unsigned long long>(PRUNE_CTRS);
    if (use_prune(x)) {
        if (x->repr == SKM_REPR_RBQ1) {
            b.planes = cv.take<uint4>((size_t)k * words_of(d));
            b.seginfo = cv.take<Rbq1SegInfo>(k);
        }
        tc_plan(-1, n, d, k, x->x, x->screen, false, cv, b.tc);  // statistics only
        // bf16 points: the tensor-core front, taken when a seed assignment is given
        if (tc_pfront_ok(x->repr, d, x->x) && !(x->flags & SKM_FLAG_PRUNE_CUDA_CORES))
            tc_plan_pfront(n, d, k, (x->flags & SKM_FLAG_WARM) != 0, cv, b.tc);
        return;
    }
    switch (x->repr) {
    case SKM_REPR_SQ8:
        if (d > TC_SQ8_MAX_D) {
            b.nx = cv.take<int32_t>(n);
            b.nc = cv.take<int32_t>(k);
        }
        break;
    case SKM_REPR_RBQ1:
        if (d > TC_RBQ1_MAX_D) {
            b.planes = cv.take<uint4>((size_t)k * words_of(d));
            b.info = cv.take<Rbq1CInfo>(k);
        }
        break;
    case SKM_REPR_LVQ4:
        if (d > TC_LVQ4_MAX_D) {
            b.yw = cv.take<uint32_t>((size_t)k * lvq4_words(d));
            b.linfo = cv.take<float4>(k);
        }
        break;
    default:
        break;
    }
    tc_plan(x->repr, n, d, k, x->x, x->screen, (x->flags & SKM_FLAG_WARM) != 0, cv, b.tc);
}

struct UpdateBufs {
    int32_t *counts32 = nullptr, *cursor = nullptr, *perm = nullptr, *scl = nullptr;
    int64_t *offsets = nullptr;
    int64_t *fq = nullptr;    // RBQ1: fixed-point weights round(F 2^e)
    uint32_t *sq = nullptr;   // LVQ4: round(s 2^e), sorted order
    int64_t *bq = nullptr;    // LVQ4: round(b 2^e), sorted order
    float *sumf = nullptr;    // F32/BF16: cluster sums [k][d]
    int64_t *sumi = nullptr;  // RBQ1: cluster sums [k][d + 1]; SQ8: [k][d]
    int32_t *flag = nullptr;  // raised by a streamed-sum wait that gave up
    int64_t *wsplit = nullptr;  // empty-cluster split: working member counts [k]
};

static void plan_update(const skm_data *x, int k, Carver &cv, UpdateBufs &b) {
    b.counts32 = cv.take<int32_t>(k);
    b.cursor = cv.take<int32_t>(k);
    b.offsets = cv.take<int64_t>((size_t)k + 1);
    b.perm = cv.take<int32_t>(x->n);
    b.scl = cv.take<int32_t>(x->n);
    if (x->repr == SKM_REPR_RBQ1) {
        b.fq = cv.take<int64_t>(x->n);
        b.sumi = cv.take<int64_t>((size_t)k * (x->d + 1));
    }
    if (x->repr == SKM_REPR_LVQ4) {
        b.sq = cv.take<uint32_t>(x->n);
        b.bq = cv.take<int64_t>(x->n);
        b.sumi = cv.take<int64_t>((size_t)k * (x->d + 1));
    }
    if (x->repr == SKM_REPR_SQ8) b.sumi = cv.take<int64_t>((size_t)k * x->d);
    if (x->repr == SKM_REPR_F32 || x->repr == SKM_REPR_BF16) b.sumf = cv.take<float>((size_t)k * x->d);
    b.flag = cv.take<int32_t>(1);
    b.wsplit = cv.take<int64_t>(k);
}

// skm_fit with SKM_FLAG_PRUNE on points the tensor-core front takes: the
// dense screen (a2) runs the iterations in which prefix pruning cannot pay
// (the first, and while more than one in FIT_MOVED_DIV of the rows change
// cluster), the pruned assignment (a) the later ones; a pruned iteration
// that keeps more than FIT_MAX_SURVIVORS centroids a row sends the next one
// back to the screen.  Both give the exact fp32 nearest centroid (they may
// break a tie within fp32 rounding differently).
constexpr int64_t FIT_MOVED_DIV = 100;
constexpr double FIT_MAX_SURVIVORS = 8.0;
static bool fit_front(const skm_data *x) {
    return use_prune(x) && tc_pfront_ok(x->repr, x->d, x->x) && !(x->flags & SKM_FLAG_PRUNE_CUDA_CORES);
}

__global__ void count_moved_kernel(const int32_t *__restrict__ a, const int32_t *__restrict__ b, int64_t n,
                                   unsigned long long *__restrict__ out) {
    unsigned long long c = 0;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        c += a[i] != b[i];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
    if ((threadIdx.x & 31) == 0 && c) atomicAdd(out, c);
}

struct FitBufs {
    uint8_t *screen = nullptr;  // built once per fit when the caller gave none
    AssignBufs a;
    AssignBufs a2;                           // fit_front: the dense screen's
    int32_t *aprev = nullptr;                // fit_front: the previous iteration's assignment
    unsigned long long *moved = nullptr;     // fit_front: rows that changed cluster
    UpdateBufs u;
    float *dist = nullptr;
    double *partials = nullptr, *sum = nullptr;
    unsigned int *maxbits = nullptr;
    int *e_dev = nullptr;
    int *status = nullptr;
    int64_t *counts = nullptr;
    int64_t *init_idx = nullptr;
    int64_t *empty_iter = nullptr;  // empty clusters after each update (first EMPTY_LOG iterations)
};

static void plan_fit(const skm_data *x, int k, Carver &cv, FitBufs &b) {
    skm_data xs = *x;
    if (x->repr == SKM_REPR_F32 || x->repr == SKM_REPR_BF16) xs.flags |= SKM_FLAG_WARM;  // as skm_fit
    // 1-bit codes the tensor-core kernel reads packed: no copy of the points
    const bool packed = tc_reads_packed(x->repr, x->d, x->x);
    if (!x->screen && !packed) {
        const size_t sb = tc_screen_bytes(x->repr, x->n, x->d, x->x);
        if (sb) {
            b.screen = cv.take<uint8_t>(sb);
            xs.screen = b.screen ? b.screen : reinterpret_cast<const void *>(1);  // measured
        }
    }
    plan_assign(&xs, k, cv, b.a);
    if (fit_front(x)) {
        skm_data xd = xs;
        xd.flags &= ~SKM_FLAG_PRUNE;
        plan_assign(&xd, k, cv, b.a2);
        b.aprev = cv.take<int32_t>(x->n);
        b.moved = cv.take<unsigned long long>(1);
    }
    plan_update(x, k, cv, b.u);
    b.dist = cv.take<float>(x->n);
    b.partials = cv.take<double>(RED_BLOCKS);
    b.sum = cv.take<double>(1);
    b.maxbits = cv.take<unsigned int>(1);
    b.e_dev = cv.take<int>(1);
    b.status = cv.take<int>(1);
    b.counts = cv.take<int64_t>(k);
    b.init_idx = cv.take<int64_t>(k);  // seeded Forgy indices (host-drawn)
    b.empty_iter = cv.take<int64_t>(EMPTY_LOG);
}

static int need_ws(const Carver &cv, size_t ws_bytes, void *ws) {
    if (fault_take(SKM_FAULT_WORKSPACE))
        return set_error(SKM_ERR_NO_MEMORY, "injected fault: workspace reported too small");
    if (cv.off > ws_bytes)
        return set_error(SKM_ERR_NO_MEMORY, "workspace too small: need %zu bytes, got %zu", cv.off,
                         ws_bytes);
    if (cv.off > 0 && !ws) return set_error(SKM_ERR_INVALID_ARG, "workspace is NULL");
    if (((uintptr_t)ws & 255) != 0)
        return set_error(SKM_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
    return SKM_OK;
}

// ------------------------------------------------------------ core steps
static int do_assign(const skm_data *x, const void *C, int k, const int32_t *prev,
                     int32_t *assign, float *dist, AssignBufs &b, cudaStream_t st) {
    const int64_t n = x->n;
    const int d = x->d;
    if (use_prune(x)) {
        if (x->repr == SKM_REPR_RBQ1) {
            SKM_CUDA_TRY(launch_rbq1_seg_cprep(static_cast<const float *>(C), k, d, x->m, b.planes, b.seginfo, st));
            SKM_CUDA_TRY(launch_assign_rbq1_seg(static_cast<const uint32_t *>(x->x), x->seg_nx2, x->seg_F,
                                                x->seg_popx, n, d, b.planes, b.seginfo, k, prev, assign, dist,
                                                b.prune, st));
            return SKM_OK;
        }
        if (prev && b.tc.pf_thr && tc_pfront_ok(x->repr, d, x->x) && ((uintptr_t)C & 15) == 0)
            return tc_assign_pfront(x, static_cast<const float *>(C), k, prev, assign, dist, b.tc, b.prune, st);
        if (x->repr == SKM_REPR_SQ8)
            SKM_CUDA_TRY(launch_prune_assign_sq8(static_cast<const uint8_t *>(x->x), n, d, static_cast<const uint8_t *>(C),
                                                 k, prev, assign, dist, b.prune, st));
        else
            SKM_CUDA_TRY(launch_prune_assign(x->x, x->repr == SKM_REPR_BF16, n, d,
                                             static_cast<const float *>(C), k, prev, assign, dist,
                                             b.prune, st));
        return SKM_OK;
    }
    switch (x->repr) {
    case SKM_REPR_F32:
        SKM_TRY(tc_assign_float(x, static_cast<const float *>(C), k, assign, dist, b.tc, st));
        break;
    case SKM_REPR_BF16:
        SKM_TRY(tc_assign_float(x, static_cast<const float *>(C), k, assign, dist, b.tc, st));
        (void)prev;
        break;
    case SKM_REPR_SQ8:
        SKM_TRY(tc_assign_sq8(x, static_cast<const uint8_t *>(C), k, b.nx, b.nc, assign, dist,
                              b.tc, st));
        break;
    case SKM_REPR_RBQ1:
        if (d <= TC_RBQ1_MAX_D) {
            SKM_TRY(tc_assign_rbq1(x, static_cast<const float *>(C), k, assign, dist, b.tc, st));
        } else if (x->flags & SKM_FLAG_SYMMETRIC) {
            uint32_t *yw = reinterpret_cast<uint32_t *>(b.planes);  // k sign words per centroid row fit
            SKM_CUDA_TRY(launch_rbq1_cprep_sym(static_cast<const float *>(C), k, d, x->m, nullptr, 0, yw, b.info, st));
            SKM_CUDA_TRY(launch_assign_rbq1_sym(static_cast<const uint32_t *>(x->x), x->nx2, x->F, n, d, yw, b.info, k,
                                                assign, dist, st));
        } else {
            SKM_CUDA_TRY(launch_rbq1_cprep(static_cast<const float *>(C), k, d, x->m, b.planes,
                                           b.info, st));
            SKM_CUDA_TRY(launch_assign_rbq1(static_cast<const uint32_t *>(x->x), x->nx2, x->F,
                                            x->popx, n, d, b.planes, b.info, k, assign, dist, st));
        }
        break;
    case SKM_REPR_LVQ4:
        if (d <= TC_LVQ4_MAX_D) {
            SKM_TRY(tc_assign_lvq4(x, static_cast<const float *>(C), k, assign, dist, b.tc, st));
        } else {
            SKM_CUDA_TRY(launch_lvq4_cprep(static_cast<const float *>(C), k, d, nullptr, 0, b.yw, b.linfo, st));
            SKM_CUDA_TRY(launch_assign_lvq4_simt(static_cast<const uint32_t *>(x->x),
                                                 reinterpret_cast<const float4 *>(x->lvq), n, d, b.yw, b.linfo, k,
                                                 assign, dist, st));
        }
        break;
    }
    return SKM_OK;
}

static int do_update(const skm_data *x, const int32_t *assign, int k, void *C, int64_t *counts,
                     void *partial, int e, UpdateBufs &b, cudaStream_t st) {
    const int64_t n = x->n;
    const int d = x->d;
    SKM_CUDA_TRY(launch_histogram(assign, n, k, b.counts32, st));
    SKM_CUDA_TRY(launch_scan_offsets(b.counts32, k, b.offsets, counts, partial ? 1 : 0, st));
    SKM_CUDA_TRY(cudaMemsetAsync(b.cursor, 0, sizeof(int32_t) * (size_t)k, st));
    SKM_CUDA_TRY(launch_scatter(assign, n, k, b.offsets, b.cursor, b.perm, b.scl, st));
    switch (x->repr) {
    case SKM_REPR_F32:
    case SKM_REPR_BF16: {
        const int bf = x->repr == SKM_REPR_BF16;
        const bool ring = ring_sum_float_ok(x->x, bf, d);
        float *Sf = partial ? nullptr : b.sumf;
        double *Sd = partial ? static_cast<double *>(partial) : nullptr;
        if (!partial) SKM_CUDA_TRY(cudaMemsetAsync(b.sumf, 0, sizeof(float) * (size_t)k * d, st));
        if (ring)
            SKM_CUDA_TRY(launch_ring_sum_float(x->x, bf, n, d, b.perm, b.scl, b.offsets, k, Sf, Sd,
                                               b.flag, st));
        else
            SKM_CUDA_TRY(launch_chunk_sum_float(x->x, bf, n, d, b.perm, b.scl, b.offsets, k, Sf, Sd, st));
        if (!partial)
            SKM_CUDA_TRY(launch_finalize_float32(b.sumf, counts, k, d, static_cast<float *>(C), st));
        break;
    }
    case SKM_REPR_SQ8: {
        const uint8_t *codes = static_cast<const uint8_t *>(x->x);
        if (ring_sum_sq8_ok(codes, d)) {
            int64_t *S = partial ? static_cast<int64_t *>(partial) : b.sumi;
            if (!partial) SKM_CUDA_TRY(cudaMemsetAsync(S, 0, sizeof(int64_t) * (size_t)k * d, st));
            SKM_CUDA_TRY(launch_ring_sum_sq8(codes, n, d, b.perm, b.scl, b.offsets, k, S, b.flag, st));
            if (!partial)
                SKM_CUDA_TRY(launch_finalize_sq8(S, counts, k, d, static_cast<uint8_t *>(C), st));
        } else {
            SKM_CUDA_TRY(launch_segsum_sq8(codes, d, b.perm, b.offsets, k, static_cast<uint8_t *>(C),
                                           static_cast<int64_t *>(partial), st));
        }
        break;
    }
    case SKM_REPR_RBQ1: {
        SKM_CUDA_TRY(launch_rbq1_fq(x->F, b.perm, b.offsets, k, n, e, b.fq, st));
        int64_t *T = partial ? static_cast<int64_t *>(partial) : b.sumi;
        if (!partial) SKM_CUDA_TRY(cudaMemsetAsync(T, 0, sizeof(int64_t) * (size_t)k * (d + 1), st));
        const uint32_t *codes = static_cast<const uint32_t *>(x->x);
        if (ring_sum_rbq1_ok(codes, d))
            SKM_CUDA_TRY(launch_ring_sum_rbq1(codes, b.fq, n, d, b.perm, b.scl, b.offsets, k, T,
                                              b.flag, st));
        else
            SKM_CUDA_TRY(launch_chunk_sum_rbq1(codes, b.fq, n, d, b.perm, b.scl, b.offsets, k, T, st));
        if (!partial)
            SKM_CUDA_TRY(launch_finalize_rbq1(T, counts, k, d, x->m, e, static_cast<float *>(C), st));
        break;
    }
    case SKM_REPR_LVQ4: {
        SKM_CUDA_TRY(launch_lvq4_q(reinterpret_cast<const float4 *>(x->lvq), b.perm, b.offsets, k, n, e, b.sq, b.bq,
                                   st));
        int64_t *T = partial ? static_cast<int64_t *>(partial) : b.sumi;
        if (!partial) SKM_CUDA_TRY(cudaMemsetAsync(T, 0, sizeof(int64_t) * (size_t)k * (d + 1), st));
        const uint32_t *codes = static_cast<const uint32_t *>(x->x);
        if (ring_sum_lvq4_ok(codes, d))
            SKM_CUDA_TRY(launch_ring_sum_lvq4(codes, b.sq, b.bq, n, d, b.perm, b.scl, b.offsets, k, T, b.flag, st));
        else
            SKM_CUDA_TRY(launch_chunk_sum_lvq4(codes, b.sq, b.bq, n, d, b.perm, b.scl, b.offsets, k, T, st));
        if (!partial) SKM_CUDA_TRY(launch_finalize_lvq4(T, counts, k, d, e, static_cast<float *>(C), st));
        break;
    }
    }
    return SKM_OK;
}

static size_t centroid_bytes(const skm_data *x, int k) {
    return (size_t)k * x->d * (x->repr == SKM_REPR_SQ8 ? 1 : 4);
}

}  // namespace skm

using namespace skm;

extern "C" {

const char *skm_last_error(void) { return g_err; }

int skm_inject_fault(int kind, int count) {
    std::call_once(g_fault_env, fault_from_env);
    if (kind < 1 || kind > 4 || count < 0) return set_error(SKM_ERR_INVALID_ARG, "fault kind %d, count %d", kind, count);
    g_fault[kind].store(count);
    return SKM_OK;
}

int skm_fault_armed(int kind) {
    std::call_once(g_fault_env, fault_from_env);
    return (kind < 1 || kind > 4) ? 0 : g_fault[kind].load();
}

int skm_version(void) { return 100; }

uint64_t skm_kernel_launches(void) { return (uint64_t)g_launches.load(std::memory_order_relaxed); }

int skm_kernel_timer(int on) {
    std::lock_guard<std::mutex> lock(g_timer_mu);
    if (on) {
        for (auto &e : g_timer_ev)
            if (!e && cudaEventCreate(&e) != cudaSuccess) {
                e = nullptr;
                return set_error(SKM_ERR_CUDA, "cudaEventCreate failed");
            }
    }
    g_timer_on.store(on ? 1 : 0);
    return SKM_OK;
}

int skm_kernel_timer_ms(float *ms) {
    if (!ms) return set_error(SKM_ERR_INVALID_ARG, "ms is NULL");
    std::lock_guard<std::mutex> lock(g_timer_mu);
    if (!g_timer_ev[0] || !g_timer_ev[1]) return set_error(SKM_ERR_INVALID_ARG, "the timer was never enabled");
    SKM_CUDA_TRY(cudaEventSynchronize(g_timer_ev[1]));
    SKM_CUDA_TRY(cudaEventElapsedTime(ms, g_timer_ev[0], g_timer_ev[1]));
    return SKM_OK;
}

size_t skm_workspace_size(int op, const skm_data *x, int k) {
    Carver cv(nullptr, 0);
    switch (op) {
    case 0: {
        if (check_data(x, false) || check_k(x, k)) return 0;
        AssignBufs b;
        plan_assign(x, k, cv, b);
        break;
    }
    case 1: {
        if (check_data(x, false) || check_k(x, k)) return 0;
        UpdateBufs b;
        plan_update(x, k, cv, b);
        break;
    }
    case 2: {
        if (check_data(x, false) || check_k(x, k, true)) return 0;
        FitBufs b;
        plan_fit(x, k, cv, b);
        break;
    }
    case 5: {  // segmented assignment
        if (check_data(x, false) || check_k(x, k)) return 0;
        AssignBufs b;
        plan_assign(x, k, cv, b);
        cv.take<int32_t>((size_t)cdiv(x->n, 128));
        cv.take<int32_t>((size_t)cdiv(x->n, 128));
        break;
    }
    case 3: {  // quantize: column reductions
        if (!x || x->d < 1 || x->d > MAX_D) {
            set_error(SKM_ERR_INVALID_ARG, "bad skm_data for op 3");
            return 0;
        }
        cv.take<double>((size_t)RED_BLOCKS * x->d);
        cv.take<float>((size_t)RED_BLOCKS * x->d);
        cv.take<float>((size_t)RED_BLOCKS * x->d);
        cv.take<unsigned int>(1);
        cv.take<int>(1);
        break;
    }
    case 6:  // skm_project on tensor cores, one pass
    case 7: {  // ... the smallest workspace (rows in chunks)
        if (!x || x->d < 1 || x->d > MAX_D || x->n < 1 || k < 1 || k > x->d) {
            set_error(SKM_ERR_INVALID_ARG, "bad skm_data / d_out for op %d", op);
            return 0;
        }
        return op == 6 ? tc_project_ws_full(x->n, x->d, k) : tc_project_ws_min(x->d, k);
    }
    case 4: {  // pca
        if (!x || x->d < 1 || x->d > MAX_D) {
            set_error(SKM_ERR_INVALID_ARG, "bad skm_data for op 4");
            return 0;
        }
        const int d = x->d;
        const int splits = 32;
        cv.take<double>((size_t)RED_BLOCKS * d);
        cv.take<double>((size_t)splits * d * d);
        cv.take<double>((size_t)d * d);
        break;
    }
    default:
        set_error(SKM_ERR_INVALID_ARG, "unknown op %d", op);
        return 0;
    }
    return cv.off < 256 ? 256 : cv.off;
}

int skm_project(const float *X, int64_t n, int d, const float *mean, const float *P, int d_out,
                int out_dtype, void *Y, void *ws, size_t ws_bytes, void *stream) {
    if (!X || !P || !Y) return set_error(SKM_ERR_INVALID_ARG, "NULL pointer");
    if (n < 1 || d < 1 || d > MAX_D || d_out < 1 || d_out > d)
        return set_error(SKM_ERR_INVALID_ARG, "bad shape n=%lld d=%d d_out=%d", (long long)n, d,
                         d_out);
    if (out_dtype != SKM_DTYPE_F32 && out_dtype != SKM_DTYPE_BF16)
        return set_error(SKM_ERR_INVALID_ARG, "bad out_dtype %d", out_dtype);
    if (ws && ((uintptr_t)ws & 255) != 0)
        return set_error(SKM_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
    if (ws && ws_bytes >= tc_project_ws_min(d, d_out) && n < (int64_t(1) << 29))
        return tc_project(X, n, d, mean, P, d_out, out_dtype == SKM_DTYPE_BF16, Y, ws, ws_bytes, S(stream));
    SKM_CUDA_TRY(launch_project(X, n, d, mean, P, d_out, out_dtype == SKM_DTYPE_BF16, Y,
                                S(stream)));
    return SKM_OK;
}

int skm_project_hadamard(const float *X, int64_t n, int d, const float *mean, const float *sigma, int D,
                         int out_dtype, void *Y, void *stream) {
    if (!X || !sigma || !Y) return set_error(SKM_ERR_INVALID_ARG, "NULL pointer");
    if (n < 1 || d < 1 || d > MAX_D) return set_error(SKM_ERR_INVALID_ARG, "bad shape n=%lld d=%d", (long long)n, d);
    if (D < 32 || D > 4096 || (D & (D - 1)) != 0 || D < d)
        return set_error(SKM_ERR_INVALID_ARG, "D = %d must be a power of two in [max(32, d), 4096]", D);
    if (out_dtype != SKM_DTYPE_F32 && out_dtype != SKM_DTYPE_BF16)
        return set_error(SKM_ERR_INVALID_ARG, "bad out_dtype %d", out_dtype);
    SKM_CUDA_TRY(launch_hadamard(X, n, d, mean, sigma, D, out_dtype == SKM_DTYPE_BF16, Y, S(stream)));
    return SKM_OK;
}

int skm_unproject(const float *Y, int64_t n, int d_out, const float *P, const float *mean, int d, float *X,
                  void *stream) {
    if (!Y || !P || !X) return set_error(SKM_ERR_INVALID_ARG, "NULL pointer");
    if (n < 1 || n > 65535LL * 16 || d < 1 || d > MAX_D || d_out < 1 || d_out > MAX_D)
        return set_error(SKM_ERR_INVALID_ARG, "bad shape n=%lld d=%d d_out=%d", (long long)n, d, d_out);
    SKM_CUDA_TRY(launch_unproject(Y, n, d_out, P, mean, d, X, S(stream)));
    return SKM_OK;
}

int skm_copy_from_host(void *dst, const void *src_host, size_t bytes, void *stream) {
    if (bytes == 0) return SKM_OK;
    if (!dst || !src_host) return set_error(SKM_ERR_INVALID_ARG, "NULL pointer");
    void *src_dev = nullptr;
    const cudaError_t e = cudaHostGetDevicePointer(&src_dev, const_cast<void *>(src_host), 0);
    if (e != cudaSuccess || !src_dev) {
        (void)cudaGetLastError();  // clear the failed query's (non-sticky) error
        return set_error(SKM_ERR_INVALID_ARG, "src_host is not mapped page-locked host memory (%s)",
                         cudaGetErrorString(e));
    }
    SKM_CUDA_TRY(launch_copy_from_host(src_dev, dst, bytes, S(stream)));
    return SKM_OK;
}

int skm_forgy_indices(uint64_t seed, int64_t n, int k, int64_t *idx_host) {
    if (!idx_host) return set_error(SKM_ERR_INVALID_ARG, "idx_host is NULL");
    if (n < 1 || k < 1 || (int64_t)k > n) return set_error(SKM_ERR_INVALID_ARG, "need 1 <= k <= n (k=%d n=%lld)", k, (long long)n);
    forgy_indices(seed, n, k, idx_host);
    return SKM_OK;
}

int skm_make_rotation(uint64_t seed, int d, float *P_host) {
    if (!P_host || d < 1 || d > MAX_D) return set_error(SKM_ERR_INVALID_ARG, "bad arguments");
    std::vector<double> A((size_t)d * d);
    philox_gaussians(seed, (int64_t)d * d, A.data());
    householder_qr_q(d, A.data());
    for (size_t i = 0; i < A.size(); ++i) P_host[i] = (float)A[i];
    return SKM_OK;
}

int skm_pca_fit(const float *X, int64_t n, int d, int d_out, float *mean, float *P,
                float *eigvals, void *ws, size_t ws_bytes, void *stream) {
    if (!X || !mean || !P) return set_error(SKM_ERR_INVALID_ARG, "NULL pointer");
    if (n < 2 || d < 1 || d > MAX_D || d_out < 1 || d_out > d)
        return set_error(SKM_ERR_INVALID_ARG, "bad shape");
    cudaStream_t st = S(stream);
    const int splits = 32;
    Carver cv(ws, ws_bytes);
    double *psum = cv.take<double>((size_t)RED_BLOCKS * d);
    double *partial = cv.take<double>((size_t)splits * d * d);
    double *cov = cv.take<double>((size_t)d * d);
    SKM_TRY(need_ws(cv, ws_bytes, ws));
    const int nblk = (int)std::min<int64_t>(RED_BLOCKS, n);
    SKM_CUDA_TRY(launch_colsum_partial(X, n, d, psum, nblk, st));
    SKM_CUDA_TRY(launch_colmean_finish(psum, nblk, d, n, mean, nullptr, st));
    SKM_CUDA_TRY(launch_cov_partial(X, n, d, mean, partial, splits, st));
    SKM_CUDA_TRY(launch_cov_reduce(partial, splits, d, cov, st));
    std::vector<double> A((size_t)d * d), w(d);
    SKM_CUDA_TRY(cudaMemcpyAsync(A.data(), cov, sizeof(double) * A.size(), cudaMemcpyDeviceToHost,
                                 st));
    SKM_CUDA_TRY(cudaStreamSynchronize(st));
    for (auto &v : A) v /= (double)n;
    if (symmetric_eigen(d, A.data(), w.data()) != 0)
        return set_error(SKM_ERR_UNSUPPORTED, "eigen-decomposition did not converge");
    std::vector<int> order(d);
    for (int i = 0; i < d; ++i) order[i] = i;
    std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return w[a] > w[b]; });
    std::vector<float> Ph((size_t)d * d_out), wh(d_out);
    for (int j = 0; j < d_out; ++j) {
        const int c = order[j];
        int piv = 0;
        for (int i = 1; i < d; ++i)
            if (fabs(A[(size_t)i * d + c]) > fabs(A[(size_t)piv * d + c])) piv = i;
        const double sg = A[(size_t)piv * d + c] < 0 ? -1.0 : 1.0;
        for (int i = 0; i < d; ++i) Ph[(size_t)i * d_out + j] = (float)(sg * A[(size_t)i * d + c]);
        wh[j] = (float)w[c];
    }
    SKM_CUDA_TRY(cudaMemcpyAsync(P, Ph.data(), sizeof(float) * Ph.size(), cudaMemcpyHostToDevice,
                                 st));
    if (eigvals)
        SKM_CUDA_TRY(cudaMemcpyAsync(eigvals, wh.data(), sizeof(float) * wh.size(),
                                     cudaMemcpyHostToDevice, st));
    SKM_CUDA_TRY(cudaStreamSynchronize(st));
    return SKM_OK;
}

int skm_quantize(int repr, const float *X, int64_t n, int d, skm_quant_params *qp, void *codes,
                 void *ws, size_t ws_bytes, void *stream) {
    if (!X || !qp || !codes) return set_error(SKM_ERR_INVALID_ARG, "NULL pointer");
    if (n < 1 || n > MAX_N || d < 1 || d > MAX_D)
        return set_error(SKM_ERR_INVALID_ARG, "bad shape n=%lld d=%d", (long long)n, d);
    cudaStream_t st = S(stream);
    Carver cv(ws, ws_bytes);
    double *psum = cv.take<double>((size_t)RED_BLOCKS * d);
    float *pmin = cv.take<float>((size_t)RED_BLOCKS * d);
    float *pmax = cv.take<float>((size_t)RED_BLOCKS * d);
    const int nblk = (int)std::min<int64_t>(RED_BLOCKS, n);
    if (repr == SKM_REPR_SQ8) {
        if (!qp->b || !qp->s) return set_error(SKM_ERR_INVALID_ARG, "SQ8 needs b and s");
        if (qp->bits != 0 && qp->bits != 8 && qp->bits != 4)
            return set_error(SKM_ERR_INVALID_ARG, "bits = %d (0, 4 or 8)", qp->bits);
        const int levels = qp->bits == 4 ? 15 : 255;
        if (qp->fit) {
            SKM_TRY(need_ws(cv, ws_bytes, ws));
            SKM_CUDA_TRY(launch_colminmax_partial(X, n, d, pmin, pmax, nblk, st));
            SKM_CUDA_TRY(launch_sq8_params(pmin, pmax, nblk, d, levels, qp->b, qp->s, st));
        }
        SKM_CUDA_TRY(launch_sq8_encode(X, n, d, qp->b, qp->s, levels, static_cast<uint8_t *>(codes), st));
        return SKM_OK;
    }
    if (repr == SKM_REPR_RBQ1) {
        if (n > MAX_N_RBQ1) return set_error(SKM_ERR_UNSUPPORTED, "RBQ1 supports n <= 2^24");
        if (!qp->m || !qp->nx2 || !qp->F || !qp->popx)
            return set_error(SKM_ERR_INVALID_ARG, "RBQ1 needs m, nx2, F and popx");
        if (qp->fit) {
            unsigned *bits = cv.take<unsigned>(1);
            int *s_dev = cv.take<int>(1);
            SKM_TRY(need_ws(cv, ws_bytes, ws));
            SKM_CUDA_TRY(launch_mean_fixed(X, n, d, bits, s_dev, reinterpret_cast<unsigned long long *>(psum), qp->m,
                                           st));
        }
        SKM_CUDA_TRY(launch_rbq1_encode(X, n, d, qp->m, static_cast<uint32_t *>(codes), qp->nx2,
                                        qp->F, qp->popx, st));
        return SKM_OK;
    }
    if (repr == SKM_REPR_LVQ4) {
        if (n > MAX_N_LVQ4) return set_error(SKM_ERR_UNSUPPORTED, "LVQ4 supports n <= 2^26");
        if (!qp->lvq) return set_error(SKM_ERR_INVALID_ARG, "LVQ4 needs lvq");
        if (((uintptr_t)qp->lvq & 15) != 0 || ((uintptr_t)codes & 3) != 0)
            return set_error(SKM_ERR_INVALID_ARG, "LVQ4 outputs: lvq 16-byte, codes 4-byte aligned");
        SKM_CUDA_TRY(launch_lvq4_encode(X, n, d, static_cast<uint32_t *>(codes), reinterpret_cast<float4 *>(qp->lvq),
                                        st));
        return SKM_OK;
    }
    return set_error(SKM_ERR_INVALID_ARG, "skm_quantize: repr must be SQ8, RBQ1 or LVQ4");
}

int skm_lvq4_exponent(const float *lvq, int64_t n, int *e_host, void *ws, size_t ws_bytes, void *stream) {
    if (!lvq || !e_host || n < 1) return set_error(SKM_ERR_INVALID_ARG, "bad arguments");
    if (((uintptr_t)lvq & 15) != 0) return set_error(SKM_ERR_INVALID_ARG, "lvq must be 16-byte aligned");
    cudaStream_t st = S(stream);
    Carver cv(ws, ws_bytes);
    unsigned int *mb = cv.take<unsigned int>(1);
    int *ed = cv.take<int>(1);
    SKM_TRY(need_ws(cv, ws_bytes, ws));
    SKM_CUDA_TRY(launch_lvq4_exponent(reinterpret_cast<const float4 *>(lvq), n, mb, ed, st));
    SKM_CUDA_TRY(cudaMemcpyAsync(e_host, ed, sizeof(int), cudaMemcpyDeviceToHost, st));
    SKM_CUDA_TRY(cudaStreamSynchronize(st));
    return SKM_OK;
}

int skm_column_absmax(const float *X, int64_t n, int d, float *amax_host, void *ws, size_t ws_bytes, void *stream) {
    if (!X || !amax_host || !ws) return set_error(SKM_ERR_INVALID_ARG, "NULL pointer");
    if (n < 1 || d < 1 || d > MAX_D) return set_error(SKM_ERR_INVALID_ARG, "bad shape n=%lld d=%d", (long long)n, d);
    if (ws_bytes < sizeof(unsigned)) return set_error(SKM_ERR_NO_MEMORY, "workspace too small");
    cudaStream_t st = S(stream);
    unsigned *bits = static_cast<unsigned *>(ws);
    SKM_CUDA_TRY(launch_absmax_bits(X, n * (int64_t)d, bits, st));
    unsigned h = 0;
    SKM_CUDA_TRY(cudaMemcpyAsync(&h, bits, sizeof(h), cudaMemcpyDeviceToHost, st));
    SKM_CUDA_TRY(cudaStreamSynchronize(st));
    memcpy(amax_host, &h, sizeof(h));
    return SKM_OK;
}

int skm_mean_scale(float amax, int64_t n_total) { return host_mean_scale(amax, n_total < 1 ? 1 : n_total); }

int skm_column_sums_fixed(const float *X, int64_t n, int d, int s, int64_t *sums, void *stream) {
    if (!X || !sums) return set_error(SKM_ERR_INVALID_ARG, "NULL pointer");
    if (n < 1 || d < 1 || d > MAX_D) return set_error(SKM_ERR_INVALID_ARG, "bad shape n=%lld d=%d", (long long)n, d);
    SKM_CUDA_TRY(
        launch_colsum_fixed(X, n, d, nullptr, s, reinterpret_cast<unsigned long long *>(sums), false, S(stream)));
    return SKM_OK;
}

int skm_mean_from_sums(const int64_t *sums, int64_t n_total, int d, int s, float *m, void *stream) {
    if (!sums || !m) return set_error(SKM_ERR_INVALID_ARG, "NULL pointer");
    if (n_total < 1 || d < 1 || d > MAX_D)
        return set_error(SKM_ERR_INVALID_ARG, "bad shape n=%lld d=%d", (long long)n_total, d);
    SKM_CUDA_TRY(launch_mean_fixed_finish(reinterpret_cast<const unsigned long long *>(sums), d, n_total, nullptr, s,
                                          m, S(stream)));
    return SKM_OK;
}

int skm_rbq1_segment_bounds(int d, int *d1, int *d2) {
    if (!d1 || !d2 || d < 1) return set_error(SKM_ERR_INVALID_ARG, "bad arguments");
    rbq1_seg_bounds(d, d1, d2);
    if (*d2 >= d || d > 1024) return set_error(SKM_ERR_UNSUPPORTED, "no segments for d = %d (need 2 d1 < d <= 1024)", d);
    return SKM_OK;
}

int skm_rbq1_segments(const float *X, int64_t n, int d, const float *m, float *nx2s, float *Fs, int32_t *popxs,
                      void *stream) {
    if (!X || !m || !nx2s || !Fs || !popxs) return set_error(SKM_ERR_INVALID_ARG, "NULL pointer");
    if (n < 1 || n > MAX_N_RBQ1) return set_error(SKM_ERR_INVALID_ARG, "bad n = %lld", (long long)n);
    int d1, d2;
    SKM_TRY(skm_rbq1_segment_bounds(d, &d1, &d2));
    SKM_CUDA_TRY(launch_rbq1_seg_encode(X, n, d, m, nx2s, Fs, popxs, S(stream)));
    return SKM_OK;
}

int skm_rbq1_exponent(const float *F, int64_t n, int *e_host, void *ws, size_t ws_bytes,
                      void *stream) {
    if (!F || !e_host || n < 1) return set_error(SKM_ERR_INVALID_ARG, "bad arguments");
    cudaStream_t st = S(stream);
    Carver cv(ws, ws_bytes);
    unsigned int *mb = cv.take<unsigned int>(1);
    int *ed = cv.take<int>(1);
    SKM_TRY(need_ws(cv, ws_bytes, ws));
    SKM_CUDA_TRY(launch_rbq1_exponent(F, n, mb, ed, st));
    SKM_CUDA_TRY(cudaMemcpyAsync(e_host, ed, sizeof(int), cudaMemcpyDeviceToHost, st));
    SKM_CUDA_TRY(cudaStreamSynchronize(st));
    return SKM_OK;
}

size_t skm_screen_bytes(const skm_data *x) {
    if (check_data(x, false)) return 0;
    return tc_screen_bytes(x->repr, x->n, x->d, x->x);
}

int skm_screen_prep(const skm_data *x, void *screen, size_t screen_bytes, void *stream) {
    SKM_TRY(check_data(x));
    const size_t need = tc_screen_bytes(x->repr, x->n, x->d, x->x);
    if (need == 0) return set_error(SKM_ERR_INVALID_ARG, "this representation has no screening copy");
    if (!screen || screen_bytes < need)
        return set_error(SKM_ERR_NO_MEMORY, "screen buffer needs %zu bytes", need);
    if (((uintptr_t)screen & 255) != 0)
        return set_error(SKM_ERR_INVALID_ARG, "screen buffer must be 256-byte aligned");
    return tc_screen_prep(x, screen, S(stream));
}

int skm_assign(const skm_data *x, const void *C, int k, const int32_t *prev_assign,
               int32_t *assign, float *dist, void *ws, size_t ws_bytes, void *stream) {
    SKM_TRY(check_data(x));
    SKM_TRY(check_k(x, k));
    if (!C || !assign) return set_error(SKM_ERR_INVALID_ARG, "C and assign are required");
    Carver cv(ws, ws_bytes);
    AssignBufs b;
    plan_assign(x, k, cv, b);
    SKM_TRY(need_ws(cv, ws_bytes, ws));
    if (use_prune(x))
        SKM_CUDA_TRY(cudaMemsetAsync(b.prune, 0, PRUNE_CTRS * sizeof(unsigned long long), S(stream)));
    return do_assign(x, C, k, prev_assign, assign, dist, b, S(stream));
}

int skm_assign_prune_stats(const void *ws, size_t ws_bytes, skm_stats *out, void *stream) {
    if (!ws || !out) return set_error(SKM_ERR_INVALID_ARG, "ws and out are required");
    // the counters are the first buffer of every assignment workspace
    Carver cv(const_cast<void *>(ws), ws_bytes);
    const unsigned long long *cnt = cv.take<unsigned long long>(PRUNE_CTRS);
    if (!cv.fits()) return set_error(SKM_ERR_INVALID_ARG, "ws_bytes is smaller than the counters");
    unsigned long long h[PRUNE_CTRS];
    SKM_CUDA_TRY(cudaMemcpyAsync(h, cnt, sizeof(h), cudaMemcpyDeviceToHost, S(stream)));
    SKM_CUDA_TRY(cudaStreamSynchronize(S(stream)));
    memset(out, 0, sizeof(*out));
    prune_stats_from(h, out);
    return SKM_OK;
}

// Segmented assignment (the fine phase of hierarchical k-means): tensor-core
// paths only; the row-tile ranges are derived on the device.
static int do_assign_seg(const skm_data *x, const void *C, int k, const int32_t *group, const int32_t *base,
                         int nseg, int32_t *assign, float *dist, AssignBufs &b, int32_t *ct0, int32_t *nct,
                         cudaStream_t st) {
    TcSeg sg;
    sg.group = group;
    sg.base = base;
    sg.nseg = nseg;
    sg.ct0 = ct0;
    sg.nct = nct;
    switch (x->repr) {
    case SKM_REPR_F32:
    case SKM_REPR_BF16:
        return tc_assign_float(x, static_cast<const float *>(C), k, assign, dist, b.tc, st, &sg);
    case SKM_REPR_SQ8:
        return tc_assign_sq8(x, static_cast<const uint8_t *>(C), k, b.nx, b.nc, assign, dist, b.tc, st, &sg);
    case SKM_REPR_LVQ4:
        if (x->d > TC_LVQ4_MAX_D)
            return set_error(SKM_ERR_UNSUPPORTED, "segmented LVQ4 assignment needs d <= %d", TC_LVQ4_MAX_D);
        return tc_assign_lvq4(x, static_cast<const float *>(C), k, assign, dist, b.tc, st, &sg);
    default:
        if (x->d > TC_RBQ1_MAX_D)
            return set_error(SKM_ERR_UNSUPPORTED, "segmented RBQ1 assignment needs d <= %d", TC_RBQ1_MAX_D);
        return tc_assign_rbq1(x, static_cast<const float *>(C), k, assign, dist, b.tc, st, &sg);
    }
}

int skm_assign_segmented(const skm_data *x, const void *C, int k, const int32_t *group, const int32_t *base,
                         int nseg, int32_t *assign, float *dist, void *ws, size_t ws_bytes, void *stream) {
    SKM_TRY(check_data(x));
    SKM_TRY(check_k(x, k));
    if (!C || !assign || !group || !base || nseg < 1)
        return set_error(SKM_ERR_INVALID_ARG, "C, assign, group, base and nseg >= 1 are required");
    if (use_prune(x)) return set_error(SKM_ERR_UNSUPPORTED, "segmented assignment has no pruning variant");
    Carver cv(ws, ws_bytes);
    AssignBufs b;
    plan_assign(x, k, cv, b);
    int32_t *ct0 = cv.take<int32_t>((size_t)cdiv(x->n, 128));
    int32_t *nct = cv.take<int32_t>((size_t)cdiv(x->n, 128));
    SKM_TRY(need_ws(cv, ws_bytes, ws));
    return do_assign_seg(x, C, k, group, base, nseg, assign, dist, b, ct0, nct, S(stream));
}

// ------------------------------------------------------ hierarchical k-means
static int64_t row_bytes(const skm_data *x) {
    switch (x->repr) {
    case SKM_REPR_F32:
        return 4LL * x->d;
    case SKM_REPR_SQ8:
        return x->d;
    case SKM_REPR_RBQ1:
        return 4LL * words_of(x->d);
    case SKM_REPR_LVQ4:
        return 4LL * lvq4_words(x->d);
    default:
        return 2LL * x->d;
    }
}

struct HierBufs {
    uint8_t *meso_ws = nullptr;
    size_t meso_ws_bytes = 0;
    void *C_meso = nullptr;
    int32_t *a_meso = nullptr;
    int32_t *perm = nullptr, *skey = nullptr, *hist = nullptr, *sizes = nullptr, *base = nullptr;
    uint8_t *rows = nullptr;  // the points in meso order
    float *nx2 = nullptr, *F = nullptr;
    int32_t *popx = nullptr;
    float4 *lvq = nullptr;  // LVQ4 per-point terms in meso order
    uint8_t *screen = nullptr;
    AssignBufs a;
    int32_t *ct0 = nullptr, *nct = nullptr;
    UpdateBufs u;
    int32_t *a_sorted = nullptr;
    int64_t *counts = nullptr;
    int64_t *init_pos = nullptr;
    int *status = nullptr;
    unsigned int *maxbits = nullptr;
    int *e_dev = nullptr;
};

static void plan_hier(const skm_data *x, int k, int m, Carver &cv, HierBufs &b) {
    const int64_t n = x->n;
    {
        Carver mc(nullptr, 0);
        FitBufs fb;
        plan_fit(x, m, mc, fb);
        b.meso_ws_bytes = mc.off;
    }
    b.meso_ws = cv.take<uint8_t>(b.meso_ws_bytes);
    b.C_meso = cv.take<uint8_t>((size_t)m * (x->repr == SKM_REPR_SQ8 ? x->d : 4 * x->d));
    b.a_meso = cv.take<int32_t>(n);
    b.perm = cv.take<int32_t>(n);
    b.skey = cv.take<int32_t>(n);
    b.hist = cv.take<int32_t>((size_t)cdiv(n, 4096) * m);
    b.sizes = cv.take<int32_t>(m);
    b.base = cv.take<int32_t>((size_t)m + 1);
    b.rows = cv.take<uint8_t>((size_t)(n * row_bytes(x)));
    if (x->repr == SKM_REPR_RBQ1) {
        b.nx2 = cv.take<float>(n);
        b.F = cv.take<float>(n);
        b.popx = cv.take<int32_t>(n);
    }
    if (x->repr == SKM_REPR_LVQ4) b.lvq = cv.take<float4>(n);
    skm_data xs = *x;
    xs.x = b.rows;
    const size_t sb = tc_screen_bytes(x->repr, n, x->d, b.rows ? b.rows : reinterpret_cast<const void *>(16));
    b.screen = cv.take<uint8_t>(sb);
    xs.screen = b.screen ? b.screen : reinterpret_cast<const void *>(1);  // measured: a screen is given
    plan_assign(&xs, k, cv, b.a);
    b.ct0 = cv.take<int32_t>((size_t)cdiv(n, 128));
    b.nct = cv.take<int32_t>((size_t)cdiv(n, 128));
    plan_update(&xs, k, cv, b.u);
    b.a_sorted = cv.take<int32_t>(n);
    b.counts = cv.take<int64_t>(k);
    b.init_pos = cv.take<int64_t>(k);
    b.status = cv.take<int>(1);
    b.maxbits = cv.take<unsigned int>(1);
    b.e_dev = cv.take<int>(1);
}

static int hier_check(const skm_hier_config *cfg, const skm_data *x) {
    if (!cfg) return set_error(SKM_ERR_INVALID_ARG, "cfg is NULL");
    SKM_TRY(check_data(x));
    SKM_TRY(check_k(x, cfg->k, true));
    if (cfg->m < 1 || cfg->m > cfg->k || cfg->m > 12288)
        return set_error(SKM_ERR_INVALID_ARG, "m = %d outside [1, min(k, 12288)]", cfg->m);
    if (cfg->meso_iters < 0 || cfg->fine_iters < 0 || cfg->meso_iters > 100000 || cfg->fine_iters > 100000)
        return set_error(SKM_ERR_INVALID_ARG, "bad iteration counts");
    if (x->repr == SKM_REPR_BF16) return set_error(SKM_ERR_UNSUPPORTED, "hierarchical fit: F32, SQ8 or RBQ1 points");
    if (use_prune(x)) return set_error(SKM_ERR_UNSUPPORTED, "hierarchical fit has no pruning variant");
    if ((x->repr == SKM_REPR_SQ8 && x->d > TC_SQ8_MAX_D) || (x->repr == SKM_REPR_RBQ1 && x->d > TC_RBQ1_MAX_D) ||
        (x->repr == SKM_REPR_LVQ4 && x->d > TC_LVQ4_MAX_D))
        return set_error(SKM_ERR_UNSUPPORTED, "hierarchical SQ8 / RBQ1 / LVQ4 fit needs d <= 1024");
    return SKM_OK;
}

// Fine clusters per meso cluster: k apportioned by size (floor of k n_i / N,
// the rest to the largest remainders k n_i mod N, ties to the lower index);
// a non-empty meso cluster left with none takes one from the largest.
static void fine_counts(const std::vector<int32_t> &sizes, int k, std::vector<int> &kf) {
    const int m = (int)sizes.size();
    int64_t N = 0;
    for (int v : sizes) N += v;
    kf.assign(m, 0);
    std::vector<int64_t> rem(m);
    int given = 0;
    for (int i = 0; i < m; ++i) {
        kf[i] = (int)((int64_t)k * sizes[i] / N);
        rem[i] = (int64_t)k * sizes[i] % N;
        given += kf[i];
    }
    std::vector<int> order(m);
    for (int i = 0; i < m; ++i) order[i] = i;
    std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return rem[a] > rem[b]; });
    for (int t = 0; t < k - given; ++t) kf[order[t]] += 1;
    for (int i = 0; i < m; ++i)
        if (sizes[i] > 0 && kf[i] == 0) {
            int j = 0;
            for (int t = 1; t < m; ++t)
                if (kf[t] > kf[j]) j = t;
            kf[j] -= 1;
            kf[i] = 1;
        }
}

int skm_fit_hierarchical(const skm_hier_config *cfg, const skm_data *x, const int64_t *meso_init_idx,
                         void *C_out, int32_t *assign_out, int32_t *meso_assign_out, int32_t *fine_counts_host,
                         skm_stats *stats_host, void *ws, size_t ws_bytes, void *stream) {
    SKM_TRY(hier_check(cfg, x));
    if (!meso_init_idx || !C_out || !assign_out)
        return set_error(SKM_ERR_INVALID_ARG, "meso_init_idx, C_out and assign_out are required");
    const int k = cfg->k, m = cfg->m;
    const int64_t n = x->n;
    const int d = x->d;
    cudaStream_t st = S(stream);
    Carver cv(ws, ws_bytes);
    HierBufs b;
    plan_hier(x, k, m, cv, b);
    SKM_TRY(need_ws(cv, ws_bytes, ws));

    // MESO-CLUSTERING: Lloyd with m clusters from the given Forgy indices
    skm_fit_config mc{};
    mc.k = m;
    mc.iters = cfg->meso_iters;
    SKM_TRY(skm_fit(&mc, x, nullptr, meso_init_idx, b.C_meso, b.a_meso, nullptr, nullptr, nullptr, b.meso_ws,
                    b.meso_ws_bytes, stream));
    if (meso_assign_out)
        SKM_CUDA_TRY(cudaMemcpyAsync(meso_assign_out, b.a_meso, sizeof(int32_t) * n, cudaMemcpyDeviceToDevice, st));

    // points in meso order (stable), fine-cluster budget per meso cluster
    SKM_CUDA_TRY(launch_stable_sort(b.a_meso, n, m, b.hist, b.sizes, b.perm, b.skey, st));
    std::vector<int32_t> sizes(m);
    SKM_CUDA_TRY(cudaMemcpyAsync(sizes.data(), b.sizes, sizeof(int32_t) * m, cudaMemcpyDeviceToHost, st));
    SKM_CUDA_TRY(cudaStreamSynchronize(st));
    std::vector<int> kf;
    fine_counts(sizes, k, kf);
    std::vector<int32_t> base(m + 1, 0);
    std::vector<int64_t> init(k);
    int64_t off = 0;
    for (int i = 0; i < m; ++i) {
        base[i + 1] = base[i] + kf[i];
        for (int t = 0; t < kf[i]; ++t) init[base[i] + t] = off + (int64_t)t * sizes[i] / kf[i];
        off += sizes[i];
    }
    if (fine_counts_host)
        for (int i = 0; i < m; ++i) fine_counts_host[i] = kf[i];
    SKM_CUDA_TRY(cudaMemcpyAsync(b.base, base.data(), sizeof(int32_t) * (m + 1), cudaMemcpyHostToDevice, st));
    SKM_CUDA_TRY(cudaMemcpyAsync(b.init_pos, init.data(), sizeof(int64_t) * k, cudaMemcpyHostToDevice, st));
    SKM_CUDA_TRY(launch_gather_rows_bytes(x->x, row_bytes(x), b.perm, n, b.rows, st));
    skm_data xs = *x;
    xs.x = b.rows;
    xs.screen = nullptr;
    if (x->repr == SKM_REPR_RBQ1) {
        SKM_CUDA_TRY(launch_gather_rows_bytes(x->nx2, 4, b.perm, n, b.nx2, st));
        SKM_CUDA_TRY(launch_gather_rows_bytes(x->F, 4, b.perm, n, b.F, st));
        SKM_CUDA_TRY(launch_gather_rows_bytes(x->popx, 4, b.perm, n, b.popx, st));
        xs.nx2 = b.nx2;
        xs.F = b.F;
        xs.popx = b.popx;
        SKM_CUDA_TRY(launch_rbq1_exponent(x->F, n, b.maxbits, b.e_dev, st));
        int e = 0;
        SKM_CUDA_TRY(cudaMemcpyAsync(&e, b.e_dev, sizeof(int), cudaMemcpyDeviceToHost, st));
        SKM_CUDA_TRY(cudaStreamSynchronize(st));
        xs.rbq1_exp = e;
    }
    if (x->repr == SKM_REPR_LVQ4) {
        SKM_CUDA_TRY(launch_gather_rows_bytes(x->lvq, 16, b.perm, n, b.lvq, st));
        xs.lvq = reinterpret_cast<const float *>(b.lvq);
        SKM_CUDA_TRY(launch_lvq4_exponent(reinterpret_cast<const float4 *>(x->lvq), n, b.maxbits, b.e_dev, st));
        int e = 0;
        SKM_CUDA_TRY(cudaMemcpyAsync(&e, b.e_dev, sizeof(int), cudaMemcpyDeviceToHost, st));
        SKM_CUDA_TRY(cudaStreamSynchronize(st));
        xs.rbq1_exp = e;
    }
    SKM_TRY(tc_screen_prep(&xs, b.screen, st));
    xs.screen = b.screen;
    SKM_TRY(tc_init_stats(b.a.tc, st));

    // FINE-CLUSTERING: every meso cluster at once, each point against its own
    // meso cluster's fine centroids; initial centroids at evenly spaced members
    SKM_CUDA_TRY(cudaMemsetAsync(b.status, 0, sizeof(int), st));
    if (x->repr == SKM_REPR_RBQ1)
        SKM_CUDA_TRY(launch_rbq1_decode_rows(static_cast<const uint32_t *>(xs.x), xs.F, n, d, x->m, xs.rbq1_exp,
                                             b.init_pos, k, static_cast<float *>(C_out), b.status, st));
    else if (x->repr == SKM_REPR_LVQ4)
        SKM_CUDA_TRY(launch_lvq4_decode_rows(static_cast<const uint32_t *>(xs.x), b.lvq, n, d, xs.rbq1_exp,
                                             b.init_pos, k, static_cast<float *>(C_out), b.status, st));
    else
        SKM_CUDA_TRY(launch_gather_rows(xs.x, n, x->repr == SKM_REPR_SQ8 ? 1 : 4, d, b.init_pos, k, C_out,
                                        b.status, st));
    SKM_CUDA_TRY(cudaMemsetAsync(b.u.flag, 0, sizeof(int32_t), st));
    for (int it = 0; it <= cfg->fine_iters; ++it) {
        SKM_TRY(do_assign_seg(&xs, C_out, k, b.skey, b.base, m, b.a_sorted, nullptr, b.a, b.ct0, b.nct, st));
        if (it == cfg->fine_iters) break;
        SKM_TRY(do_update(&xs, b.a_sorted, k, C_out, b.counts, nullptr, xs.rbq1_exp, b.u, st));
    }
    if (cfg->refine) {  // one vanilla iteration over all points, then the final assignment
        SKM_TRY(do_assign(&xs, C_out, k, nullptr, b.a_sorted, nullptr, b.a, st));
        SKM_TRY(do_update(&xs, b.a_sorted, k, C_out, b.counts, nullptr, xs.rbq1_exp, b.u, st));
        SKM_TRY(do_assign(&xs, C_out, k, nullptr, b.a_sorted, nullptr, b.a, st));
    }
    SKM_CUDA_TRY(launch_unpermute(b.a_sorted, b.perm, n, assign_out, st));
    SKM_CUDA_TRY(cudaStreamSynchronize(st));
    skm_stats local;
    memset(&local, 0, sizeof(local));
    SKM_TRY(tc_read_stats(b.a.tc, &local, st));
    int32_t uflag = 0;
    SKM_CUDA_TRY(cudaMemcpy(&uflag, b.u.flag, sizeof(uflag), cudaMemcpyDeviceToHost));
    if (uflag) return set_error(SKM_ERR_TIMEOUT, "an update pipeline wait exceeded its limit");
    if (stats_host) {
        local.empty_per_iter = stats_host->empty_per_iter;  // an input field, left as given
        *stats_host = local;
    }
    return SKM_OK;
}

size_t skm_hier_workspace_size(const skm_hier_config *cfg, const skm_data *x) {
    if (hier_check(cfg, x)) return 0;
    Carver cv(nullptr, 0);
    HierBufs b;
    plan_hier(x, cfg->k, cfg->m, cv, b);
    return cv.off;
}

int skm_update(const skm_data *x, const int32_t *assign, int k, void *C_inout, int64_t *counts,
               void *partial, void *ws, size_t ws_bytes, void *stream) {
    SKM_TRY(check_data(x));
    SKM_TRY(check_k(x, k));
    if (!assign || !counts || (!C_inout && !partial))
        return set_error(SKM_ERR_INVALID_ARG, "assign, counts and C_inout/partial are required");
    Carver cv(ws, ws_bytes);
    UpdateBufs b;
    plan_update(x, k, cv, b);
    SKM_TRY(need_ws(cv, ws_bytes, ws));
    SKM_CUDA_TRY(cudaMemsetAsync(b.flag, 0, sizeof(int32_t), S(stream)));
    return do_update(x, assign, k, C_inout, counts, partial, x->rbq1_exp, b, S(stream));
}

int skm_merge_partials(void *dst, const void *src, int64_t count, int elem_type, void *stream) {
    if (!dst || !src || count < 0 || (elem_type != 0 && elem_type != 1))
        return set_error(SKM_ERR_INVALID_ARG, "bad arguments");
    SKM_CUDA_TRY(launch_merge(dst, src, count, elem_type, S(stream)));
    return SKM_OK;
}

int skm_update_finalize(const skm_data *x, const void *partial, const int64_t *counts, int k,
                        void *C_inout, void *stream) {
    SKM_TRY(check_data(x, false));
    if (!partial || !counts || !C_inout || k < 1)
        return set_error(SKM_ERR_INVALID_ARG, "bad arguments");
    cudaStream_t st = S(stream);
    switch (x->repr) {
    case SKM_REPR_F32:
    case SKM_REPR_BF16:
        SKM_CUDA_TRY(launch_finalize_float(static_cast<const double *>(partial), counts, k, x->d,
                                           static_cast<float *>(C_inout), st));
        break;
    case SKM_REPR_SQ8:
        SKM_CUDA_TRY(launch_finalize_sq8(static_cast<const int64_t *>(partial), counts, k, x->d,
                                         static_cast<uint8_t *>(C_inout), st));
        break;
    case SKM_REPR_RBQ1:
        if (!x->m) return set_error(SKM_ERR_INVALID_ARG, "RBQ1 finalize needs m");
        SKM_CUDA_TRY(launch_finalize_rbq1(static_cast<const int64_t *>(partial), counts, k, x->d,
                                          x->m, x->rbq1_exp, static_cast<float *>(C_inout), st));
        break;
    case SKM_REPR_LVQ4:
        SKM_CUDA_TRY(launch_finalize_lvq4(static_cast<const int64_t *>(partial), counts, k, x->d, x->rbq1_exp,
                                          static_cast<float *>(C_inout), st));
        break;
    }
    return SKM_OK;
}

int skm_fit(const skm_fit_config *cfg, const skm_data *x, const void *C_init,
            const int64_t *init_idx, void *C_out, int32_t *assign_out, float *dist_out,
            double *objective_host, skm_stats *stats_host, void *ws, size_t ws_bytes,
            void *stream) {
    if (!cfg) return set_error(SKM_ERR_INVALID_ARG, "cfg is NULL");
    SKM_TRY(check_data(x));
    const int k = cfg->k;
    SKM_TRY(check_k(x, k, true));
    if (cfg->iters < 0 || cfg->iters > 100000)
        return set_error(SKM_ERR_INVALID_ARG, "iters = %d", cfg->iters);
    if (cfg->empty_policy != SKM_EMPTY_KEEP && cfg->empty_policy != SKM_EMPTY_SPLIT)
        return set_error(SKM_ERR_INVALID_ARG, "empty_policy = %d", cfg->empty_policy);
    if (!C_out || !assign_out) return set_error(SKM_ERR_INVALID_ARG, "C_out and assign_out required");
    if (!C_init && x->repr == SKM_REPR_BF16)
        return set_error(SKM_ERR_INVALID_ARG, "BF16 fit needs fp32 C_init");
    cudaStream_t st = S(stream);
    Carver cv(ws, ws_bytes);
    FitBufs b;
    plan_fit(x, k, cv, b);
    SKM_TRY(need_ws(cv, ws_bytes, ws));
    const int64_t n = x->n;
    const int d = x->d;

    skm_data xd = *x;
    if (!x->screen && b.screen) {
        SKM_TRY(tc_screen_prep(x, b.screen, st));
        xd.screen = b.screen;
    }
    // the iterations' screens start from the bounds the previous one left; the
    // first starts cold whatever state the workspace held (other points)
    if (x->repr == SKM_REPR_F32 || x->repr == SKM_REPR_BF16) xd.flags |= SKM_FLAG_WARM;
    for (AssignBufs *ab : {&b.a, &b.a2}) {
        if (ab->tc.warm_hdr) SKM_CUDA_TRY(cudaMemsetAsync(ab->tc.warm_hdr, 0, 4 * sizeof(int64_t), st));
        if (ab->tc.pf_whdr) SKM_CUDA_TRY(cudaMemsetAsync(ab->tc.pf_whdr, 0, 8 * sizeof(int64_t), st));
    }
    const bool adaptive = fit_front(x);
    skm_data xdense = xd;
    xdense.flags &= ~SKM_FLAG_PRUNE;
    if (adaptive) SKM_TRY(tc_init_stats(b.a2.tc, st));
    SKM_TRY(tc_init_stats(b.a.tc, st));
    SKM_CUDA_TRY(cudaMemsetAsync(b.a.prune, 0, PRUNE_CTRS * sizeof(unsigned long long), st));
    int e = 0;
    if (x->repr == SKM_REPR_RBQ1) {
        SKM_CUDA_TRY(launch_rbq1_exponent(x->F, n, b.maxbits, b.e_dev, st));
        SKM_CUDA_TRY(cudaMemcpyAsync(&e, b.e_dev, sizeof(int), cudaMemcpyDeviceToHost, st));
        SKM_CUDA_TRY(cudaStreamSynchronize(st));
        xd.rbq1_exp = e;
    }
    if (x->repr == SKM_REPR_LVQ4) {
        SKM_CUDA_TRY(launch_lvq4_exponent(reinterpret_cast<const float4 *>(x->lvq), n, b.maxbits, b.e_dev, st));
        SKM_CUDA_TRY(cudaMemcpyAsync(&e, b.e_dev, sizeof(int), cudaMemcpyDeviceToHost, st));
        SKM_CUDA_TRY(cudaStreamSynchronize(st));
        xd.rbq1_exp = e;
    }
    // STEP 1: initial centroids (Forgy from cfg->seed when neither C_init
    // nor init_idx is given)
    std::vector<int64_t> seeded;
    if (!C_init && !init_idx) {
        seeded.resize(k);
        forgy_indices(cfg->seed, n, k, seeded.data());
        SKM_CUDA_TRY(cudaMemcpyAsync(b.init_idx, seeded.data(), sizeof(int64_t) * (size_t)k, cudaMemcpyHostToDevice,
                                     st));
        init_idx = b.init_idx;
    }
    SKM_CUDA_TRY(cudaMemsetAsync(b.status, 0, sizeof(int), st));
    SKM_CUDA_TRY(cudaMemsetAsync(b.u.flag, 0, sizeof(int32_t), st));
    if (C_init) {
        SKM_CUDA_TRY(cudaMemcpyAsync(C_out, C_init, centroid_bytes(x, k), cudaMemcpyDeviceToDevice,
                                     st));
    } else if (x->repr == SKM_REPR_RBQ1) {
        SKM_CUDA_TRY(launch_rbq1_decode_rows(static_cast<const uint32_t *>(x->x), x->F, n, d, x->m,
                                             e, init_idx, k, static_cast<float *>(C_out), b.status,
                                             st));
    } else if (x->repr == SKM_REPR_LVQ4) {
        SKM_CUDA_TRY(launch_lvq4_decode_rows(static_cast<const uint32_t *>(x->x),
                                             reinterpret_cast<const float4 *>(x->lvq), n, d, e, init_idx, k,
                                             static_cast<float *>(C_out), b.status, st));
    } else {
        const int eb = x->repr == SKM_REPR_SQ8 ? 1 : (x->repr == SKM_REPR_BF16 ? 2 : 4);
        if (x->repr == SKM_REPR_BF16)
            return set_error(SKM_ERR_INVALID_ARG, "BF16 fit needs fp32 C_init");
        SKM_CUDA_TRY(launch_gather_rows(x->x, n, eb, d, init_idx, k, C_out, b.status, st));
    }
    if (!C_init) {
        int bad = 0;
        SKM_CUDA_TRY(cudaMemcpyAsync(&bad, b.status, sizeof(int), cudaMemcpyDeviceToHost, st));
        SKM_CUDA_TRY(cudaStreamSynchronize(st));
        if (bad) return set_error(SKM_ERR_DEVICE_CHECK, "init_idx holds an index outside [0, n)");
    }
    float *dist = dist_out ? dist_out : b.dist;
    const int nblk = (int)std::min<int64_t>(RED_BLOCKS, n);
    int32_t *assign = assign_out;
    bool pruning = false;                 // adaptive: the pruned assignment is in use
    unsigned long long surv_seen = 0;     // adaptive: front survivors counted so far
    for (int it = 0; it <= cfg->iters; ++it) {
        const bool want_obj = objective_host != nullptr;
        float *dist_it = (want_obj || it == cfg->iters) ? dist : nullptr;
        if (adaptive && !pruning) {
            if (it > 0)
                SKM_CUDA_TRY(cudaMemcpyAsync(b.aprev, assign, sizeof(int32_t) * (size_t)n, cudaMemcpyDeviceToDevice,
                                             st));
            SKM_TRY(do_assign(&xdense, C_out, k, nullptr, assign, dist_it, b.a2, st));
            if (it > 0 && it < cfg->iters) {  // settled enough for pruning to pay?
                unsigned long long moved = 0;
                SKM_CUDA_TRY(cudaMemsetAsync(b.moved, 0, sizeof(moved), st));
                count_moved_kernel<<<(int)std::min<int64_t>(152 * 8, (n + 255) / 256), 256, 0, st>>>(assign, b.aprev,
                                                                                             n, b.moved);
                SKM_CUDA_TRY(launched());
                SKM_CUDA_TRY(cudaMemcpyAsync(&moved, b.moved, sizeof(moved), cudaMemcpyDeviceToHost, st));
                SKM_CUDA_TRY(cudaStreamSynchronize(st));
                pruning = (int64_t)moved * FIT_MOVED_DIV <= n;
            }
        } else {
            SKM_TRY(do_assign(&xd, C_out, k, it > 0 ? assign : nullptr, assign, dist_it, b.a, st));
            if (adaptive && it < cfg->iters) {  // still pruning well?
                unsigned long long surv = 0;
                SKM_CUDA_TRY(cudaMemcpyAsync(&surv, b.a.prune, sizeof(surv), cudaMemcpyDeviceToHost, st));
                SKM_CUDA_TRY(cudaStreamSynchronize(st));
                pruning = (double)(surv - surv_seen) <= FIT_MAX_SURVIVORS * (double)n;
                surv_seen = surv;
            }
        }
        if (want_obj) {
            SKM_CUDA_TRY(launch_sum_float_to_double(dist, n, b.partials, nblk, st));
            SKM_CUDA_TRY(launch_sum_double(b.partials, nblk, b.sum, st));
            SKM_CUDA_TRY(cudaMemcpyAsync(&objective_host[it], b.sum, sizeof(double),
                                         cudaMemcpyDeviceToHost, st));
        }
        if (it == cfg->iters) break;
        SKM_TRY(do_update(&xd, assign, k, C_out, b.counts, nullptr, e, b.u, st));
        if (stats_host && stats_host->empty_per_iter && it < EMPTY_LOG)
            SKM_CUDA_TRY(launch_count_zeros(b.counts, k, b.empty_iter + it, st));
        if (cfg->empty_policy == SKM_EMPTY_SPLIT)
            SKM_CUDA_TRY(launch_split_empty(C_out, x->repr == SKM_REPR_SQ8 ? 1 : 4, b.counts, k, x->d,
                                            b.u.wsplit, st));
    }
    if (fault_take(SKM_FAULT_STATUS)) SKM_CUDA_TRY(cudaMemsetAsync(b.status, 0xff, sizeof(int), st));
    {
        int bad = 0;
        SKM_CUDA_TRY(cudaMemcpyAsync(&bad, b.status, sizeof(int), cudaMemcpyDeviceToHost, st));
        SKM_CUDA_TRY(cudaStreamSynchronize(st));
        if (bad) return set_error(SKM_ERR_DEVICE_CHECK, "the device status word is set (%d)", bad);
    }
    skm_stats local;
    memset(&local, 0, sizeof(local));
    SKM_TRY(tc_read_stats(b.a.tc, &local, st));
    if (adaptive) {  // the dense screen's iterations
        skm_stats l2;
        memset(&l2, 0, sizeof(l2));
        SKM_TRY(tc_read_stats(b.a2.tc, &l2, st));
        local.rescored_rows += l2.rescored_rows;
        local.fallback_rows += l2.fallback_rows;
    }
    int32_t uflag = 0;
    SKM_CUDA_TRY(cudaMemcpy(&uflag, b.u.flag, sizeof(uflag), cudaMemcpyDeviceToHost));
    if (uflag) return set_error(SKM_ERR_TIMEOUT, "an update pipeline wait exceeded its limit");
    unsigned long long pr[PRUNE_CTRS] = {};
    SKM_CUDA_TRY(cudaMemcpy(pr, b.a.prune, sizeof(pr), cudaMemcpyDeviceToHost));
    prune_stats_from(pr, &local);
    if (stats_host) {
        int64_t *per_iter = stats_host->empty_per_iter;
        local.empty_per_iter = per_iter;
        *stats_host = local;
        std::vector<int64_t> cnt(k);
        if (cfg->iters > 0) {
            SKM_CUDA_TRY(cudaMemcpy(cnt.data(), b.counts, sizeof(int64_t) * k,
                                    cudaMemcpyDeviceToHost));
            for (int j = 0; j < k; ++j) stats_host->empty_clusters += cnt[j] == 0;
        }
        if (per_iter && cfg->iters > 0)
            SKM_CUDA_TRY(cudaMemcpy(per_iter, b.empty_iter, sizeof(int64_t) * (size_t)std::min(cfg->iters, EMPTY_LOG),
                                    cudaMemcpyDeviceToHost));
        // balance of the final assignment: the standard deviation of the sizes
        SKM_CUDA_TRY(launch_histogram(assign, n, k, b.u.counts32, st));
        std::vector<int32_t> sz(k);
        SKM_CUDA_TRY(cudaMemcpyAsync(sz.data(), b.u.counts32, sizeof(int32_t) * (size_t)k, cudaMemcpyDeviceToHost, st));
        SKM_CUDA_TRY(cudaStreamSynchronize(st));
        double mean = 0.0, var = 0.0;
        for (int j = 0; j < k; ++j) mean += sz[j];
        mean /= k;
        for (int j = 0; j < k; ++j) var += (sz[j] - mean) * (sz[j] - mean);
        stats_host->cluster_size_std = std::sqrt(var / k);
    }
    return SKM_OK;
}

int skm_split_empty(const skm_data *x, void *C_inout, const int64_t *counts, int k, void *ws,
                    size_t ws_bytes, void *stream) {
    SKM_TRY(check_data(x, false));
    if (!C_inout || !counts || k < 1) return set_error(SKM_ERR_INVALID_ARG, "bad arguments");
    Carver cv(ws, ws_bytes);
    int64_t *w = cv.take<int64_t>(k);
    SKM_TRY(need_ws(cv, ws_bytes, ws));
    SKM_CUDA_TRY(launch_split_empty(C_inout, x->repr == SKM_REPR_SQ8 ? 1 : 4, counts, k, x->d, w,
                                    S(stream)));
    return SKM_OK;
}

int skm_objective(const void *X, int x_is_bf16, int64_t n, int d, const float *C, int k,
                  const int32_t *assign, double *out_host, void *ws, size_t ws_bytes,
                  void *stream) {
    if (!X || !C || !assign || !out_host) return set_error(SKM_ERR_INVALID_ARG, "NULL pointer");
    if (n < 1 || d < 1 || d > MAX_D || k < 1) return set_error(SKM_ERR_INVALID_ARG, "bad shape");
    cudaStream_t st = S(stream);
    Carver cv(ws, ws_bytes);
    double *partials = cv.take<double>(RED_BLOCKS);
    double *sum = cv.take<double>(1);
    SKM_TRY(need_ws(cv, ws_bytes, ws));
    const int nblk = (int)std::min<int64_t>(RED_BLOCKS, n);
    SKM_CUDA_TRY(launch_objective(X, x_is_bf16, n, d, C, assign, partials, nblk, st));
    SKM_CUDA_TRY(launch_sum_double(partials, nblk, sum, st));
    SKM_CUDA_TRY(cudaMemcpyAsync(out_host, sum, sizeof(double), cudaMemcpyDeviceToHost, st));
    SKM_CUDA_TRY(cudaStreamSynchronize(st));
    return SKM_OK;
}

int skm_sq8_decode(const uint8_t *codes, int64_t n, int d, const float *b, const float *s,
                   float *Y, void *stream) {
    if (!codes || !b || !s || !Y || n < 1 || d < 1 || d > MAX_D)
        return set_error(SKM_ERR_INVALID_ARG, "bad arguments");
    SKM_CUDA_TRY(launch_sq8_decode(codes, n, d, b, s, Y, S(stream)));
    return SKM_OK;
}

}  // extern "C"

namespace skm {

// skm_lloyd_step_host's pruned ranges after the first: the tensor-core
// front's centroid side (operand, records, sort, the centroids' moves) was
// prepared by the first range's call this step, in its workspace ws0 planned
// for x0; only this range's rows are done here.  Anything else is a plain
// skm_assign.
int assign_range_shared(const skm_data *x, const void *C, int k, const int32_t *prev, int32_t *assign,
                        float *dist, void *ws, size_t ws_bytes, const skm_data *x0, void *ws0, size_t ws0_bytes,
                        cudaStream_t st) {
    SKM_TRY(check_data(x));
    SKM_TRY(check_k(x, k));
    if (!C || !assign) return set_error(SKM_ERR_INVALID_ARG, "C and assign are required");
    Carver cv(ws, ws_bytes);
    AssignBufs b;
    plan_assign(x, k, cv, b);
    SKM_TRY(need_ws(cv, ws_bytes, ws));
    Carver cv0(ws0, ws0_bytes);
    AssignBufs b0;
    plan_assign(x0, k, cv0, b0);
    SKM_TRY(need_ws(cv0, ws0_bytes, ws0));
    const bool front = use_prune(x) && prev && b.tc.pf_thr && b0.tc.pf_thr && x0->flags == x->flags &&
                       tc_pfront_ok(x->repr, x->d, x->x) && tc_pfront_ok(x0->repr, x0->d, x0->x) &&
                       x0->d == x->d && ((uintptr_t)C & 15) == 0;
    if (!front) return skm_assign(x, C, k, prev, assign, dist, ws, ws_bytes, st);
    SKM_CUDA_TRY(cudaMemsetAsync(b.prune, 0, PRUNE_CTRS * sizeof(unsigned long long), st));
    return tc_assign_pfront(x, static_cast<const float *>(C), k, prev, assign, dist, b.tc, b.prune, st, &b0.tc);
}

}  // namespace skm
