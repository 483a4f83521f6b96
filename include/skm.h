/*
 * skm.h -- C ABI of libskm, the GB300 (sm_103a) Lloyd k-means hot path for
 * clustering embeddings after dimensionality reduction, quantization or with
 * dimension pruning ("Stop Indexing at Full Precision: Revisiting Clustering
 * for Vector Embeddings", arxiv 2608.14648).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - Data pointers are DEVICE pointers owned by the caller, row-major and
 *    contiguous, unless an argument says "host".  The library never frees or
 *    retains a caller pointer after the call returns.
 *  - `stream` is a cudaStream_t passed as void* (NULL = the legacy default
 *    stream).  Calls are asynchronous on that stream unless documented
 *    otherwise; outputs are valid once the stream has reached the call.
 *  - Scratch memory: entry points that need it take `ws`/`ws_bytes`, a device
 *    buffer of at least skm_workspace_size(...) bytes, 256-byte aligned,
 *    owned by the caller and not used by anything else on other streams while
 *    the call's work is in flight.  The library itself never allocates device
 *    memory.
 *  - Return value: SKM_OK (0) or an skm_status error code.  Arguments are
 *    validated on the host BEFORE any launch; on an error nothing has been
 *    enqueued and outputs are untouched.  skm_last_error() returns a
 *    thread-local description of the last error.  No C++ exception crosses
 *    the ABI.
 *  - Distances are squared L2.  Ties in every argmin go to the LOWEST
 *    centroid index.
 *  - Limits: 1 <= d <= 4096, 1 <= k <= 65536, 1 <= n < 2^31 (RBQ1: n <= 2^24;
 *    LVQ4: n <= 2^26).
 */
#ifndef SKM_H
#define SKM_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes ------------------------------------------------------ */
typedef enum skm_status {
    SKM_OK = 0,
    SKM_ERR_INVALID_ARG = 1,  /* bad shape, null pointer, k > n, bad enum    */
    SKM_ERR_UNSUPPORTED = 2,  /* valid but outside the library's limits     */
    SKM_ERR_CUDA = 3,         /* a CUDA runtime/driver call failed            */
    SKM_ERR_NO_MEMORY = 4,    /* ws_bytes smaller than skm_workspace_size()  */
    SKM_ERR_TIMEOUT = 5,      /* a bounded device wait gave up               */
    SKM_ERR_DEVICE_CHECK = 6, /* a device-side check recorded a failure      */
    SKM_ERR_EXCHANGE = 7      /* a caller's exchange hook reported a failure */
} skm_status;

/* ---- representations of the points being clustered (Table 1) ---------- */
typedef enum skm_repr {
    SKM_REPR_F32 = 0,  /* float32 [n][d]                                    */
    SKM_REPR_SQ8 = 1,  /* uint8 SQ8 codes [n][d] (Section 3.1, per-dim b,s)  */
    SKM_REPR_RBQ1 = 2, /* RabitQ 1-bit codes uint32 [n][ceil(d/32)]
                          (bit j of word w = dimension 32w+j) + factors     */
    SKM_REPR_BF16 = 3, /* bfloat16 bit patterns uint16 [n][d] (projected
                          points stored in bf16), fp32 centroids            */
    SKM_REPR_LVQ4 = 4  /* LVQ 4-bit codes uint32 [n][ceil(d/8)] (dimension
                          8w+j in bits 4j..4j+3 of word w, unused nibbles
                          0) + per-point terms `lvq` (Section 3.1 "LVQ4")   */
} skm_repr;

typedef enum skm_dtype { SKM_DTYPE_F32 = 0, SKM_DTYPE_BF16 = 1 } skm_dtype;

/* skm_data.flags */
enum {
    /* F32 / BF16 / SQ8, d <= 1024: assign by exact dimension pruning on CUDA
     * cores (Section 3.1 "SuperKMeans", extended to SQ8 codes as the section
     * describes: partial distances over 32-dimension prefix blocks, a
     * centroid is dropped as soon as its partial distance exceeds the row's
     * current best) instead of the tensor-core path.  Same result (the fp32
     * nearest centroid; for SQ8 the exact integer code-space nearest, with
     * integer partial sums).
     * RBQ1, d <= 1024 (with d2 < d, skm_rbq1_segment_bounds): SuperKMeans'
     * checkpoints for RabitQ codes (Section 3.1): the estimate of Eq.
     * rabitq_l2 is split over the segments [0, d1), [d1, d2), [d2, d), each
     * with its own factors (x->seg_*, skm_rbq1_segments) and the centroid's
     * SQ4 code sums and ||rho_t||^2 per segment, evaluated per segment in the
     * fp32 order of skm_assign's RBQ1 estimate with fl(1/sqrt(d_t)); partial
     * estimates D1, D2 and D3 = D2 + est_2 (fp32 sums).  With beta = D3 of
     * the row's previous centroid (prev_assign; outside [0, k) or NULL:
     * centroid 0), a centroid other than that one is dropped at checkpoint t
     * when D_t > fl32(beta g_t), g_t = fl32((e_t / d) (1 + 2.1 / sqrt(e_t))^2)
     * (ADSampling's scaled test, e_1 = d1, e_2 = d2); the result is the
     * remaining centroid with the smallest D3, ties to the lowest index, and
     * dist receives that D3.  AND + popcount on CUDA cores. */
    SKM_FLAG_PRUNE = 1,
    /* RBQ1 only: symmetric 1-bit assignment -- every centroid is binarized
     * like a point (rho = c - m, bit = rho_i > 0) instead of SQ4-coded, and
     * the estimate of Eq. rabitq_l2 uses RabitQ's <o, q> ~ <obar, q>/<obar, o>
     * on both sides: <x - m, c - m> ~ F_x F_y (d - 2 h) / d with h the Hamming
     * distance (XOR + POPCOUNT) of the sign codes.  fp32 order: fy =
     * fl32((||rho||^2 / ||rho||_1) / sqrt(d)) per centroid (fp64, blocked
     * order), u = fy (d - 2 h), est = fma(-2 F, u, nx2 + ||rho||^2).  Tensor
     * cores (e4m3 +-1 codes on both sides) for d <= 1024, XOR + POPC beyond.
     * The update is unchanged (the points' fused decode-average). */
    SKM_FLAG_SYMMETRIC = 2,
    /* F32 / BF16 (tensor-core screen) only: the points and the workspace are
     * those of the previous skm_assign call on this workspace, as between
     * Lloyd iterations.  Each row decided by the screen leaves in the
     * workspace an upper bound U on s = ||c||^2 - 2 <x, c> for its centroid;
     * the next call grows it by that centroid's move (s(x, c') <= U + (||c'||^2
     * - ||c||^2) + 2 ||x|| ||c' - c||, both terms from the copy of the
     * previous centroids it keeps) and starts the row's threshold there, so
     * pairs far from the nearest are not listed as candidates.  The result
     * is the same; only the work changes.  A workspace whose last call had
     * other n, d or k, or did not finish, starts cold.  The caller must not
     * change the points between such calls, and a workspace first used with
     * this flag must be zero-filled (or come from a call on these points).
     * skm_fit uses it between its iterations (clearing it first).
     * BF16 with SKM_FLAG_PRUNE and the tensor-core front (see skm_assign): each
     * row keeps an upper bound U of its pruned distance to its centroid; the
     * next call grows it by the centroid's move, U' = (sqrt(U (1 + g)) +
     * ||c' - c||)^2 (1 + g) with g covering the fp32 rounding, and forms the
     * front's threshold from U' without reading the points.  Calls that want
     * distances use the exact seed distances instead. */
    SKM_FLAG_WARM = 4,
    /* With SKM_FLAG_PRUNE on BF16: no tensor-core front, the CUDA-core
     * pruning kernels only (the same result; for comparisons). */
    SKM_FLAG_PRUNE_CUDA_CORES = 8
};

/* Points being clustered.  Which fields are read depends on repr. */
typedef struct skm_data {
    int32_t repr;       /* skm_repr                                          */
    int32_t d;          /* dimensions                                        */
    int64_t n;          /* points                                            */
    const void *x;      /* the points / codes, layout per repr               */
    /* RBQ1 only (outputs of skm_quantize): per-point factors of Eq. rabitq_l2 */
    const float *nx2;   /* ||x_r - m||^2                 [n]                 */
    const float *F;     /* ||x_r - m|| / <xbar, x>       [n]                 */
    const int32_t *popx;/* number of set bits            [n]                 */
    const float *m;     /* centring mean m               [d]                 */
    int32_t rbq1_exp;   /* fixed-point exponent e of the decode-average
                           (RBQ1: skm_rbq1_exponent, LVQ4: skm_lvq4_exponent);
                           fit() computes it itself                          */
    int32_t flags;      /* SKM_FLAG_* (0 = defaults)                          */
    /* Optional screening copy for F32 / BF16 / SQ8 assignment, built once by
     * skm_screen_prep (the points never change across Lloyd iterations).
     * NULL: skm_assign builds it in its workspace on every call.            */
    const void *screen;
    /* LVQ4 only (output of skm_quantize): per point (s, b, N, A) of
     * Eq. final:lvq, float32 [n][4], 16-byte aligned                        */
    const float *lvq;
    /* RBQ1 with SKM_FLAG_PRUNE only (output of skm_rbq1_segments): per point
     * and dimension segment t = 0, 1, 2: ||r_t||^2, F_t, set bits, [n][3]   */
    const float *seg_nx2;
    const float *seg_F;
    const int32_t *seg_popx;
} skm_data;

/* Optional per-call statistics (host struct, filled after the call's work
 * completes only when the call synchronises, i.e. skm_fit). */
typedef struct skm_stats {
    int64_t rescored_rows;    /* F32/BF16: rows whose screen was not decisive */
    int64_t fallback_rows;    /* F32/BF16: rows rescanned over all k in fp32  */
    int64_t empty_clusters;   /* after the last update                         */
    int64_t prune_first_block;/* SKM_FLAG_PRUNE: (row, centroid) pairs alive
                                 after the first 32-dimension block (after the
                                 prune_front_dims dimensions when the
                                 tensor-core front ran)                        */
    int64_t prune_complete;   /* ... alive after the last block                 */
    double cluster_size_std;  /* population standard deviation of the k
                                 cluster sizes of the final assignment (the
                                 balance measure of the paper's Table 3)       */
    int64_t *empty_per_iter;  /* INPUT: host int64 array of min(iters, 4096)
                                 entries, or NULL; skm_fit writes the number of
                                 empty clusters after each update (before any
                                 split) of its first 4096 iterations           */
    int64_t prune_blocks;     /* SKM_FLAG_PRUNE on F32/BF16/SQ8: 32-dimension
                                 block partial sums evaluated after the first
                                 block (the executed work beyond the n k first
                                 blocks); 0 for RBQ1, whose checkpoints are
                                 counted by the two fields above.  With the
                                 tensor-core front: every block partial sum
                                 evaluated on CUDA cores (the front's work is
                                 n k prune_front_dims products)               */
    int64_t prune_front_dims; /* BF16 with SKM_FLAG_PRUNE and a seed
                                 assignment: dimensions screened on tensor
                                 cores for every pair (0: none)                */
    int64_t prune_rows_finished; /* ... rows whose 2 or more survivors were
                                 finished on CUDA cores (the rest were decided
                                 by the front, or:)                            */
    int64_t prune_rows_full;  /* ... rows pruned over all k on CUDA cores
                                 (more survivors than the front keeps)         */
} skm_stats;

const char *skm_last_error(void);

/* Kernel timer, for profiling callers (the paper has no counterpart).  With
 * skm_kernel_timer(1), CUDA events are recorded on the launch stream right
 * before and after every tensor-core kernel launch (assignment, projection);
 * skm_kernel_timer_ms waits for the later event and returns the time between
 * the two, i.e. the last such launch's duration.  0 disables it (no events
 * recorded).  Not for calls captured into a CUDA graph.  Errors:
 * SKM_ERR_CUDA (event creation), SKM_ERR_INVALID_ARG (NULL ms, or never
 * enabled). */
int skm_kernel_timer(int on);
int skm_kernel_timer_ms(float *ms);
int skm_version(void); /* major*10000 + minor*100 + patch */

/* Fault injection, for tests of the error paths (the paper has no
 * counterpart).  Arms `count` occurrences (0 disarms) of one fault, process
 * wide; each occurrence is used up by the first place that checks for it:
 *  SKM_FAULT_WORKSPACE  a workspace check reports SKM_ERR_NO_MEMORY, before
 *                       anything is enqueued;
 *  SKM_FAULT_LAUNCH     a kernel launch reports a launch failure: that kernel
 *                       still runs, the entry point enqueues nothing more and
 *                       returns SKM_ERR_CUDA;
 *  SKM_FAULT_STATUS     skm_fit's final read of its device status word finds
 *                       it set (the fault writes it on the device), so the
 *                       call returns SKM_ERR_DEVICE_CHECK;
 *  SKM_FAULT_WAIT       a tensor-core assignment launch starts with a 1 ms
 *                       bounded wait on a barrier that nothing arrives on: it
 *                       gives up before loading anything, raises its abort
 *                       flag, and skm_fit reports SKM_ERR_TIMEOUT.
 * The environment variable SKM_FAULT=workspace|launch|status|wait arms one
 * occurrence when the library first checks.  Nothing faults the GPU: every
 * injected failure is a status the host reads.  Returns SKM_OK, or
 * SKM_ERR_INVALID_ARG for an unknown kind or a negative count. */
enum { SKM_FAULT_WORKSPACE = 1, SKM_FAULT_LAUNCH = 2, SKM_FAULT_STATUS = 3, SKM_FAULT_WAIT = 4 };
int skm_inject_fault(int kind, int count);
int skm_fault_armed(int kind); /* occurrences left (0 for an unknown kind) */

/* Number of CUDA kernels this library has enqueued in this process so far
 * (host-side counter over all threads and devices; diagnostic only, e.g. to
 * count the kernels inside a timed region). */
uint64_t skm_kernel_launches(void);

/* Bytes of scratch needed by op for these points and k centroids.
 * op: 0 = skm_assign, 1 = skm_update, 2 = skm_fit, 3 = skm_quantize,
 *     4 = skm_pca_fit, 5 = skm_assign_segmented, 6 = skm_project on tensor
 *     cores in one pass (k = d_out), 7 = the smallest workspace skm_project
 *     takes for its tensor-core path (rows in chunks of 128).
 * Returns 0 with skm_last_error() set when the arguments are invalid. */
size_t skm_workspace_size(int op, const skm_data *x, int k);

/* ------------------------------------------------------------------------
 * Projection (Section 3.1: JLT / PCA; the random orthogonal rotation that
 * SuperKMeans and RabitQ require).  Y = (X - mean) P.
 *   X      float32 [n][d]
 *   mean   float32 [d] or NULL (no centring)
 *   P      float32 [d][d_out], row-major (column j = output direction j)
 *   Y      out_dtype [n][d_out]: SKM_DTYPE_F32 (float) or SKM_DTYPE_BF16
 *          (bf16 bit patterns, rounded half to even from the fp32 result)
 * fp32 accuracy.  d_out <= d.  With a workspace of at least
 * skm_workspace_size(6, x = {n, d}, k = d_out) bytes (or the smaller minimum
 * it reports as skm_workspace_size(7, ...), rows then go in chunks) the
 * product runs on the tensor cores: x - mean and P are split into three bf16
 * parts each (x = x1 + x2 + x3 exactly, each part the round-to-nearest bf16
 * of the remainder) and the six products with i + j <= 4 are accumulated in
 * fp32 (the three left out are below 2^-24 relative).  ws == NULL (or
 * smaller than the minimum): an fp32 CUDA-core tile GEMM.  Asynchronous. */
int skm_project(const float *X, int64_t n, int d, const float *mean, const float *P,
                int d_out, int out_dtype, void *Y, void *ws, size_t ws_bytes, void *stream);

/* Unprojection of centroids found in a projected space back to the original
 * space (Section 4, "Dimensionality Reduction and Vector Search", approach 2):
 * X = Y P^T + mean, Y float32 [n][d_out], P the projection matrix of
 * skm_project (float32 [d][d_out], row-major), mean float32[d] or NULL, X
 * float32 [n][d] (all device).  fp32 arithmetic; n <= 1,048,560 (centroids).
 * Approach 1 (full-dimensional centroids from the cluster membership) and the
 * raw-vector last update of RabitQ (Section 4, "Closing RabitQ's Gap in
 * Balance") are skm_update on the raw float32 points with the assignment.
 * Asynchronous. */
int skm_unproject(const float *Y, int64_t n, int d_out, const float *P, const float *mean, int d,
                  float *X, void *stream);

/* Host-to-device copy by the SMs: bytes bytes from src_host (host memory the
 * device can address: page-locked memory mapped into the device address space,
 * e.g. cudaHostAlloc or a pinned PyTorch tensor; on hardware-coherent host
 * links any host memory) to dst (device), loaded over the host link by a small
 * grid of thread blocks instead of a copy engine.  A copy-engine copy can wait
 * behind larger copies queued before it on the same engine; this call lets a
 * small input (a step's centroids) land while a large one (the next step's
 * points) is still streaming in.  The device address of src_host comes from
 * cudaHostGetDevicePointer: when that fails the call returns
 * SKM_ERR_INVALID_ARG and launches nothing.  bytes = 0 is a no-op.
 * Asynchronous on stream: src_host must stay valid until the copy is done. */
int skm_copy_from_host(void *dst, const void *src_host, size_t bytes, void *stream);

/* Randomized Hadamard rotation (a structured random orthogonal transform in
 * place of a dense random rotation before RabitQ / SuperKMeans, Section 3.1;
 * O(D log D) per point): Y = (1/sqrt(D)) H_D diag(sigma) [X - mean; 0] with
 * H_D the Sylvester Hadamard matrix (H_1 = 1, H_2m = [[H_m, H_m], [H_m, -H_m]]),
 * every row zero-padded from d to D dimensions.  D: power of two, max(32, d)
 * <= D <= 4096.  sigma: device float32[D] of +1/-1 (the random draw, supplied
 * by the caller); mean: device float32[d] or NULL.  Y (device): float32 or bf16
 * [n][D] (out_dtype, bf16 rounded to nearest even).  fp32 arithmetic.
 * Distances are preserved up to rounding.  Asynchronous. */
int skm_project_hadamard(const float *X, int64_t n, int d, const float *mean, const float *sigma,
                         int D, int out_dtype, void *Y, void *stream);

/* Forgy initialisation (Section 2.3 STEP 1: k points sampled at random),
 * HOST helper: idx_host[0..k) = positions 0..k-1 of a Fisher-Yates shuffle
 * of (0, 1, ..., n-1) in which position i = 0, 1, ..., k-1 swaps with
 * i + floor(r (n - i) / 2^64), r = w0 2^32 + w1 from (w0, w1, w2, w3) =
 * Philox4x32-10 of counter (i mod 2^32, i div 2^32, 0x466F7267, 0) under key
 * (seed mod 2^32, seed div 2^32) (Salmon et al., SC'11).  O(k) time and memory.
 * Requires 1 <= k <= n.  Synchronous, no GPU use. */
int skm_forgy_indices(uint64_t seed, int64_t n, int k, int64_t *idx_host);

/* Haar-random orthogonal d x d matrix (HOST helper, host output P_host[d][d],
 * float32 row-major): Householder QR of a Gaussian matrix drawn with
 * Philox4x32-10 + Box-Muller from `seed`, signs fixed so R has a positive
 * diagonal.  Synchronous, no GPU use. */
int skm_make_rotation(uint64_t seed, int d, float *P_host);

/* PCA fit (Section 3.1 "PCA"): mean and population covariance of X on the
 * GPU (fp32 products, fp64 accumulation), then a symmetric eigen-
 * decomposition on the host (fp64 Householder tridiagonalisation + implicit
 * QL).  Outputs (device): mean float32[d]; P float32 [d][d_out] whose columns
 * are the top-d_out eigenvectors by descending eigenvalue, each signed so its
 * largest-magnitude entry is positive; eigvals float32[d_out] (may be NULL).
 * Synchronises `stream` (the covariance is copied to the host). */
int skm_pca_fit(const float *X, int64_t n, int d, int d_out, float *mean, float *P,
                float *eigvals, void *ws, size_t ws_bytes, void *stream);

/* ------------------------------------------------------------------------
 * Quantization of the points before clustering (Section 3.1).
 *  repr = SKM_REPR_SQ8: per-dimension bias b_i = min over points and scale
 *    s_i = (max - b_i) / 255 (s_i = 1 for a flat dimension) when fit != 0,
 *    else the supplied b, s are used; code = clip(round((x - b)/s), 0, 255)
 *    in fp32, rounding half to even.  Outputs: codes uint8[n][d], b,s [d].
 *  repr = SKM_REPR_RBQ1 (RabitQ, 1-bit): mean m when fit != 0 (in exact
 *    fixed point, see skm_mean_from_sums: m_c = fl32(S_c / (n 2^s)) with
 *    S_c = sum of rint(x 2^s), s = skm_mean_scale(max |x|, n)), else the
 *    supplied m; r = x - m; bit i = (r_i > 0);
 *    nx2 = ||r||^2; F = sqrt(d) ||r||^2 / ||r||_1 (0 when r = 0), i.e.
 *    ||r|| / <xbar, x>; popx = set bits.  nx2 and F come from compensated
 *    fp32 sums: within about 5 x 2^-24 and 12 x 2^-24 relative of the exact
 *    values (the bits are exact).  Outputs: codes uint32[n][W],
 *    W = ceil(d/32), bit j of word w = dim 32w+j (unused high bits are 0);
 *    nx2, F float[n]; popx int32[n]; m float[d].
 *  repr = SKM_REPR_LVQ4 (Section 3.1 "LVQ4", per-vector): b = min_i x_i,
 *    s = (max_i x_i - b) / 15 in fp32 (s = 1 for a flat vector), code_i =
 *    clip(round((x_i - b) / s), 0, 15) in fp32, rounding half to even; with
 *    S = sum code_i and Q = sum code_i^2 the per-point terms of Eq. final:lvq
 *    are N = s s Q + 2 b s S + d b b and A = s S + d b, each evaluated in
 *    fp64 left to right and rounded once to fp32.  Outputs: codes uint32
 *    [n][ceil(d/8)] (nibbles, layout of SKM_REPR_LVQ4), lvq float [n][4] =
 *    (s, b, N, A).  No fitted parameters (fit is ignored).
 *  X float32 [n][d].  The x rows are assumed already rotated when RabitQ's
 *  random rotation is wanted (skm_project with skm_make_rotation's P).
 * ------------------------------------------------------------------------ */
typedef struct skm_quant_params {
    int32_t fit;   /* 1: fit b,s (SQ8) or m (RBQ1) from X; 0: use supplied  */
    int32_t bits;  /* SQ8 repr: 8 (or 0) for 8-bit codes, 4 for SQ4: 15 levels,
                      b = min, s = (max - b) / 15, one code 0..15 per byte; SQ4
                      codes then use every SQ8 entry point unchanged (the
                      code-domain distance and mean are the same definitions)  */
    float *b;      /* SQ8 bias  [d] (device; output when fit, else input)    */
    float *s;      /* SQ8 scale [d]                                          */
    float *m;      /* RBQ1 mean [d]                                          */
    float *nx2;    /* RBQ1 outputs [n]                                       */
    float *F;
    int32_t *popx;
    float *lvq;    /* LVQ4 output [n][4] (s, b, N, A), 16-byte aligned     */
} skm_quant_params;

int skm_quantize(int repr, const float *X, int64_t n, int d, skm_quant_params *qp,
                 void *codes, void *ws, size_t ws_bytes, void *stream);

/* The RabitQ dataset mean over row shards (one process per GPU), equal bit
 * for bit to the single-process mean of skm_quantize(SKM_REPR_RBQ1, fit):
 *  1. skm_column_absmax on each shard (device X float32 [n][d]; ws: device,
 *     >= 4 bytes; writes max |x| to *amax_host; synchronises); take the
 *     maximum over the shards;
 *  2. s = skm_mean_scale(global max, total rows) (host): with 2^(E-1) <=
 *     max |x| < 2^E and L = ceil(log2 n), s = 61 - L - E (0 when max = 0);
 *  3. skm_column_sums_fixed on each shard ADDS sums[c] += S_c, the sum over
 *     its rows of rint(x_rc 2^s) (round half to even; device int64 [d],
 *     zeroed by the caller); every term is below 2^(61-L) in magnitude, so the sums are
 *     exact integers and their order does not matter; sum S over the shards;
 *  4. skm_mean_from_sums: m_c = fl32(fl64(S_c) / (n 2^s)) (one fp64
 *     division, device float32 [d]).
 * The fixed point keeps |m - mean| below 2^-(s+1) (about 2^-38 for unit-norm
 * data and n = 10M).  Points must be finite.  Steps 3-4 are asynchronous. */
int skm_column_absmax(const float *X, int64_t n, int d, float *amax_host, void *ws, size_t ws_bytes,
                      void *stream);
int skm_mean_scale(float amax, int64_t n_total);
int skm_column_sums_fixed(const float *X, int64_t n, int d, int s, int64_t *sums, void *stream);
int skm_mean_from_sums(const int64_t *sums, int64_t n_total, int d, int s, float *m, void *stream);

/* SuperKMeans with RabitQ codes (SKM_FLAG_PRUNE on RBQ1): the dimension
 * segments [0, d1), [d1, d2), [d2, d) with d1 = 32 max(1, floor((d + 128) /
 * 256)) (12.5% of d in whole 32-dimension words) and d2 = 2 d1; returns
 * SKM_ERR_UNSUPPORTED when d2 >= d.  Host helper, no GPU use. */
int skm_rbq1_segment_bounds(int d, int *d1, int *d2);

/* Per point and segment t (r = x - m, the RabitQ mean): nx2s[n][3] =
 * ||r_t||^2, Fs[n][3] = sqrt(d_t) ||r_t||^2 / ||r_t||_1 (0 when r_t = 0), both
 * fp64 and rounded once, popxs[n][3] = the set bits of the segment's code
 * (device outputs; X float32 [n][d], m float32 [d] as given to
 * skm_quantize).  d <= 1024 with d2 < d.  Asynchronous. */
int skm_rbq1_segments(const float *X, int64_t n, int d, const float *m, float *nx2s, float *Fs, int32_t *popxs,
                      void *stream);

/* Fixed-point exponent e of the RBQ1 decode-average: e = 24 - ceil(log2 max F)
 * (0 when every F is 0), so round(F 2^e) <= 2^24 (the largest F keeps its
 * 24-bit precision) and the per-cluster sums of
 * up to 2^24 points are exact in int64.  Writes *e_host; synchronises. */
int skm_rbq1_exponent(const float *F, int64_t n, int *e_host, void *ws, size_t ws_bytes,
                      void *stream);

/* Fixed-point exponent e of the LVQ4 decode-average: with M = max over points
 * of max(s, |b|) (lvq: float [n][4] from skm_quantize), e = 31 - ceil(log2 M)
 * (0 when M = 0), so round(s 2^e) and |round(b 2^e)| are at most 2^31 and the
 * per-cluster sums of up to 2^26 points are exact in int64.  Writes *e_host;
 * synchronises. */
int skm_lvq4_exponent(const float *lvq, int64_t n, int *e_host, void *ws, size_t ws_bytes,
                      void *stream);

/* Screening copy of the points for the tensor-core assignment (opaque
 * layout): F32 -> bf16 copy + per-point (||x~||, ||x~ - x||); SQ8 -> centred
 * codes (code - 128) in bf16 + centred squared norms; BF16 -> per-point norms
 * (plus a padded copy when d is not a multiple of 8); RBQ1 / LVQ4 (d <= 1024)
 * -> the codes as e4m3 bytes.  skm_screen_bytes returns its size (0 when the
 * representation needs none: SQ8, RBQ1 or LVQ4 with d > 1024);
 * skm_screen_prep fills `screen` (device, 256-byte aligned,
 * caller-owned) from x->x.  Asynchronous.
 * RBQ1 / LVQ4 without a copy (x->screen NULL): when a code row is a multiple
 * of 16 bytes (ceil(d/32), resp. ceil(d/8), a multiple of 4) at a 16-byte
 * aligned address, the assignment reads the codes packed (each CTA expands
 * its point tiles into a slot of the workspace, at most 160 x 4 x 128 x
 * round16(d) bytes), so the points occupy their code words in HBM instead of
 * round16(d) bytes; the copy saves that per-tile expansion (measured on
 * GB300, 1M x 768, k = 1000: RBQ1 0.61 ms packed, 0.50 ms from the copy;
 * LVQ4 0.76 and 0.52 ms; at k = 3162 and d = 1024 the gap is 7-9%).
 * Otherwise skm_assign builds the copy in its workspace on every call. */
size_t skm_screen_bytes(const skm_data *x);
int skm_screen_prep(const skm_data *x, void *screen, size_t screen_bytes, void *stream);

/* ------------------------------------------------------------------------
 * Assignment, Section 2.3 STEP 2: assign[p] = argmin_j dist(x_p, c_j).
 *  C (device), per repr:
 *   F32  float [k][d] centroids.  Exact fp32 nearest centroid: a bf16
 *        tensor-core screen with a rigorous per-pair error bound, fp32
 *        rescoring (direct differences) of every centroid the bound cannot
 *        rule out, and an fp32 scan over all k for rows the screen could not
 *        narrow down.  dist = fp32 sum of squared differences.
 *   BF16 float [k][d] centroids against bf16 points (the projected points
 *        stored in bf16): the tensor-core screen as for F32 (the bf16
 *        points are the screen operand exactly), or, with SKM_FLAG_PRUNE,
 *        exact dimension pruning over 32-dimension prefix blocks.
 *   SQ8  uint8 [k][d] centroid codes; exact integer code-space distance
 *        sum (xbar_i - cbar_i)^2 (dist is that integer, as float).
 *   RBQ1 float [k][d] decoded centroids; per iteration each centroid is
 *        re-encoded with per-centroid SQ4 (b = min, s = (max-b)/15 of
 *        c - m; ny2 = ||c - m||^2 in fp64, pairwise inside 32-dimension
 *        blocks, blocks added in order) and the distance is the estimator
 *        of Eq. rabitq_l2 with
 *        Eq. final:rabitq, evaluated in fp32 in the order
 *          sd = s fl(1/sqrt d), bd = b fl(1/sqrt d)      (per centroid)
 *          u = fma(sd, 2P - sum ybar, bd (2 popx - d))
 *          dist = fma(-2 F, u, nx2 + ny2)
 *        where P = sum_i xbar_i ybar_i is an exact integer (tensor cores in
 *        e4m3 for d <= 1024, AND + popcount beyond).
 *   LVQ4 float [k][d] decoded centroids; per call each centroid is
 *        re-encoded with LVQ4 exactly as skm_quantize encodes a point
 *        (s_y, b_y, ybar, N_y; G_y = s_y sum ybar rounded once to fp32) and
 *        Eq. final:lvq is evaluated in fp32 in the order
 *          key = fma(b_y, -2 A_x, N_y)
 *          key = fma(G_y, -2 b_x, key)
 *          key = fma(-2 s_x, s_y * P, key)
 *        with P = sum_i xbar_i ybar_i an exact integer (tensor cores in
 *        e4m3 for d <= 1024, __dp4a beyond); the argmin is taken over key
 *        (N_x is the same for every centroid of a row) and dist = N_x + key.
 *  assign int32[n] (required); dist float[n] (may be NULL).
 *  prev_assign int32[n] or NULL: with SKM_FLAG_PRUNE, seeds each row's
 *  pruning bound with the distance to its previous centroid (entries outside
 *  [0, k) seed with centroid 0; results do not depend on it).  May alias
 *  `assign`.
 *  BF16 with SKM_FLAG_PRUNE, prev_assign given, 256 <= d <= 1024, d % 8 == 0
 *  and x 16-byte aligned: the first 128 dimensions of every pair are screened
 *  on tensor cores (Section 3.1 "SuperKMeans": a GEMM over the front
 *  dimensions).  A rigorous lower bound of each pair's pruned distance from
 *  the bf16 product drops the pairs that cannot beat the seed's distance; a
 *  row whose one survivor is its seed is decided there, rows with 2..128
 *  survivors finish on CUDA cores with the same block sums, rows with more
 *  are pruned over all k.  The result is the same as without the front, bit
 *  for bit (assignments and distances); the workspace then holds about
 *  280 bytes per point (the survivor lists).
 * ------------------------------------------------------------------------ */
int skm_assign(const skm_data *x, const void *C, int k, const int32_t *prev_assign,
               int32_t *assign, float *dist, void *ws, size_t ws_bytes, void *stream);

/* Pruning counters of the last skm_assign call with SKM_FLAG_PRUNE that ran
 * on workspace `ws` (Section 3.1 "SuperKMeans": the work the bounds skipped).
 * skm_assign zeroes them at the start of such a call.  Fills
 * prune_first_block, prune_complete and prune_blocks of *out (the other
 * fields are zero); for RBQ1 the first two count the pairs alive after the
 * 12.5% and 25% checkpoints.  Synchronises `stream` (the caller's device
 * pointer `ws`, at least the size skm_workspace_size returned for that call).
 * Errors: SKM_ERR_INVALID_ARG (NULL ws or out, ws_bytes too small for the
 * counters), SKM_ERR_CUDA. */
int skm_assign_prune_stats(const void *ws, size_t ws_bytes, skm_stats *out, void *stream);

/* RBQ1 assignment that allocates nothing.  The paper has no counterpart:
 * this entry point exists for callers that cannot allocate device memory
 * (code inside a host engine that owns all device memory through its own pool
 * or budget, or a latency-critical path where cudaMalloc/cudaFree and their
 * possible device-wide synchronisation are not acceptable).  Same inputs,
 * outputs and results as skm_assign with x->repr == SKM_REPR_RBQ1; the
 * per-centroid scratch (SQ4 bit planes and estimator terms) lives in one
 * file-scope device array of 2.25 MiB that every GPU which loads the
 * library keeps until exit.
 *   Limits: k <= 16384 and k * ceil(d/32) <= 131072, else SKM_ERR_UNSUPPORTED
 *   (nothing is launched).
 *   Every call looks up the array's device address in the current context
 *   (cudaGetSymbolAddress, which allocates nothing), so the entry point stays
 *   valid when that context is destroyed and recreated (cudaDeviceReset); the
 *   first call on a device may load the library's module, so make it before
 *   any stream capture.
 *   All calls share the array and it keeps the last call's contents: calls
 *   whose work overlaps on the GPU (other streams, other threads) race; order
 *   them on one stream or synchronise between them.
 *   No cudaMalloc, cudaFree or allocating library call is made. */
int skm_assign_rbq1_noalloc(const skm_data *x, const float *C, int k, int32_t *assign, float *dist,
                            void *stream);

/* Segmented assignment (the FINE-CLUSTERING phase of hierarchical k-means):
 * the rows of x are sorted by group (group[n] non-decreasing, device int32 in
 * [0, nseg)); row r takes the nearest of the centroids [base[g], base[g+1])
 * of its group g = group[r] only (base: device int32[nseg + 1], base[0] = 0,
 * non-decreasing, base[nseg] <= k, every group referenced by a row non-empty),
 * with the same per-representation rules as skm_assign (F32/BF16 exact fp32
 * argmin; SQ8, RBQ1 and LVQ4 bit-exact), ties to the lowest index.
 * Tensor-core paths only: SQ8, RBQ1 and LVQ4 need d <= 1024; no pruning flag.  Group ids
 * outside [0, nseg) are clamped (never an out-of-bounds access); unsorted
 * groups give undefined assignments.  Workspace: skm_workspace_size(5, x, k).
 * Asynchronous. */
int skm_assign_segmented(const skm_data *x, const void *C, int k, const int32_t *group,
                         const int32_t *base, int nseg, int32_t *assign, float *dist, void *ws,
                         size_t ws_bytes, void *stream);

/* ------------------------------------------------------------------------
 * Update, Section 2.3 STEP 3 (and the quantized-domain variants of 3.1).
 *  C_inout (device), per repr as in skm_assign; clusters with no member keep
 *  their centroid.  counts int64[k] (device, output).
 *   F32/BF16  c_j = mean of members (fp32 sums per cluster)
 *   SQ8       cbar_j = round-half-even(sum of member codes / count), exact
 *   RBQ1      fused decode-average: c_ji = m_i + (2 T_ji - U_j) f_j in fp64,
 *             rounded to fp32, with f_j = (fl(1/sqrt(d)) 2^-e) / count_j, where
 *             T_ji = sum Fq xbar_i, U_j = sum Fq, Fq = round(F 2^e) (int64,
 *             exact), e = x->rbq1_exp.
 *   LVQ4      fused decode-average (Section 3.1 "LVQ4"): c_ji = (T_ji +
 *             U_j) f_j in fp64, rounded to fp32, f_j = 2^-e / count_j, where
 *             T_ji = sum Sq xbar_i, U_j = sum Bq, Sq = round(s 2^e),
 *             Bq = round(b 2^e) (int64, exact), e = x->rbq1_exp.
 *  Assignments outside [0, k) are skipped (not counted, not summed).
 *  partial != NULL selects the sharded form: nothing is finalised; the
 *  cluster sums are ADDED into `partial` and the member counts into
 *  `counts` (both zeroed by the caller before the first shard) so that
 *  shards can be merged (skm_merge_partials) and finalised
 *  (skm_update_finalize).  partial layout: F32/BF16 double[k][d];
 *  SQ8 int64[k][d]; RBQ1 and LVQ4 int64[k][d+1] (T then U).
 * ------------------------------------------------------------------------ */
int skm_update(const skm_data *x, const int32_t *assign, int k, void *C_inout,
               int64_t *counts, void *partial, void *ws, size_t ws_bytes, void *stream);

/* dst += src over `count` elements of the partial layout (elem_type 0 =
 * double, 1 = int64); device pointers. */
int skm_merge_partials(void *dst, const void *src, int64_t count, int elem_type, void *stream);

/* Finalise merged partial sums into centroids (same rules as skm_update). */
int skm_update_finalize(const skm_data *x, const void *partial, const int64_t *counts,
                        int k, void *C_inout, void *stream);

/* ------------------------------------------------------------------------
 * Lloyd k-means, Section 2.3: `iters` x (STEP 2 assign, STEP 3 update), then
 * STEP 2 once more for the final assignment.
 *  cfg->iters >= 0.  Initial centroids: C_init (device, per-repr layout of
 *  skm_assign) when non-NULL, else the points init_idx[0..k) (device int64,
 *  Forgy, STEP 1): F32 rows, SQ8 codes, RBQ1 / LVQ4 decoded points (the
 *  decode-average of one member); when init_idx is NULL too, the points
 *  skm_forgy_indices(cfg->seed, n, k) (drawn on the host, copied to the
 *  workspace).  BF16 points need C_init (fp32 centroids).
 *  An init_idx entry outside [0, n) makes the call fail with
 *  SKM_ERR_DEVICE_CHECK before any iteration; a tensor-core pipeline wait
 *  that exceeds its 2 s limit makes it return SKM_ERR_TIMEOUT.
 *  Outputs (device): C_out (per-repr layout), assign_out int32[n],
 *  dist_out float[n] or NULL (from the final assignment).
 *  objective_host (host, iters+1 doubles, may be NULL): sum of the
 *  assignment's dist at each STEP 2 (fp64 sum of the per-row values).
 *  stats_host may be NULL.  Synchronises `stream` before returning.
 * ------------------------------------------------------------------------ */
typedef struct skm_fit_config {
    int32_t k;
    int32_t iters;
    int32_t empty_policy;  /* SKM_EMPTY_KEEP (0) or SKM_EMPTY_SPLIT (1), below */
    int32_t reserved0;
    uint64_t seed;         /* Forgy seed, used when C_init and init_idx are NULL */
    int32_t reserved[2];
} skm_fit_config;

/* Empty clusters after an update (Section 2.3 STEP 3: splitting large clusters
 * helps).  SKM_EMPTY_KEEP: an empty cluster keeps its centroid.
 * SKM_EMPTY_SPLIT: after every update of skm_fit, skm_split_empty below. */
enum { SKM_EMPTY_KEEP = 0, SKM_EMPTY_SPLIT = 1 };

int skm_fit(const skm_fit_config *cfg, const skm_data *x, const void *C_init,
            const int64_t *init_idx, void *C_out, int32_t *assign_out, float *dist_out,
            double *objective_host, skm_stats *stats_host, void *ws, size_t ws_bytes,
            void *stream);

/* ------------------------------------------------------------------------
 * One Lloyd iteration (Section 2.3: STEP 2 then STEP 3) of points held in
 * HOST memory, for callers whose points do not stay on the GPU: the points
 * cross the host link once per iteration, so the call overlaps that copy with
 * the work.  The rows are cut into cfg->chunks ranges of ceil(n / chunks)
 * rows; range i is copied to the device on cfg->copy_stream into one of three
 * range buffers of the workspace while `stream` assigns earlier ranges
 * (skm_assign on a device view of the range) and adds their cluster sums into
 * partial sums (skm_update's sharded form); a buffer is refilled once its
 * range's assignments have been sent back.  Then cfg->exchange (if set) runs,
 * the partial sums are finalised (skm_update_finalize) and the centroids are
 * copied back.
 *  x: a HOST view of the points: repr F32, BF16 or SQ8, flags 0, screen NULL,
 *     x->x in page-locked host memory (cudaHostAlloc, cudaHostRegister or a
 *     pinned PyTorch tensor), else SKM_ERR_INVALID_ARG before any work.
 *  C_host (host): the centroids this iteration assigns to (per-repr layout
 *     of skm_assign); C_host_out (host, may equal C_host): the updated
 *     centroids; assign_host (host int32[n]): the assignments of STEP 2;
 *     counts_host (host int64[k] or NULL): member counts; objective_host
 *     (host double or NULL): fp64 sum of the STEP 2 distances.
 *  cfg->copy_stream: cudaStream_t of the host-to-device copies (NULL: they go
 *     on `stream`, without overlap).
 *  cfg->partial / cfg->counts: device buffers for the partial sums (double
 *     [k][d], int64 [k][d] for SQ8) and member counts (int64 [k]); NULL: taken
 *     from the workspace.
 *  cfg->exchange: NULL, or a host function called once all ranges are
 *     summed with (partial, counts, cfg->user, stream) and enqueued work on
 *     `stream` before it returns (a multi-process caller all-reduces the
 *     partial sums and counts there: the path's one exchange per iteration);
 *     a non-zero return ends the call with SKM_ERR_EXCHANGE.
 *  ws: device workspace of skm_step_host_workspace_size(cfg, x) bytes (0 when
 *     the arguments are invalid), 256-byte aligned.
 * Synchronous: returns once the outputs are in host memory (both streams
 * synchronised).  Results equal skm_assign followed by skm_update with
 * partial sums and skm_update_finalize on the same points.
 * ------------------------------------------------------------------------ */
typedef int (*skm_exchange_fn)(void *partial, int64_t *counts, void *user, void *stream);
typedef struct skm_step_host_config {
    int32_t k;
    int32_t chunks;         /* row ranges, 1..256                              */
    void *copy_stream;
    void *partial;
    int64_t *counts;
    skm_exchange_fn exchange;
    void *user;
    int32_t warm;           /* F32 / BF16: 1 when x's host points are those of
                               the previous call with this workspace and
                               configuration (Lloyd iterations): each range
                               keeps its own assignment workspace and its
                               screen starts from the bounds that range's
                               previous call left (SKM_FLAG_WARM); the
                               workspace then holds one assignment workspace
                               per range.  0: every call starts cold.        */
    int32_t prune;          /* BF16 with warm = 1: each range's assignment is
                               the exact pruned one (SKM_FLAG_PRUNE, the
                               tensor-core front), seeded with the previous
                               call's assignments, which assign_host must
                               hold on entry (the caller passes the array
                               back unchanged; the first call's seeds decide
                               only its work).  The range's seeds are copied
                               in with its points.  The front's centroid
                               side (operand, records, sort, the centroids'
                               moves) is prepared once a call, by the first
                               range, and reused by the others; each range's
                               kept bounds apply only if taken against the
                               previous centroids that preparation started
                               from (else that range starts cold).           */
    int32_t reserved[2];
} skm_step_host_config;

size_t skm_step_host_workspace_size(const skm_step_host_config *cfg, const skm_data *x);
int skm_lloyd_step_host(const skm_step_host_config *cfg, const skm_data *x, const void *C_host,
                        void *C_host_out, int32_t *assign_host, int64_t *counts_host,
                        double *objective_host, void *ws, size_t ws_bytes, void *stream);

/* ------------------------------------------------------------------------
 * Hierarchical k-means (Section 4, "Other Accelerators": Hierarchical k-Means): MESO-CLUSTERING
 * of all points into m clusters (Lloyd, `meso_iters` iterations, Forgy
 * initial centroids meso_init_idx[0..m), device int64), then FINE-CLUSTERING
 * inside every meso cluster at once: meso cluster i gets k_i of the k fine
 * clusters, k apportioned by the meso sizes n_i (floor of k n_i / N, the
 * rest to the largest remainders k n_i mod N, ties to the lower index; a
 * non-empty meso cluster left with none takes one from the one with the
 * most; the paper states sqrt(n_i) per meso cluster, this keeps the total at
 * k), initial fine centroids the members at positions floor(t n_i / k_i),
 * t < k_i, in increasing point order, and `fine_iters` Lloyd iterations in
 * which a point only takes its own meso cluster's fine centroids, then a
 * final such assignment.  refine != 0 adds the optional vanilla iteration
 * over all points and all k centroids, then a final vanilla assignment.
 * Fine centroids of meso cluster i are rows sum_{j<i} k_j .. + k_i - 1.
 *  Representations: F32, SQ8, RBQ1 and LVQ4 (SQ8 / RBQ1 / LVQ4 with
 *  d <= 1024); no pruning flag.  m <= min(k, 12288); k <= n.
 *  Outputs (device): C_out (k rows, per-repr layout of skm_assign),
 *  assign_out int32[n]; optional meso_assign_out int32[n] (device) and
 *  fine_counts_host int32[m] (host); stats_host may be NULL.
 *  Workspace: skm_hier_workspace_size (it holds a copy of the points in meso
 *  order).  Synchronises `stream`. */
typedef struct skm_hier_config {
    int32_t k;
    int32_t m;
    int32_t meso_iters;
    int32_t fine_iters;
    int32_t refine;
    int32_t reserved[3];
} skm_hier_config;

size_t skm_hier_workspace_size(const skm_hier_config *cfg, const skm_data *x);
int skm_fit_hierarchical(const skm_hier_config *cfg, const skm_data *x, const int64_t *meso_init_idx,
                         void *C_out, int32_t *assign_out, int32_t *meso_assign_out,
                         int32_t *fine_counts_host, skm_stats *stats_host, void *ws, size_t ws_bytes,
                         void *stream);

/* Split large clusters into the empty ones (the library's reading of
 * Section 2.3 STEP 3).  Clusters with counts[j] == 0, in increasing j, each
 * take the current largest cluster L (most members, ties to the lowest
 * index; nothing more happens once L has fewer than 2 members): both become
 * L's centroid moved by a relative step of 2^-10 in opposite directions,
 * +eps on even and -eps on odd dimensions for j (the reverse for L), one
 * rounded fp32 multiply per element (F32/BF16/RBQ1/LVQ4 centroids float32[k][d]);
 * SQ8 code centroids move by one code step instead (clipped to [0, 255]).
 * L then counts as ceil(n_L / 2) members and j as floor(n_L / 2) for later
 * choices; `counts` (device int64[k], from skm_update) is not modified.
 * ws: device workspace of at least 8 k + 256 bytes.  Asynchronous. */
int skm_split_empty(const skm_data *x, void *C_inout, const int64_t *counts, int k, void *ws,
                    size_t ws_bytes, void *stream);

/* Objective helpers (reporting, Section 4 WCSS): fp64 sum over n of
 * ||x_p - c_{a_p}||^2 with x float32 [n][d] (or bf16 bits when x_is_bf16)
 * and C float32 [k][d].  Writes *out_host; synchronises. */
int skm_objective(const void *X, int x_is_bf16, int64_t n, int d, const float *C, int k,
                  const int32_t *assign, double *out_host, void *ws, size_t ws_bytes,
                  void *stream);

/* SQ8 reconstruction x ~ code * s + b (fp32): codes uint8[n][d] -> Y float[n][d]. */
int skm_sq8_decode(const uint8_t *codes, int64_t n, int d, const float *b, const float *s,
                   float *Y, void *stream);

#ifdef __cplusplus
}
#endif
#endif /* SKM_H */
