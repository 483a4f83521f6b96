// Exact dimension pruning (Section 3.1 "SuperKMeans": partial distances over
// prefix blocks of the projected dimensions; a centroid is dropped once its
// partial distance exceeds the row's current best).  CUDA cores, fp32 (points
// fp32 or bf16, centroids fp32) or exact integers (SQ8 codes).
//
// One warp per point row.  The bound beta starts at the exact distance to a
// seed centroid (the previous assignment when given, else centroid 0).
// Centroids are taken 256 at a time: lane l computes the first 32-dimension
// block of centroid c0 + 32 s + l, the survivors (partial <= beta * slack) are
// compacted into a shared-memory queue with __ballot_sync / __popc, and each
// further block re-filters the queue the same way.  Candidates that complete
// all blocks carry their full distance; the warp keeps the smallest (ties to
// the lowest index).  Partial sums only grow block by block and every term is
// non-negative, so dropping a centroid whose partial already exceeds beta
// never drops the nearest one; `slack` covers the fp32 rounding of the sums,
// so the result is the exact fp32 argmin whatever the seed.
#include <climits>

#include "skm_internal.cuh"

namespace skm {
namespace {

constexpr int PR_WARPS = 4;  // 32 KiB of static shared memory per block
constexpr int PR_BATCH = 256;
constexpr int PR_MAX_D = 1024;

template <typename TX>
__device__ __forceinline__ float ldx(const TX *p);
template <>
__device__ __forceinline__ float ldx<float>(const float *p) {
    return __ldg(p);
}
template <>
__device__ __forceinline__ float ldx<uint16_t>(const uint16_t *p) {
    return __uint_as_float(((uint32_t)__ldg(p)) << 16);
}

// sum over dims [32b, min(32b + 32, d)) of (x_i - c_i)^2, in increasing i
__device__ __forceinline__ float block_partial(const float *sx, const float *c, int d, int b) {
    float s = 0.0f;
    const int i0 = 32 * b;
    if (i0 + 32 <= d && (d % 4) == 0) {
        const float4 *c4 = reinterpret_cast<const float4 *>(c + i0);
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            const float4 cv = __ldg(c4 + q);
            float t = __fsub_rn(sx[i0 + 4 * q], cv.x);
            s = __fmaf_rn(t, t, s);
            t = __fsub_rn(sx[i0 + 4 * q + 1], cv.y);
            s = __fmaf_rn(t, t, s);
            t = __fsub_rn(sx[i0 + 4 * q + 2], cv.z);
            s = __fmaf_rn(t, t, s);
            t = __fsub_rn(sx[i0 + 4 * q + 3], cv.w);
            s = __fmaf_rn(t, t, s);
        }
    } else {
        const int i1 = min(d, i0 + 32);
        for (int i = i0; i < i1; ++i) {
            const float t = __fsub_rn(sx[i], __ldg(c + i));
            s = __fmaf_rn(t, t, s);
        }
    }
    return s;
}

// Coalesced gather of 32 (centroid, block) pairs, one per lane: the warp
// copies pair p's block (row j_p of C, dims [32 b_p, min(32 b_p + 32, d)))
// to stg + p * STG_LD with 16-byte cp.async copies (no registers held, eight
// in flight a lane), eight lanes per 128-byte block, so one instruction
// touches four lines instead of one line per lane; each lane then reads its
// own block from shared memory (rows 144 bytes apart: the eight lanes of a
// 16-byte access phase hit distinct banks).  Needs d % 4 == 0, C 16-byte
// aligned and k d <= 2^26.  Lanes with `valid` false stage nothing.
constexpr int STG_LD = 36;
__device__ __forceinline__ void stage_blocks(float *stg, const float *__restrict__ C, int d, int j, int b,
                                             bool valid) {
    const int lane = threadIdx.x & 31, q = lane & 7;
    // (element offset of the block) * 16 + its length in float4s
    const int key = valid ? (j * d + 32 * b) * 16 + (min(32, d - 32 * b) >> 2) : 0;
    const uint32_t s0 = (uint32_t)__cvta_generic_to_shared(stg) + 16u * q;
    __syncwarp();  // every lane has read the previous pairs
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const int p = 4 * i + (lane >> 3);
        const int kp = __shfl_sync(0xffffffffu, key, p);
        if (q < (kp & 15))
            asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(s0 + (uint32_t)(p * STG_LD * 4)),
                         "l"(C + (kp >> 4) + 4 * q)
                         : "memory");
    }
    asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
    __syncwarp();
}
// block_partial with the centroid block from shared memory (stage_blocks):
// the same terms in the same order, so the same value
__device__ __forceinline__ float block_partial_staged(const float *sx, const float *cb, int d, int b) {
    float s = 0.0f;
    const int i0 = 32 * b;
    if (i0 + 32 <= d) {
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            const float4 cv = reinterpret_cast<const float4 *>(cb)[q];
            float t = __fsub_rn(sx[i0 + 4 * q], cv.x);
            s = __fmaf_rn(t, t, s);
            t = __fsub_rn(sx[i0 + 4 * q + 1], cv.y);
            s = __fmaf_rn(t, t, s);
            t = __fsub_rn(sx[i0 + 4 * q + 2], cv.z);
            s = __fmaf_rn(t, t, s);
            t = __fsub_rn(sx[i0 + 4 * q + 3], cv.w);
            s = __fmaf_rn(t, t, s);
        }
    } else {
        for (int i = i0; i < d; ++i) {
            const float t = __fsub_rn(sx[i], cb[i - i0]);
            s = __fmaf_rn(t, t, s);
        }
    }
    return s;
}

// One warp prunes the centroid batches [c0, c0 + PR_BATCH) for c0 = c_first,
// c_first + c_step, ... below k against its running bound (beta, best): per
// batch, lane l takes the first block of centroids c0 + 32 s + l, the
// survivors (partial <= beta * slack) are compacted into the warp's queue
// with __ballot_sync / __popc, each further block re-filters the queue the
// same way, and the complete candidates' full distances update the bound
// (ties to the lowest index).  qid / qps: the warp's two queues.
template <bool STAGED = false>
__device__ __forceinline__ void prune_batches(const float *sx, const float *__restrict__ C, int d, int k, int c_first,
                                              int c_step, float slack, float &beta, int &best,
                                              int (&qid)[2][PR_BATCH], float (&qps)[2][PR_BATCH],
                                              unsigned long long &first_alive, unsigned long long &complete,
                                              unsigned long long &later, float *stg = nullptr) {
    const int lane = threadIdx.x & 31;
    // STAGED: blocks gathered coalesced into stg, the warp's stage_blocks buffer
    auto partial = [&](int j, int b, bool valid) {
        if constexpr (STAGED) {
            stage_blocks(stg, C, d, j, b, valid);
            return block_partial_staged(sx, stg + lane * STG_LD, d, b);
        }
        return valid ? block_partial(sx, C + (int64_t)j * d, d, b) : 0.0f;  // no load past k
    };
    const unsigned lt = (1u << lane) - 1u;
    const int nb = (d + 31) >> 5;
    for (int c0 = c_first; c0 < k; c0 += c_step) {
        __syncwarp();  // queue 0 may still be read by the previous batch
        // first block over the whole batch, survivors compacted into queue 0
        int cnt = 0;
        for (int s = 0; s < PR_BATCH / 32; ++s) {
            const int j = c0 + 32 * s + lane;
            float p = partial(j, 0, j < k);
            if (j >= k) p = INFINITY;
            const bool alive = p <= beta * slack;
            const unsigned m = __ballot_sync(0xffffffffu, alive);
            if (alive) {
                const int pos = cnt + __popc(m & lt);
                qid[0][pos] = j;
                qps[0][pos] = p;
            }
            cnt += __popc(m);
        }
        first_alive += cnt;
        int src = 0;
        for (int b = 1; b < nb && cnt > 0; ++b) {
            __syncwarp();
            later += cnt;
            int ncnt = 0;
            for (int t0 = 0; t0 < cnt; t0 += 32) {
                const int t = t0 + lane;
                const bool valid = t < cnt;
                const int j = valid ? qid[src][t] : 0;
                const float pb = partial(j, b, valid);
                const float p = valid ? qps[src][t] + pb : INFINITY;
                const bool alive = valid && p <= beta * slack;
                const unsigned m = __ballot_sync(0xffffffffu, alive);
                if (alive) {
                    const int pos = ncnt + __popc(m & lt);
                    qid[src ^ 1][pos] = j;
                    qps[src ^ 1][pos] = p;
                }
                ncnt += __popc(m);
            }
            cnt = ncnt;
            src ^= 1;
        }
        __syncwarp();
        complete += cnt;
        // complete candidates: full distances; keep the smallest (lowest index on ties)
        for (int t0 = 0; t0 < cnt; t0 += 32) {
            const int t = t0 + lane;
            float p = INFINITY;
            int j = 0x7fffffff;
            if (t < cnt) {
                p = qps[src][t];
                j = qid[src][t];
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                const float op = __shfl_xor_sync(0xffffffffu, p, o);
                const int oj = __shfl_xor_sync(0xffffffffu, j, o);
                if (op < p || (op == p && oj < j)) {
                    p = op;
                    j = oj;
                }
            }
            if (p < beta || (p == beta && j < best)) {
                beta = p;
                best = j;
            }
        }
    }
}

// relative rounding of a d-term fp32 sum of non-negative terms is below
// d * 2^-24; keep anything within twice that of beta
__device__ __forceinline__ float prune_slack(int d) { return 1.0f + 2.0f * (float)(d + 1) * 0x1p-24f; }

template <typename TX, bool STG>
__global__ void __launch_bounds__(PR_WARPS * 32) prune_assign_kernel(
    const TX *__restrict__ X, int64_t n, int d, const float *__restrict__ C, int k,
    const int32_t *__restrict__ prev, int32_t *__restrict__ assign, float *__restrict__ dist,
    unsigned long long *__restrict__ counters) {
    __shared__ float sx_all[PR_WARPS][PR_MAX_D];
    __shared__ int qid[PR_WARPS][2][PR_BATCH];
    __shared__ float qps[PR_WARPS][2][PR_BATCH];
    extern __shared__ __align__(16) float pa_stg[];  // STG: per warp 32 x STG_LD floats (stage_blocks)
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    float *sx = sx_all[warp];
    const int nb = (d + 31) >> 5;
    const float slack = prune_slack(d);
    const int64_t nw = (int64_t)gridDim.x * PR_WARPS;
    unsigned long long first_alive = 0, complete = 0, later = 0;
    for (int64_t row = (int64_t)blockIdx.x * PR_WARPS + warp; row < n; row += nw) {
        __syncwarp();
        for (int i = lane; i < d; i += 32) sx[i] = ldx<TX>(X + row * d + i);
        __syncwarp();
        int best = prev ? prev[row] : 0;
        if (best < 0 || best >= k) best = 0;
        float beta = 0.0f;
        for (int b = 0; b < nb; ++b) beta += block_partial(sx, C + (int64_t)best * d, d, b);
        prune_batches<STG>(sx, C, d, k, 0, PR_BATCH, slack, beta, best, qid[warp], qps[warp], first_alive, complete,
                           later, STG ? pa_stg + warp * 32 * STG_LD : nullptr);
        if (lane == 0) {
            assign[row] = best;
            if (dist) dist[row] = beta;
        }
    }
    if (counters && lane == 0) {
        atomicAdd(&counters[0], first_alive);
        atomicAdd(&counters[1], complete);
        atomicAdd(&counters[2], later);
    }
}

// The same pruning for a list of rows (those the tensor-core front could
// not keep the survivors of), one CTA of PRC_WARPS warps per row: the warps
// split the centroid batches, each starting from the row's seed distance
// beta0 (already computed, the same value as above) and its seed, and the
// CTA keeps the smallest (distance, index) of the warps' results.
constexpr int PRC_WARPS = 8;
__global__ void __launch_bounds__(PRC_WARPS * 32) prune_rows_cta_kernel(
    const uint16_t *__restrict__ X, int d, const float *__restrict__ C, int k, const int32_t *__restrict__ seeds,
    const float2 *__restrict__ thr, int2 *__restrict__ wrow, const int32_t *__restrict__ rows,
    const int32_t *__restrict__ nrows, int32_t *__restrict__ assign, float *__restrict__ dist,
    unsigned long long *__restrict__ counters, int max_rows) {
    __shared__ float sx[PR_MAX_D];
    __shared__ int qid[PRC_WARPS][2][PR_BATCH];
    __shared__ float qps[PRC_WARPS][2][PR_BATCH];
    __shared__ float wp[PRC_WARPS];
    __shared__ int wj[PRC_WARPS];
    extern __shared__ __align__(16) float prc_stg[];  // per warp 32 x STG_LD floats (stage_blocks)
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const float slack = prune_slack(d);
    const int64_t nr = (int64_t)*nrows;
    if (nr >= max_rows) return;  // the tiled kernel takes a list this long
    unsigned long long first_alive = 0, complete = 0, later = 0;
    for (int64_t ri = blockIdx.x; ri < nr; ri += gridDim.x) {
        const int64_t row = rows[ri];
        __syncthreads();  // the previous row's sx and results are read
        for (int i = threadIdx.x; i < d; i += blockDim.x) sx[i] = ldx<uint16_t>(X + row * d + i);
        __syncthreads();
        // the seed and its distance, or an upper bound of it (kept bounds): the
        // seed itself then completes below it, so the result is the same
        int best = seeds[row];
        float beta = thr[row].y;
        prune_batches<true>(sx, C, d, k, warp * PR_BATCH, PRC_WARPS * PR_BATCH, slack, beta, best, qid[warp],
                            qps[warp], first_alive, complete, later, prc_stg + warp * 32 * STG_LD);
        if (lane == 0) {
            wp[warp] = beta;
            wj[warp] = best;
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            float bp = wp[0];
            int bj = wj[0];
            for (int w = 1; w < PRC_WARPS; ++w)
                if (wp[w] < bp || (wp[w] == bp && wj[w] < bj)) {
                    bp = wp[w];
                    bj = wj[w];
                }
            assign[row] = bj;
            if (dist) dist[row] = bp;
            if (wrow) wrow[row] = make_int2(__float_as_int(bp), bj);
        }
    }
    if (lane == 0 && (first_alive | complete | later)) {
        atomicAdd(&counters[0], first_alive);
        atomicAdd(&counters[1], complete);
        atomicAdd(&counters[2], later);
    }
}

// ---------------------------------------------------------------- SQ8 codes
// The same pruning on SQ8 codes (Section 3.1: SuperKMeans extended to SQ8):
// partial distances are exact integers, sum over a 32-dimension block of
// (xbar_i - cbar_i)^2 as |x - c| per byte (__vabsdiffu4) squared and summed by
// __dp4a, so a centroid is dropped exactly when its partial exceeds beta (no
// slack) and the result is the exact code-space argmin.  Point codes are
// staged as 32-bit words (d % 4 == 0) or bytes.
__device__ __forceinline__ int32_t block_partial_u8(const uint8_t *sx, const uint8_t *c, int d, int b, bool words) {
    const int i0 = 32 * b;
    int32_t s = 0;
    if (words && i0 + 32 <= d) {
        const uint32_t *xw = reinterpret_cast<const uint32_t *>(sx + i0);
        const uint32_t *cw = reinterpret_cast<const uint32_t *>(c + i0);
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            const uint32_t df = __vabsdiffu4(xw[q], __ldg(cw + q));
            s = (int32_t)__dp4a(df, df, (uint32_t)s);
        }
    } else {
        const int i1 = min(d, i0 + 32);
        for (int i = i0; i < i1; ++i) {
            const int32_t t = (int32_t)sx[i] - (int32_t)__ldg(c + i);
            s += t * t;
        }
    }
    return s;
}

__global__ void __launch_bounds__(PR_WARPS * 32) prune_assign_sq8_kernel(
    const uint8_t *__restrict__ X, int64_t n, int d, const uint8_t *__restrict__ C, int k,
    const int32_t *__restrict__ prev, int32_t *__restrict__ assign, float *__restrict__ dist,
    unsigned long long *__restrict__ counters) {
    __shared__ __align__(16) uint8_t sx_all[PR_WARPS][PR_MAX_D];
    __shared__ int qid[PR_WARPS][2][PR_BATCH];
    __shared__ int32_t qps[PR_WARPS][2][PR_BATCH];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const unsigned lt = (1u << lane) - 1u;
    uint8_t *sx = sx_all[warp];
    const int nb = (d + 31) >> 5;
    const bool words = (d % 4) == 0 && (reinterpret_cast<uintptr_t>(C) & 3) == 0;
    const int64_t nw = (int64_t)gridDim.x * PR_WARPS;
    unsigned long long first_alive = 0, complete = 0, later = 0;
    for (int64_t row = (int64_t)blockIdx.x * PR_WARPS + warp; row < n; row += nw) {
        __syncwarp();
        for (int i = lane; i < d; i += 32) sx[i] = __ldg(X + row * d + i);
        __syncwarp();
        int best = prev ? prev[row] : 0;
        if (best < 0 || best >= k) best = 0;
        int32_t beta = 0;
        for (int b = 0; b < nb; ++b) beta += block_partial_u8(sx, C + (int64_t)best * d, d, b, words);
        for (int c0 = 0; c0 < k; c0 += PR_BATCH) {
            __syncwarp();
            int cnt = 0;
            for (int s = 0; s < PR_BATCH / 32; ++s) {
                const int j = c0 + 32 * s + lane;
                const int32_t p = (j < k) ? block_partial_u8(sx, C + (int64_t)j * d, d, 0, words) : INT32_MAX;
                const bool alive = j < k && p <= beta;
                const unsigned m = __ballot_sync(0xffffffffu, alive);
                if (alive) {
                    const int pos = cnt + __popc(m & lt);
                    qid[warp][0][pos] = j;
                    qps[warp][0][pos] = p;
                }
                cnt += __popc(m);
            }
            first_alive += cnt;
            int src = 0;
            for (int b = 1; b < nb && cnt > 0; ++b) {
                __syncwarp();
                later += cnt;
                int ncnt = 0;
                for (int t0 = 0; t0 < cnt; t0 += 32) {
                    const int t = t0 + lane;
                    const bool valid = t < cnt;
                    const int j = valid ? qid[warp][src][t] : 0;
                    const int32_t p = valid ? qps[warp][src][t] + block_partial_u8(sx, C + (int64_t)j * d, d, b, words) : 0;
                    const bool alive = valid && p <= beta;
                    const unsigned m = __ballot_sync(0xffffffffu, alive);
                    if (alive) {
                        const int pos = ncnt + __popc(m & lt);
                        qid[warp][src ^ 1][pos] = j;
                        qps[warp][src ^ 1][pos] = p;
                    }
                    ncnt += __popc(m);
                }
                cnt = ncnt;
                src ^= 1;
            }
            __syncwarp();
            complete += cnt;
            for (int t0 = 0; t0 < cnt; t0 += 32) {
                const int t = t0 + lane;
                int32_t p = INT32_MAX;
                int j = 0x7fffffff;
                if (t < cnt) {
                    p = qps[warp][src][t];
                    j = qid[warp][src][t];
                }
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) {
                    const int32_t op = __shfl_xor_sync(0xffffffffu, p, o);
                    const int oj = __shfl_xor_sync(0xffffffffu, j, o);
                    if (op < p || (op == p && oj < j)) {
                        p = op;
                        j = oj;
                    }
                }
                if (p < beta || (p == beta && j < best)) {
                    beta = p;
                    best = j;
                }
            }
        }
        if (lane == 0) {
            assign[row] = best;
            if (dist) dist[row] = (float)beta;
        }
    }
    if (counters && lane == 0) {
        atomicAdd(&counters[0], first_alive);
        atomicAdd(&counters[1], complete);
        atomicAdd(&counters[2], later);
    }
}

// ------------------------------------------------------------ tiled kernels
// A CTA takes TP_PTS points (TP_PTS / 8 per warp) and walks the centroids in
// chunks of TP_KC staged in shared memory (rows padded so that lanes reading
// different centroids at the same offset hit different banks), so a chunk
// is read from L2 once per TP_PTS points instead of once per point.  Per
// point and chunk, lane l takes the first block of centroids l and l + 32;
// the survivors are gathered across the warp (ballots, __fns) into dense
// passes that carry them block by block in lockstep (x's block in registers,
// read once per pass), leaving as soon as no lane survives.  Each pair's
// partial sums are the same fp32 (or integer) values as in the kernels above,
// so the result is the same exact argmin.
constexpr int TP_PTS = 64;
constexpr int TP_KC = 64;
constexpr int TP_WARPS = 8;
constexpr int TP_MAX_D_F32 = 256;

// sum over the 32 dims of a block: x (registers) against c (shared memory),
// increasing index order (the order of block_partial)
__device__ __forceinline__ float block32(const float (&xb)[32], const float *c) {
    float s = 0.0f;
#pragma unroll
    for (int q = 0; q < 8; ++q) {
        const float4 cv = *reinterpret_cast<const float4 *>(c + 4 * q);
        float t = __fsub_rn(xb[4 * q], cv.x);
        s = __fmaf_rn(t, t, s);
        t = __fsub_rn(xb[4 * q + 1], cv.y);
        s = __fmaf_rn(t, t, s);
        t = __fsub_rn(xb[4 * q + 2], cv.z);
        s = __fmaf_rn(t, t, s);
        t = __fsub_rn(xb[4 * q + 3], cv.w);
        s = __fmaf_rn(t, t, s);
    }
    return s;
}

// the i-th survivor of slot masks (M0, M1): slot and owner lane
__device__ __forceinline__ void survivor(unsigned M0, unsigned M1, int i, int &slot, int &owner) {
    const int n0 = __popc(M0);
    slot = i < n0 ? 0 : 1;
    const unsigned ms = slot == 0 ? M0 : M1;
    const int rank = slot == 0 ? i : i - n0;
    owner = (i < n0 + __popc(M1)) ? (int)__fns(ms, 0, rank + 1) : 0;
}

// rows (NULL: every row, one tile of TP_PTS points per CTA): a list of
// *nrows rows walked tile by tile over the grid, whose seeds and seed
// distances (or bounds) come from seeds / thr (the tensor-core front's rows
// pruned over all k); with fewer than min_rows listed rows the kernel leaves
// them to the one-CTA-per-row kernel.  wrow (optional): (distance bits,
// centroid) of each row for the next call.
template <typename TX, bool LIST>
__global__ void __launch_bounds__(TP_WARPS * 32) prune_tiled_kernel(
    const TX *__restrict__ X, int64_t n, int d, const float *__restrict__ C, int k,
    const int32_t *__restrict__ prev, int32_t *__restrict__ assign, float *__restrict__ dist,
    unsigned long long *__restrict__ counters, const int32_t *__restrict__ rows, const int32_t *__restrict__ nrows,
    int min_rows, const int32_t *__restrict__ seeds, const float2 *__restrict__ thr, int2 *__restrict__ wrow) {
    extern __shared__ __align__(16) float tp_smem[];
    const int dp = ((d + 31) & ~31) + 4;  // padded centroid row (floats): a 16-byte multiple, banks shift by 4
    const int dx = (d + 31) & ~31;
    float *cs = tp_smem;                       // [TP_KC][dp]
    float *xs = cs + (size_t)TP_KC * dp;       // [TP_PTS][dx], zero-padded
    float *s_beta = xs + (size_t)TP_PTS * dx;  // [TP_PTS]
    int *s_best = reinterpret_cast<int *>(s_beta + TP_PTS);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nb = (d + 31) >> 5;
    const float slack = 1.0f + 2.0f * (float)(d + 1) * 0x1p-24f;
    const int64_t nr = LIST ? (int64_t)*nrows : n;
    if (LIST && nr < min_rows) return;
    unsigned long long first_alive = 0, complete = 0, later = 0;
    // a list: tiles over the grid; otherwise one tile per CTA
    const int64_t pstep = LIST ? (int64_t)gridDim.x * TP_PTS : nr;
    for (int64_t p0 = (int64_t)blockIdx.x * TP_PTS; p0 < nr; p0 += pstep) {
    const int np = (int)min((int64_t)TP_PTS, nr - p0);
    auto row_of = [&](int q) { return LIST ? (int64_t)rows[p0 + q] : p0 + q; };
    __syncthreads();  // the previous tile's results are written
    for (int e = threadIdx.x; e < TP_PTS * dx; e += blockDim.x) {
        const int q = e / dx, i = e - q * dx;
        xs[e] = (q < np && i < d) ? ldx<TX>(X + row_of(q) * d + i) : 0.0f;
    }
    __syncthreads();
    // each point's bound: its full distance to the seed centroid (block sums
    // in order), or the listed row's seed distance (or bound) already formed
    for (int q = warp; q < np; q += TP_WARPS) {
        const int64_t row = row_of(q);
        if (lane == 0) {
            if (LIST) {
                s_beta[q] = thr[row].y;
                s_best[q] = seeds[row];
            } else {
                int best = prev ? prev[row] : 0;
                if (best < 0 || best >= k) best = 0;
                float beta = 0.0f;
                for (int b = 0; b < nb; ++b) beta += block_partial(xs + q * dx, C + (int64_t)best * d, d, b);
                s_beta[q] = beta;
                s_best[q] = best;
            }
        }
    }
    for (int c0 = 0; c0 < k; c0 += TP_KC) {
        const int kc = min(TP_KC, k - c0);
        __syncthreads();
        for (int e = threadIdx.x; e < TP_KC * dx; e += blockDim.x) {
            const int c = e / dx, i = e - c * dx;
            cs[c * dp + i] = (c < kc && i < d) ? C[(int64_t)(c0 + c) * d + i] : 0.0f;
        }
        __syncthreads();
        for (int q = warp; q < np; q += TP_WARPS) {
            const float *xq = xs + q * dx;
            float beta = s_beta[q];
            int best = s_best[q];
            float lim = beta * slack;
            float xb[32];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const float4 v = *reinterpret_cast<const float4 *>(xq + 4 * u);  // broadcast
                xb[4 * u] = v.x;
                xb[4 * u + 1] = v.y;
                xb[4 * u + 2] = v.z;
                xb[4 * u + 3] = v.w;
            }
            float pa[2];
            unsigned M[2];
#pragma unroll
            for (int s2 = 0; s2 < 2; ++s2) {
                const int c = 32 * s2 + lane;
                // a partial block past d sums zeros (both sides padded), as block_partial
                pa[s2] = c < kc ? block32(xb, cs + c * dp) : INFINITY;
                M[s2] = __ballot_sync(0xffffffffu, c < kc && pa[s2] <= lim);
            }
            const int total = __popc(M[0]) + __popc(M[1]);
            first_alive += lane == 0 ? (unsigned long long)total : 0ull;
            for (int base = 0; base < total; base += 32) {
                const int i = base + lane;
                int slot, owner;
                survivor(M[0], M[1], i, slot, owner);
                const float v0 = __shfl_sync(0xffffffffu, pa[0], owner);
                const float v1 = __shfl_sync(0xffffffffu, pa[1], owner);
                const bool mine = i < total;
                const int c = 32 * slot + owner;
                float p = slot == 0 ? v0 : v1;
                bool alive = mine;
                for (int b = 1; b < nb; ++b) {
                    if (!__any_sync(0xffffffffu, alive)) break;
#pragma unroll
                    for (int u = 0; u < 8; ++u) {
                        const float4 v = *reinterpret_cast<const float4 *>(xq + 32 * b + 4 * u);
                        xb[4 * u] = v.x;
                        xb[4 * u + 1] = v.y;
                        xb[4 * u + 2] = v.z;
                        xb[4 * u + 3] = v.w;
                    }
                    if (alive) {
                        p += block32(xb, cs + c * dp + 32 * b);
                        alive = p <= lim;
                        ++later;
                    }
                }
                complete += alive ? 1ull : 0ull;
                float bp = alive ? p : INFINITY;
                int bj = alive ? c0 + c : 0x7fffffff;
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) {
                    const float op = __shfl_xor_sync(0xffffffffu, bp, o);
                    const int oj = __shfl_xor_sync(0xffffffffu, bj, o);
                    if (op < bp || (op == bp && oj < bj)) {
                        bp = op;
                        bj = oj;
                    }
                }
                if (bp < beta || (bp == beta && bj < best)) {
                    beta = bp;
                    best = bj;
                    lim = beta * slack;
                }
            }
            if (lane == 0) {
                s_beta[q] = beta;
                s_best[q] = best;
            }
        }
    }
    __syncthreads();
    for (int q = threadIdx.x; q < np; q += blockDim.x) {
        const int64_t row = row_of(q);
        assign[row] = s_best[q];
        if (dist) dist[row] = s_beta[q];
        if (LIST && wrow) wrow[row] = make_int2(__float_as_int(s_beta[q]), s_best[q]);
    }
    }  // tiles
    if (counters) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            complete += __shfl_xor_sync(0xffffffffu, complete, o);
            later += __shfl_xor_sync(0xffffffffu, later, o);
        }
        if (lane == 0) {
            atomicAdd(&counters[0], first_alive);
            atomicAdd(&counters[1], complete);
            atomicAdd(&counters[2], later);
        }
    }
}

// ------------------------------------------------ tensor-core front (bf16)
// The seeds' pruned distances and the front's thresholds.  G lanes per row
// (a power of two at least the number of 32-dimension blocks), lane b
// computing block b's partial exactly as block_partial does (x_i - c_i then
// an FMA chain in increasing i), the row's first lane summing the partials
// in block order: beta0 is the very value the pruning kernels compute for
// the seed.
//
// Threshold: the pruned distance D(x, c) is at least the fp32 partial over
// the first F dimensions (fp32 sums of non-negative terms never decrease),
// which is at least (1 - gamma) S_F, S_F = sum_{i < F} (x_i - c_i)^2 =
// ||x_F||^2 + s_F with s_F = ||c_F||^2 - 2 <x_F, c_F>, gamma = (34 + F/32)
// 2^-24 (one rounding per subtraction and square, 32 per block chain, one
// per block sum).  The tensor-core front evaluates s~_F with |s~_F - s_F| <=
// 2 ||x_F|| h'_j + z_j <= W = 2 ||x_F|| max h' + max z (the screen's interval
// with prefix norms; bf16 points are their own operand).  A centroid with
// s~_F > thr = beta0 slack (1 + 2^-16) - ||x_F||^2 + W (each step rounded
// outwards; 2^-16 covers 1 / (1 - gamma) and the rounding of beta0 slack)
// therefore has D(x, c) > fl(beta0 slack) >= the row's minimum and is
// dropped: the pruning kernels, seeded alike, never complete it either
// (slack is theirs).  A non-finite seed distance keeps everything (the row then
// overflows to the full pruning).
// One 32-dimension block of (x_i - c_i)^2 for a lane: x from bf16 (16-byte
// loads), c from fp32 (16-byte loads), every load issued before the chain;
// the sum runs in increasing i as in block_partial.  q (when wanted) gets the
// sum of x_i^2 over the block.  m = dimensions in the block (32 unless it is
// the ragged last one).
__device__ __forceinline__ float block_bf16(const uint16_t *xr, const float *cr, int m, bool want_q, float &q) {
    float part = 0.0f;
    q = 0.0f;
    if (m == 32) {
        uint4 xw[4];
        float4 cv[8];
#pragma unroll
        for (int u = 0; u < 4; ++u) xw[u] = __ldg(reinterpret_cast<const uint4 *>(xr) + u);
#pragma unroll
        for (int u = 0; u < 8; ++u) cv[u] = __ldg(reinterpret_cast<const float4 *>(cr) + u);
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const uint32_t w0 = (u & 1) ? xw[u >> 1].z : xw[u >> 1].x;
            const uint32_t w1 = (u & 1) ? xw[u >> 1].w : xw[u >> 1].y;
            const float xs[4] = {__uint_as_float(w0 << 16), __uint_as_float(w0 & 0xffff0000u),
                                 __uint_as_float(w1 << 16), __uint_as_float(w1 & 0xffff0000u)};
            const float cs[4] = {cv[u].x, cv[u].y, cv[u].z, cv[u].w};
#pragma unroll
            for (int h = 0; h < 4; ++h) {
                const float t = __fsub_rn(xs[h], cs[h]);
                part = __fmaf_rn(t, t, part);
                if (want_q) q = __fmaf_rn(xs[h], xs[h], q);
            }
        }
    } else {
        for (int i = 0; i < m; ++i) {
            const float xv = __uint_as_float(((uint32_t)__ldg(xr + i)) << 16);
            const float t = __fsub_rn(xv, __ldg(cr + i));
            part = __fmaf_rn(t, t, part);
            if (want_q) q = __fmaf_rn(xv, xv, q);
        }
    }
    return part;
}

//
// Kept bounds (the state a previous call on these points left, when its stamp
// matches and no distances are wanted): the row's bound U >= D(x, c) for its
// centroid c grows by that centroid's move delta = ||c' - c|| (rounded up).
// With g = (40 + blocks) 2^-23 (twice the rounding of a pruned distance in
// either direction), the real squared distance is at most U (1 + g), its root
// grows by at most delta (triangle inequality), and the new pruned distance
// is at most U' = (sqrt(U (1 + g)) + delta)^2 (1 + g), every step rounded up;
// the threshold is then formed from U' as above, with the kept prefix norms.
__global__ void front_prep_kernel(const uint16_t *__restrict__ X, int64_t n, int d, int F, int G,
                                  const float *__restrict__ C, int k, const int32_t *__restrict__ prev,
                                  const float *__restrict__ hz, PfRows r, int force_cold,
                                  unsigned long long *__restrict__ ctr) {
    float2 *__restrict__ thr = r.thr;
    const int lane = threadIdx.x & 31;
    const int sub = lane / G, b = lane % G;
    const int rpw = 32 / G;  // rows per warp
    const int nb = (d + 31) >> 5;
    const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    if (blockIdx.x == 0 && threadIdx.x == 0) {
        ctr[3] = (unsigned long long)F;
        ctr[9] = (unsigned long long)k;
    }
    const float H = __ldg(hz), Z = __ldg(hz + 1);
    const float slack = prune_slack(d);
    const float K1 = __fmul_ru(slack, 1.0f + 0x1p-16f);
    if (r.warm_ok && *r.warm_ok && !force_cold) {
        const float g = (float)(40 + nb) * 0x1p-23f;
        const int64_t nt = (int64_t)gridDim.x * blockDim.x;
        for (int64_t row = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; row < n; row += nt) {
            const int2 w = r.wrow[row];
            const float U = __int_as_float(w.x);
            float t = INFINITY, Un = INFINITY;
            int seed = 0;
            if (w.y >= 0 && w.y < k && U >= 0.0f && U < INFINITY) {
                seed = w.y;
                const float rr = __fadd_ru(__fsqrt_ru(__fmul_ru(U, 1.0f + g)), __ldg(&r.shift[seed].y));
                Un = __fmul_ru(__fmul_ru(rr, rr), 1.0f + g);
                const float2 xn = r.xn[row];
                const float W = __fmaf_ru(2.0f * xn.x, H, Z);
                t = __fadd_ru(__fadd_ru(__fsub_ru(__fmul_ru(Un, K1), xn.y), W), 0x1p-100f);
                if (!(t == t) || !(Un < INFINITY)) t = INFINITY;
            }
            thr[row] = make_float2(t, Un);
            r.seed[row] = seed;
        }
        return;
    }
    for (int64_t r0 = warp * rpw; r0 < n; r0 += nw * rpw) {
        const int64_t row = r0 + sub;
        const bool act = row < n;
        int seed = act && prev ? __ldg(prev + row) : 0;
        if (seed < 0 || seed >= k) seed = 0;
        float part = 0.0f, q = 0.0f;
        if (act && b < nb)
            part = block_bf16(X + row * d + 32 * b, C + (int64_t)seed * d + 32 * b, min(32, d - 32 * b), 32 * b < F,
                              q);
        // the row's blocks in order (every lane of the group forms the same sum)
        float beta0 = __shfl_sync(0xffffffffu, part, 0, G);
        for (int t = 1; t < nb; ++t) beta0 = __fadd_rn(beta0, __shfl_sync(0xffffffffu, part, t, G));
        for (int o = G >> 1; o > 0; o >>= 1) q = __fadd_rn(q, __shfl_xor_sync(0xffffffffu, q, o, G));
        if (act && b == 0) {
            // q: fp32 sum of F exact squares, relative error far below (F + 8) 2^-23
            const float grow = (float)(F + 8) * 0x1p-23f;
            const float xn_up = __fsqrt_ru(__fmul_ru(q, 1.0f + grow));
            const float xn2_lo = __fmul_rd(q, 1.0f - grow);
            const float W = __fmaf_ru(2.0f * xn_up, H, Z);
            float t = __fadd_ru(__fsub_ru(__fmul_ru(beta0, K1), xn2_lo), W);
            t = __fadd_ru(t, 0x1p-100f);
            if (!(t == t) || !(beta0 < INFINITY)) t = INFINITY;
            thr[row] = make_float2(t, beta0);
            r.seed[row] = seed;
            if (r.xn) r.xn[row] = make_float2(xn_up, xn2_lo);
        }
    }
}

// Rows the front left with 2 .. cap survivors: each survivor's pruned
// distance, G lanes per survivor (lane b: block b, the terms of block_bf16 in
// its order, the group summing the partials in block order: the very value
// of the pruning kernels), 32 / G survivors a round, their centroid blocks
// gathered coalesced through shared memory (stage_blocks); the smallest (lowest index on
// ties) is the row's argmin, the seed (on the list, at exactly beta0)
// guaranteeing one.  A survivor is complete when its distance is within the
// seed distance times the slack (its partial sums never exceed the full
// one).  One warp per row.
constexpr int PF_FIN_WARPS = 8;
__global__ void __launch_bounds__(PF_FIN_WARPS * 32, 4) prune_finish_kernel(
    const uint16_t *__restrict__ X, int d, int G, const float *__restrict__ C, const float2 *__restrict__ thr,
    const uint16_t *__restrict__ cand, const int32_t *__restrict__ cnt, int cap, int nsub,
    const int32_t *__restrict__ perm, const int32_t *__restrict__ rows, const int32_t *__restrict__ nrows,
    int32_t *__restrict__ assign, float *__restrict__ dist, int2 *__restrict__ wrow, unsigned long long *__restrict__ ctr) {
    __shared__ __align__(16) float stg_all[PF_FIN_WARPS][32 * STG_LD];
    const int lane = threadIdx.x & 31;
    float *stg = stg_all[threadIdx.x >> 5];
    const float *cb = stg + lane * STG_LD;
    const int slot = lane / G, b = lane % G, S = 32 / G;
    const int nb = (d + 31) >> 5;
    const bool full = b < nb && 32 * b + 32 <= d;  // this lane's block has 32 dimensions
    const float slack = prune_slack(d);
    const int64_t nr = (int64_t)*nrows;
    const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    unsigned long long complete = 0, blocks = 0;
    for (int64_t ri = warp; ri < nr; ri += nw) {
        const int64_t row = __ldg(rows + ri);
        const float lim = __ldg(&thr[row].y) * slack;
        const uint32_t pc = (uint32_t)__ldg(cnt + row);
        const int csub = cap / nsub;
        const int c0 = min((int)(pc & 255u), csub);
        const int c1 = nsub > 1 ? min((int)((pc >> 8) & 255u), csub) : 0;
        const int c2 = nsub > 2 ? min((int)((pc >> 16) & 255u), csub) : 0;
        const int c3 = nsub > 3 ? min((int)(pc >> 24), csub) : 0;
        const int tot = c0 + c1 + c2 + c3;
        const uint16_t *xr = X + row * d + 32 * b;
        float bp = INFINITY;
        int bj = 0x7fffffff;
        for (int t0 = 0; t0 < tot; t0 += S) {
            int t = t0 + slot, h = 0;
            const bool valid = t < tot;
            if (t >= c0) {  // sub-list h and the position in it
                t -= c0;
                h = 1;
                if (t >= c1) {
                    t -= c1;
                    h = 2;
                    if (t >= c2) {
                        t -= c2;
                        h = 3;
                    }
                }
            }
            const int j = valid ? __ldg(perm + __ldg(cand + row * cap + h * csub + t)) : 0;
            stage_blocks(stg, C, d, j, b, valid && b < nb);
            float part = 0.0f;
            if (valid && full) {
                // the lane's 32 point values (bf16; the slots of a round read
                // the same 512 bytes, four lines an instruction)
                uint4 xw[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) xw[u] = __ldg(reinterpret_cast<const uint4 *>(xr) + u);
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const float4 cv = reinterpret_cast<const float4 *>(cb)[u];
                    const uint32_t w0 = (u & 1) ? xw[u >> 1].z : xw[u >> 1].x;
                    const uint32_t w1 = (u & 1) ? xw[u >> 1].w : xw[u >> 1].y;
                    float tt = __fsub_rn(__uint_as_float(w0 << 16), cv.x);
                    part = __fmaf_rn(tt, tt, part);
                    tt = __fsub_rn(__uint_as_float(w0 & 0xffff0000u), cv.y);
                    part = __fmaf_rn(tt, tt, part);
                    tt = __fsub_rn(__uint_as_float(w1 << 16), cv.z);
                    part = __fmaf_rn(tt, tt, part);
                    tt = __fsub_rn(__uint_as_float(w1 & 0xffff0000u), cv.w);
                    part = __fmaf_rn(tt, tt, part);
                }
            } else if (valid && b < nb) {  // the last, shorter block
                for (int i = 0; i < d - 32 * b; ++i) {
                    const float tt = __fsub_rn(__uint_as_float(((uint32_t)__ldg(xr + i)) << 16), cb[i]);
                    part = __fmaf_rn(tt, tt, part);
                }
            }
            float D = __shfl_sync(0xffffffffu, part, 0, G);
            for (int u = 1; u < nb; ++u) D = __fadd_rn(D, __shfl_sync(0xffffffffu, part, u, G));
            if (valid && b == 0) {
                blocks += (unsigned long long)nb;
                if (D <= lim) {
                    ++complete;
                    if (D < bp || (D == bp && j < bj)) {
                        bp = D;
                        bj = j;
                    }
                }
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float op = __shfl_xor_sync(0xffffffffu, bp, o);
            const int oj = __shfl_xor_sync(0xffffffffu, bj, o);
            if (op < bp || (op == bp && oj < bj)) {
                bp = op;
                bj = oj;
            }
        }
        if (lane == 0) {
            assign[row] = bj;
            if (dist) dist[row] = bp;
            if (wrow) wrow[row] = make_int2(__float_as_int(bp), bj);
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        complete += __shfl_xor_sync(0xffffffffu, complete, o);
        blocks += __shfl_xor_sync(0xffffffffu, blocks, o);
    }
    if (lane == 0 && (complete | blocks)) {
        atomicAdd(&ctr[1], complete);
        atomicAdd(&ctr[2], blocks);
    }
}

}  // namespace

cudaError_t launch_prune_assign_sq8(const uint8_t *X, int64_t n, int d, const uint8_t *C, int k, const int32_t *prev,
                                    int32_t *assign, float *dist, unsigned long long *counters, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    int64_t blocks = (n + PR_WARPS - 1) / PR_WARPS;
    if (blocks > 152 * 16) blocks = 152 * 16;
    prune_assign_sq8_kernel<<<(int)blocks, PR_WARPS * 32, 0, st>>>(X, n, d, C, k, prev, assign, dist, counters);
    return launched();
}

cudaError_t launch_prune_assign(const void *X, int x_is_bf16, int64_t n, int d, const float *C,
                                int k, const int32_t *prev, int32_t *assign, float *dist,
                                unsigned long long *counters, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    if (d <= TP_MAX_D_F32 && (reinterpret_cast<uintptr_t>(C) & 15) == 0) {
        const int dx = (d + 31) & ~31, dp = dx + 4;
        const size_t smem = ((size_t)TP_KC * dp + (size_t)TP_PTS * dx + 2 * TP_PTS) * sizeof(float);
        const int64_t blocks = (n + TP_PTS - 1) / TP_PTS;
        if (x_is_bf16) {
            cudaError_t e = cudaFuncSetAttribute(prune_tiled_kernel<uint16_t, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 (int)smem);
            if (e != cudaSuccess) return e;
            prune_tiled_kernel<uint16_t, false><<<(unsigned)blocks, TP_WARPS * 32, smem, st>>>(
                static_cast<const uint16_t *>(X), n, d, C, k, prev, assign, dist, counters, nullptr, nullptr, 0,
                nullptr, nullptr, nullptr);
        } else {
            cudaError_t e = cudaFuncSetAttribute(prune_tiled_kernel<float, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 (int)smem);
            if (e != cudaSuccess) return e;
            prune_tiled_kernel<float, false><<<(unsigned)blocks, TP_WARPS * 32, smem, st>>>(
                static_cast<const float *>(X), n, d, C, k, prev, assign, dist, counters, nullptr, nullptr, 0,
                nullptr, nullptr, nullptr);
        }
        return launched();
    }
    int64_t blocks = (n + PR_WARPS - 1) / PR_WARPS;
    if (blocks > 152 * 16) blocks = 152 * 16;
    // centroid blocks gathered coalesced (stage_blocks) when the rows allow it
    const bool stg = (d % 4) == 0 && (reinterpret_cast<uintptr_t>(C) & 15) == 0 && (int64_t)k * d <= (1LL << 26);
    const int stg_bytes = PR_WARPS * 32 * STG_LD * (int)sizeof(float);
    cudaError_t e = cudaSuccess;
    if (x_is_bf16) {
        if (stg) {
            e = cudaFuncSetAttribute(prune_assign_kernel<uint16_t, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     stg_bytes);
            if (e != cudaSuccess) return e;
            prune_assign_kernel<uint16_t, true><<<(int)blocks, PR_WARPS * 32, stg_bytes, st>>>(
                static_cast<const uint16_t *>(X), n, d, C, k, prev, assign, dist, counters);
        } else {
            prune_assign_kernel<uint16_t, false><<<(int)blocks, PR_WARPS * 32, 0, st>>>(
                static_cast<const uint16_t *>(X), n, d, C, k, prev, assign, dist, counters);
        }
    } else {
        if (stg) {
            e = cudaFuncSetAttribute(prune_assign_kernel<float, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     stg_bytes);
            if (e != cudaSuccess) return e;
            prune_assign_kernel<float, true><<<(int)blocks, PR_WARPS * 32, stg_bytes, st>>>(
                static_cast<const float *>(X), n, d, C, k, prev, assign, dist, counters);
        } else {
            prune_assign_kernel<float, false><<<(int)blocks, PR_WARPS * 32, 0, st>>>(
                static_cast<const float *>(X), n, d, C, k, prev, assign, dist, counters);
        }
    }
    return launched();
}

cudaError_t launch_prune_rows_cta(const uint16_t *X, int d, const float *C, int k, const PfRows &r,
                                  const int32_t *rows, const int32_t *nrows, int32_t *assign,
                                  float *dist, unsigned long long *counters, cudaStream_t st) {
    if (d > PR_MAX_D) return cudaErrorInvalidValue;
    // a long list (d <= 256): the tiled kernel (centroid chunks staged once
    // per TP_PTS rows); a short one: one CTA per row (more rows in flight)
    const bool tiled = d <= TP_MAX_D_F32 && (reinterpret_cast<uintptr_t>(C) & 15) == 0;
    constexpr int LONG_LIST = 8192;
    // the centroid blocks are gathered coalesced through shared memory
    // (stage_blocks: d % 4 == 0, C 16-byte aligned, k d < 2^26)
    if ((d % 4) != 0 || (reinterpret_cast<uintptr_t>(C) & 15) != 0 || (int64_t)k * d > (1LL << 26))
        return cudaErrorInvalidValue;
    const int stg_bytes = PRC_WARPS * 32 * STG_LD * (int)sizeof(float);
    cudaError_t e = cudaFuncSetAttribute(prune_rows_cta_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, stg_bytes);
    if (e != cudaSuccess) return e;
    prune_rows_cta_kernel<<<152 * 3, PRC_WARPS * 32, stg_bytes, st>>>(X, d, C, k, r.seed, r.thr, r.wrow, rows, nrows,
                                                                      assign, dist, counters,
                                                                      tiled ? LONG_LIST : INT_MAX);
    e = launched();
    if (e != cudaSuccess || !tiled) return e;
    const int dx = (d + 31) & ~31, dp = dx + 4;
    const size_t smem = ((size_t)TP_KC * dp + (size_t)TP_PTS * dx + 2 * TP_PTS) * sizeof(float);
    e = cudaFuncSetAttribute(prune_tiled_kernel<uint16_t, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
    if (e != cudaSuccess) return e;
    prune_tiled_kernel<uint16_t, true><<<152, TP_WARPS * 32, smem, st>>>(X, 0, d, C, k, nullptr, assign, dist, counters,
                                                                    rows, nrows, LONG_LIST, r.seed, r.thr, r.wrow);
    return launched();
}

cudaError_t launch_prune_front_prep(const uint16_t *X, int64_t n, int d, int F, const float *C, int k,
                                    const int32_t *prev, const float *hz, const PfRows &r, int force_cold,
                                    unsigned long long *ctr, cudaStream_t st) {
    const int nb = (d + 31) >> 5;
    int G = 1;
    while (G < nb) G <<= 1;
    if (G > 32 || F % 32 != 0 || F > d || (d % 8) != 0) return cudaErrorInvalidValue;
    const int64_t per_block = 256 / G;  // rows per block of 256 threads
    int64_t blocks = (n + per_block - 1) / per_block;
    if (blocks > 152 * 16) blocks = 152 * 16;
    if (blocks < 1) blocks = 1;
    front_prep_kernel<<<(int)blocks, 256, 0, st>>>(X, n, d, F, G, C, k, prev, hz, r, force_cold, ctr);
    return launched();
}

cudaError_t launch_prune_finish(const uint16_t *X, int d, const float *C, const float2 *thr, const uint16_t *cand,
                                const int32_t *cnt, int cap, int nsub, const int32_t *perm, const int32_t *rows,
                                const int32_t *nrows, int32_t *assign, float *dist, int2 *wrow,
                                unsigned long long *ctr, cudaStream_t st) {
    const int nb = (d + 31) >> 5;
    int G = 1;
    while (G < nb) G <<= 1;
    if (G > 32 || (d % 8) != 0 || nsub < 1 || nsub > 4 || cap % nsub != 0 || cap / nsub > 255)
        return cudaErrorInvalidValue;
    // stage_blocks: C 16-byte aligned, k d <= 2^26 (the front's positions are
    // 16-bit, k <= 65536, and d <= 1024); the point rows 16-byte aligned
    if ((reinterpret_cast<uintptr_t>(C) & 15) != 0 || (reinterpret_cast<uintptr_t>(X) & 15) != 0 || d > 1024)
        return cudaErrorInvalidValue;
    prune_finish_kernel<<<152 * 4, PF_FIN_WARPS * 32, 0, st>>>(X, d, G, C, thr, cand, cnt, cap, nsub, perm, rows, nrows,
                                                               assign, dist, wrow, ctr);
    return launched();
}

}  // namespace skm
