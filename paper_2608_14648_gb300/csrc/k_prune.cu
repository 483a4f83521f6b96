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

template <typename TX>
__global__ void __launch_bounds__(PR_WARPS * 32) prune_assign_kernel(
    const TX *__restrict__ X, int64_t n, int d, const float *__restrict__ C, int k,
    const int32_t *__restrict__ prev, int32_t *__restrict__ assign, float *__restrict__ dist,
    unsigned long long *__restrict__ counters) {
    __shared__ float sx_all[PR_WARPS][PR_MAX_D];
    __shared__ int qid[PR_WARPS][2][PR_BATCH];
    __shared__ float qps[PR_WARPS][2][PR_BATCH];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const unsigned lt = (1u << lane) - 1u;
    float *sx = sx_all[warp];
    const int nb = (d + 31) >> 5;
    // relative rounding of a d-term fp32 sum of non-negative terms is below
    // d * 2^-24; keep anything within twice that of beta
    const float slack = 1.0f + 2.0f * (float)(d + 1) * 0x1p-24f;
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
        for (int c0 = 0; c0 < k; c0 += PR_BATCH) {
            __syncwarp();  // queue 0 may still be read by the previous batch
            // first block over the whole batch, survivors compacted into queue 0
            int cnt = 0;
            for (int s = 0; s < PR_BATCH / 32; ++s) {
                const int j = c0 + 32 * s + lane;
                const float p = (j < k) ? block_partial(sx, C + (int64_t)j * d, d, 0) : INFINITY;
                const bool alive = p <= beta * slack;
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
                    const float p =
                        valid ? qps[warp][src][t] + block_partial(sx, C + (int64_t)j * d, d, b) : INFINITY;
                    const bool alive = valid && p <= beta * slack;
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
            // complete candidates: full distances; keep the smallest (lowest index on ties)
            for (int t0 = 0; t0 < cnt; t0 += 32) {
                const int t = t0 + lane;
                float p = INFINITY;
                int j = 0x7fffffff;
                if (t < cnt) {
                    p = qps[warp][src][t];
                    j = qid[warp][src][t];
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

template <typename TX>
__global__ void __launch_bounds__(TP_WARPS * 32) prune_tiled_kernel(
    const TX *__restrict__ X, int64_t n, int d, const float *__restrict__ C, int k,
    const int32_t *__restrict__ prev, int32_t *__restrict__ assign, float *__restrict__ dist,
    unsigned long long *__restrict__ counters) {
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
    const int64_t p0 = (int64_t)blockIdx.x * TP_PTS;
    const int np = (int)min((int64_t)TP_PTS, n - p0);
    unsigned long long first_alive = 0, complete = 0, later = 0;
    for (int e = threadIdx.x; e < TP_PTS * dx; e += blockDim.x) {
        const int q = e / dx, i = e - q * dx;
        xs[e] = (q < np && i < d) ? ldx<TX>(X + (p0 + q) * d + i) : 0.0f;
    }
    __syncthreads();
    // each point's bound: its full distance to the seed centroid (block sums in order)
    for (int q = warp; q < np; q += TP_WARPS) {
        int best = prev ? prev[p0 + q] : 0;
        if (best < 0 || best >= k) best = 0;
        if (lane == 0) {
            float beta = 0.0f;
            for (int b = 0; b < nb; ++b) beta += block_partial(xs + q * dx, C + (int64_t)best * d, d, b);
            s_beta[q] = beta;
            s_best[q] = best;
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
        assign[p0 + q] = s_best[q];
        if (dist) dist[p0 + q] = s_beta[q];
    }
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
            cudaError_t e = cudaFuncSetAttribute(prune_tiled_kernel<uint16_t>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 (int)smem);
            if (e != cudaSuccess) return e;
            prune_tiled_kernel<uint16_t><<<(unsigned)blocks, TP_WARPS * 32, smem, st>>>(
                static_cast<const uint16_t *>(X), n, d, C, k, prev, assign, dist, counters);
        } else {
            cudaError_t e = cudaFuncSetAttribute(prune_tiled_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 (int)smem);
            if (e != cudaSuccess) return e;
            prune_tiled_kernel<float><<<(unsigned)blocks, TP_WARPS * 32, smem, st>>>(
                static_cast<const float *>(X), n, d, C, k, prev, assign, dist, counters);
        }
        return launched();
    }
    int64_t blocks = (n + PR_WARPS - 1) / PR_WARPS;
    if (blocks > 152 * 16) blocks = 152 * 16;
    if (x_is_bf16)
        prune_assign_kernel<uint16_t><<<(int)blocks, PR_WARPS * 32, 0, st>>>(
            static_cast<const uint16_t *>(X), n, d, C, k, prev, assign, dist, counters);
    else
        prune_assign_kernel<float><<<(int)blocks, PR_WARPS * 32, 0, st>>>(
            static_cast<const float *>(X), n, d, C, k, prev, assign, dist, counters);
    return launched();
}

}  // namespace skm
