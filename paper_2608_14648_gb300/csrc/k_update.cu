// Centroid update, Section 2.3 STEP 3 (and the quantized-domain forms of
// Section 3.1): a sort-by-cluster segmented reduction.
//   1. histogram of assignments (shared-memory privatised counters),
//   2. exclusive scan -> per-cluster offsets,
//   3. scatter point ids (and their cluster) into cluster-contiguous order,
//   4. fp32/bf16 and 1-bit: warps take equal runs of the sorted order and
//      flush per-cluster register sums with global atomics (load balanced
//      whatever the cluster sizes); SQ8: one CTA per cluster;
//   5. finalise: divide by the counts (or add into caller partial sums).
// Integer representations accumulate in int64 and are exact, so their result
// does not depend on the member order produced by the scatter.
#include "skm_internal.cuh"

namespace skm {

// ---------------------------------------------------------------- histogram
__global__ void histogram_kernel(const int32_t *__restrict__ assign, int64_t n, int k,
                                 int32_t *__restrict__ counts, int use_smem) {
    extern __shared__ int32_t sh[];
    if (use_smem) {
        for (int j = threadIdx.x; j < k; j += blockDim.x) sh[j] = 0;
        __syncthreads();
    }
    for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < n;
         t += (int64_t)gridDim.x * blockDim.x) {
        const int a = assign[t];
        if (a < 0 || a >= k) continue;  // out-of-range assignments are skipped
        if (use_smem)
            atomicAdd(&sh[a], 1);
        else
            atomicAdd(&counts[a], 1);
    }
    if (use_smem) {
        __syncthreads();
        for (int j = threadIdx.x; j < k; j += blockDim.x)
            if (sh[j]) atomicAdd(&counts[j], sh[j]);
    }
}

// One block: the number of zero entries of counts[0..k) into *out.
__global__ void count_zeros_kernel(const int64_t *__restrict__ counts, int k, int64_t *__restrict__ out) {
    __shared__ int part[32];
    int z = 0;
    for (int j = threadIdx.x; j < k; j += blockDim.x) z += counts[j] == 0;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) z += __shfl_xor_sync(0xffffffffu, z, o);
    if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = z;
    __syncthreads();
    if (threadIdx.x < 32) {
        z = threadIdx.x < (blockDim.x >> 5) ? part[threadIdx.x] : 0;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) z += __shfl_xor_sync(0xffffffffu, z, o);
        if (threadIdx.x == 0) *out = z;
    }
}

cudaError_t launch_count_zeros(const int64_t *counts, int k, int64_t *out, cudaStream_t st) {
    count_zeros_kernel<<<1, 1024, 0, st>>>(counts, k, out);
    return launched();
}

cudaError_t launch_histogram(const int32_t *assign, int64_t n, int k, int32_t *counts32,
                             cudaStream_t st) {
    cudaError_t e = cudaMemsetAsync(counts32, 0, sizeof(int32_t) * (size_t)k, st);
    if (e != cudaSuccess) return e;
    if (n == 0) return cudaSuccess;
    const int use_smem = k <= 12288;
    const size_t smem = use_smem ? sizeof(int32_t) * (size_t)k : 0;
    // few blocks: each one adds its nonzero shared counters to the global ones,
    // so the global atomics grow with blocks x k
    int64_t blocks = (n + 4095) / 4096;
    if (blocks > 152 * 2) blocks = 152 * 2;
    histogram_kernel<<<(unsigned)blocks, 1024, smem, st>>>(assign, n, k, counts32, use_smem);
    return launched();
}

// --------------------------------------------------------------------- scan
// Single block of 1024 threads; each thread scans a contiguous run of counts.
__global__ void scan_offsets_kernel(const int32_t *__restrict__ counts, int k,
                                    int64_t *__restrict__ offsets, int64_t *__restrict__ counts64,
                                    int accumulate) {
    __shared__ int64_t wsum[32];
    const int t = threadIdx.x, lane = t & 31, w = t >> 5;
    const int per = (k + blockDim.x - 1) / blockDim.x;
    const int lo = min(k, t * per), hi = min(k, lo + per);
    int64_t s = 0;
    for (int j = lo; j < hi; ++j) s += counts[j];
    // exclusive scan of the threads' run sums: shuffles inside each warp, then
    // the warp totals (exact integer sums, so any order gives the same offsets)
    int64_t v = s;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int64_t u = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += u;
    }
    if (lane == 31) wsum[w] = v;
    __syncthreads();
    if (w == 0) {
        int64_t x = lane < (int)(blockDim.x >> 5) ? wsum[lane] : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int64_t u = __shfl_up_sync(0xffffffffu, x, o);
            if (lane >= o) x += u;
        }
        wsum[lane] = x;  // inclusive over warps
    }
    __syncthreads();
    int64_t run = v - s + (w > 0 ? wsum[w - 1] : 0);
    if (t == (int)blockDim.x - 1) offsets[k] = run + s;
    for (int j = lo; j < hi; ++j) {
        offsets[j] = run;
        run += counts[j];
        if (counts64) {
            if (accumulate)
                counts64[j] += counts[j];
            else
                counts64[j] = counts[j];
        }
    }
}

cudaError_t launch_scan_offsets(const int32_t *counts32, int k, int64_t *offsets,
                                int64_t *counts64_out, int accumulate_counts, cudaStream_t st) {
    scan_offsets_kernel<<<1, 1024, 0, st>>>(counts32, k, offsets, counts64_out,
                                            accumulate_counts);
    return launched();
}

// ------------------------------------------------------------------ scatter
__global__ void scatter_kernel(const int32_t *__restrict__ assign, int64_t n, int k,
                               const int64_t *__restrict__ offsets, int32_t *__restrict__ cursor,
                               int32_t *__restrict__ perm, int32_t *__restrict__ scl) {
    for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < n;
         t += (int64_t)gridDim.x * blockDim.x) {
        const int a = assign[t];
        if (a < 0 || a >= k) continue;  // skipped consistently with the histogram
        const int pos = atomicAdd(&cursor[a], 1);
        perm[offsets[a] + pos] = (int32_t)t;
        if (scl) scl[offsets[a] + pos] = a;
    }
}

// Block-aggregated form: a block counts its SC_POINTS points per cluster in
// shared memory, reserves one range per cluster with a single global atomic,
// then places its points inside those ranges (shared-memory atomics), so the
// global atomics drop from one per point to one per (block, cluster).
constexpr int SC_POINTS = 4096;
constexpr int SC_THREADS = 512;
constexpr int SC_MAX_K = 12288;  // 48 KiB of counters

__global__ void __launch_bounds__(SC_THREADS) scatter_blocked_kernel(
    const int32_t *__restrict__ assign, int64_t n, int k, const int64_t *__restrict__ offsets,
    int32_t *__restrict__ cursor, int32_t *__restrict__ perm, int32_t *__restrict__ scl) {
    extern __shared__ int32_t cnt_sh[];
    const int64_t p0 = (int64_t)blockIdx.x * SC_POINTS;
    const int64_t p1 = min(n, p0 + SC_POINTS);
    for (int j = threadIdx.x; j < k; j += SC_THREADS) cnt_sh[j] = 0;
    __syncthreads();
    for (int64_t t = p0 + threadIdx.x; t < p1; t += SC_THREADS) {
        const int a = assign[t];
        if (a >= 0 && a < k) atomicAdd(&cnt_sh[a], 1);
    }
    __syncthreads();
    for (int j = threadIdx.x; j < k; j += SC_THREADS) {
        const int c = cnt_sh[j];
        if (c) cnt_sh[j] = (int32_t)offsets[j] + atomicAdd(&cursor[j], c);
    }
    __syncthreads();
    for (int64_t t = p0 + threadIdx.x; t < p1; t += SC_THREADS) {
        const int a = assign[t];
        if (a < 0 || a >= k) continue;  // skipped consistently with the histogram
        const int pos = atomicAdd(&cnt_sh[a], 1);
        perm[pos] = (int32_t)t;
        if (scl) scl[pos] = a;
    }
}

cudaError_t launch_scatter(const int32_t *assign, int64_t n, int k, const int64_t *offsets,
                           int32_t *cursor, int32_t *perm, int32_t *scl, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    if (k <= SC_MAX_K) {
        const int64_t blocks = (n + SC_POINTS - 1) / SC_POINTS;
        scatter_blocked_kernel<<<(unsigned)blocks, SC_THREADS, sizeof(int32_t) * (size_t)k, st>>>(
            assign, n, k, offsets, cursor, perm, scl);
        return launched();
    }
    int64_t blocks = (n + 255) / 256;
    if (blocks > 152 * 8) blocks = 152 * 8;
    scatter_kernel<<<(unsigned)blocks, 256, 0, st>>>(assign, n, k, offsets, cursor, perm, scl);
    return launched();
}

// ------------------------------------------------------ row loads for the sums
// Lane l reads 16-byte column groups l, l + 32, ... of a 1024-element column
// chunk of a point row (fp32 or bf16), zero past d.
constexpr int SEG_WARPS = 8;
constexpr int SEG_THREADS = SEG_WARPS * 32;
constexpr int SEG_CHUNK = 1024;  // columns per pass (float: 8 float4 per lane)

template <bool BF16>
__device__ __forceinline__ void seg_load8(const void *X, int64_t p, int d, int c0, int lane,
                                          float (&v)[SEG_CHUNK / 32]) {
    // columns c0 + 4*(lane + 32*g) .. +3 for g = 0..7 (zero past d)
#pragma unroll
    for (int g = 0; g < SEG_CHUNK / 128; ++g) {
        const int c = c0 + 4 * (lane + 32 * g);
        float4 f = make_float4(0.f, 0.f, 0.f, 0.f);
        if (BF16) {
            const uint16_t *x = reinterpret_cast<const uint16_t *>(X) + p * d;
            if (c + 3 < d && (d % 4) == 0) {
                const uint2 w = __ldg(reinterpret_cast<const uint2 *>(x + c));
                f = make_float4(__uint_as_float(w.x << 16), __uint_as_float(w.x & 0xffff0000u),
                                __uint_as_float(w.y << 16), __uint_as_float(w.y & 0xffff0000u));
            } else {
                float t[4];
#pragma unroll
                for (int u = 0; u < 4; ++u)
                    t[u] = (c + u < d) ? __uint_as_float(((uint32_t)__ldg(x + c + u)) << 16) : 0.f;
                f = make_float4(t[0], t[1], t[2], t[3]);
            }
        } else {
            const float *x = reinterpret_cast<const float *>(X) + p * d;
            if (c + 3 < d && (d % 4) == 0) {
                f = __ldg(reinterpret_cast<const float4 *>(x + c));
            } else {
                float t[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) t[u] = (c + u < d) ? __ldg(x + c + u) : 0.f;
                f = make_float4(t[0], t[1], t[2], t[3]);
            }
        }
        v[4 * g] = f.x;
        v[4 * g + 1] = f.y;
        v[4 * g + 2] = f.z;
        v[4 * g + 3] = f.w;
    }
}

// ------------------------------------------------------- segmented sums: SQ8
__device__ __forceinline__ uint8_t round_half_even_div(int64_t S, int64_t m) {
    int64_t q = S / m;
    const int64_t r = S - q * m;
    if (2 * r > m || (2 * r == m && (q & 1))) q += 1;
    return (uint8_t)q;
}

// Warp w takes members w, w + 8, ...; lane l sums bytes 4l..4l+3 of each
// 128-byte column group; exact integer partials are combined with shared
// memory atomics (order-independent).
__global__ void __launch_bounds__(SEG_THREADS) segsum_sq8_kernel(
    const uint8_t *__restrict__ X, int d, const int32_t *__restrict__ perm,
    const int64_t *__restrict__ offsets, uint8_t *__restrict__ C, int64_t *__restrict__ partial) {
    __shared__ unsigned long long tot[SEG_CHUNK];
    const int j = blockIdx.x;
    const int64_t lo = offsets[j], hi = offsets[j + 1];
    const int64_t cnt = hi - lo;
    if (cnt == 0) return;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const bool vec = (d % 4) == 0;
    for (int c0 = 0; c0 < d; c0 += SEG_CHUNK) {
        for (int t = threadIdx.x; t < SEG_CHUNK; t += SEG_THREADS) tot[t] = 0ull;
        __syncthreads();
        uint32_t acc[SEG_CHUNK / 32];  // columns c0 + 4*(lane + 32 g) + u
#pragma unroll
        for (int t = 0; t < SEG_CHUNK / 32; ++t) acc[t] = 0u;
        for (int64_t q = lo + warp; q < hi; q += SEG_WARPS) {
            const uint8_t *x = X + (int64_t)perm[q] * d;
#pragma unroll
            for (int g = 0; g < SEG_CHUNK / 128; ++g) {
                const int c = c0 + 4 * (lane + 32 * g);
                uint32_t w = 0;
                if (vec && c + 3 < d) {
                    w = __ldg(reinterpret_cast<const uint32_t *>(x + c));
                } else {
#pragma unroll
                    for (int u = 0; u < 4; ++u)
                        if (c + u < d) w |= ((uint32_t)__ldg(x + c + u)) << (8 * u);
                }
#pragma unroll
                for (int u = 0; u < 4; ++u) acc[4 * g + u] += (w >> (8 * u)) & 0xffu;
            }
        }
#pragma unroll
        for (int g = 0; g < SEG_CHUNK / 128; ++g)
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int t = 4 * (lane + 32 * g) + u;
                if (c0 + t < d && acc[4 * g + u]) atomicAdd(&tot[t], (unsigned long long)acc[4 * g + u]);
            }
        __syncthreads();
        for (int t = threadIdx.x; t < SEG_CHUNK; t += SEG_THREADS) {
            const int i = c0 + t;
            if (i >= d) break;
            const int64_t S = (int64_t)tot[t];
            if (partial)
                partial[(int64_t)j * d + i] += S;
            else
                C[(int64_t)j * d + i] = round_half_even_div(S, cnt);
        }
        __syncthreads();
    }
}

cudaError_t launch_segsum_sq8(const uint8_t *X, int d, const int32_t *perm,
                              const int64_t *offsets, int k, uint8_t *C_inout, int64_t *partial,
                              cudaStream_t st) {
    segsum_sq8_kernel<<<k, SEG_THREADS, 0, st>>>(X, d, perm, offsets, C_inout, partial);
    return launched();
}

// ------------------------------------------------------ segmented sums: RBQ1
// Fused decode-average with exact fixed-point sums: Fq = rint(F 2^e),
// T_i = sum Fq xbar_i, U = sum Fq;
// c_i = m_i + (2 T_i - U) f in fp64 -> fp32, with one factor per cluster
// f = (fl(1/sqrt(d)) 2^-e) / count.
__device__ __forceinline__ float rbq1_finish(int64_t T, int64_t U, float m, double f) {
    return __double2float_rn(__dadd_rn((double)m, __dmul_rn(__ll2double_rn(2 * T - U), f)));
}

// Fixed-point weights Fq = rint(F 2^e), once per update call, written in the
// cluster-sorted order (position q holds the weight of member perm[q]).
__global__ void rbq1_fq_kernel(const float *__restrict__ F, const int32_t *__restrict__ perm,
                               const int64_t *__restrict__ offsets, int k, int e,
                               int64_t *__restrict__ fq) {
    const int64_t nval = offsets[k];
    for (int64_t q = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; q < nval;
         q += (int64_t)gridDim.x * blockDim.x)
        fq[q] = fixed_rint(F[perm[q]], e);
}

cudaError_t launch_rbq1_fq(const float *F, const int32_t *perm, const int64_t *offsets, int k,
                           int64_t n, int e, int64_t *fq, cudaStream_t st) {
    int64_t blocks = (n + 255) / 256;
    if (blocks > 152 * 8) blocks = 152 * 8;
    if (blocks < 1) blocks = 1;
    rbq1_fq_kernel<<<(int)blocks, 256, 0, st>>>(F, perm, offsets, k, e, fq);
    return launched();
}

// -------------------------------------------- chunked segmented sums (load balanced)
// Warps take CH_ROWS consecutive members of the cluster-sorted order, so
// every warp has the same work whatever the cluster sizes.  A warp adds its
// rows into register accumulators and flushes them with global atomics into
// the cluster's accumulator whenever the cluster changes (and at the end).
// The member count of the sorted order is offsets[k].
constexpr int CH_WARPS = 8;
constexpr int CH_ROWS = 128;

// fp32 / bf16 points -> float or double accumulators S[k][d].
template <bool BF16, typename ACC>
__global__ void __launch_bounds__(CH_WARPS * 32) chunk_sum_float_kernel(
    const void *__restrict__ Xv, int d, const int32_t *__restrict__ perm,
    const int32_t *__restrict__ scl, const int64_t *__restrict__ offsets, int k,
    ACC *__restrict__ S, int64_t stride) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t nval = offsets[k];
    const int64_t q0 = ((int64_t)blockIdx.x * CH_WARPS + warp) * CH_ROWS;
    if (q0 >= nval) return;
    const int64_t q1 = min(nval, q0 + CH_ROWS);
    for (int c0 = 0; c0 < d; c0 += SEG_CHUNK) {
        float acc[SEG_CHUNK / 32];
#pragma unroll
        for (int t = 0; t < SEG_CHUNK / 32; ++t) acc[t] = 0.0f;
        int cur = scl[q0];
        auto flush = [&](int c) {
#pragma unroll
            for (int g = 0; g < SEG_CHUNK / 128; ++g)
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int col = c0 + 4 * (lane + 32 * g) + u;
                    if (col < d) atomicAdd(S + (int64_t)c * stride + col, (ACC)acc[4 * g + u]);
                    acc[4 * g + u] = 0.0f;
                }
        };
        int64_t q = q0;
        for (; q + 1 < q1; q += 2) {
            const int ca = scl[q], cb = scl[q + 1];
            float v0[SEG_CHUNK / 32], v1[SEG_CHUNK / 32];
            seg_load8<BF16>(Xv, perm[q], d, c0, lane, v0);
            seg_load8<BF16>(Xv, perm[q + 1], d, c0, lane, v1);
            if (ca != cur) {
                flush(cur);
                cur = ca;
            }
#pragma unroll
            for (int t = 0; t < SEG_CHUNK / 32; ++t) acc[t] += v0[t];
            if (cb != cur) {
                flush(cur);
                cur = cb;
            }
#pragma unroll
            for (int t = 0; t < SEG_CHUNK / 32; ++t) acc[t] += v1[t];
        }
        if (q < q1) {
            const int ca = scl[q];
            float v0[SEG_CHUNK / 32];
            seg_load8<BF16>(Xv, perm[q], d, c0, lane, v0);
            if (ca != cur) {
                flush(cur);
                cur = ca;
            }
#pragma unroll
            for (int t = 0; t < SEG_CHUNK / 32; ++t) acc[t] += v0[t];
        }
        flush(cur);
    }
}

// 1-bit codes -> int64 accumulators T[k][d+1] (column d holds U = sum Fq);
// fqs in the sorted order.  Lane l holds dimension l of each code word.  A
// warp's member ids, cluster ids and weights are read lane-parallel up
// front; the member rows (W words, lane w loads word w) are read RB_DEPTH
// rows ahead into a register ring, and each row's words reach every lane by
// shuffles, so the loads of later rows overlap the sums of earlier ones.
constexpr int RB_DEPTH = 8;

__device__ __forceinline__ int pick4(const int (&a)[4], int i) {
    const int t = i >> 5;
    const int v = t == 0 ? a[0] : t == 1 ? a[1] : t == 2 ? a[2] : a[3];
    return __shfl_sync(0xffffffffu, v, i & 31);
}
__device__ __forceinline__ int64_t pick4(const int64_t (&a)[4], int i) {
    const int t = i >> 5;
    const int64_t v = t == 0 ? a[0] : t == 1 ? a[1] : t == 2 ? a[2] : a[3];
    return __shfl_sync(0xffffffffu, v, i & 31);
}

template <int WM>
__global__ void __launch_bounds__(CH_WARPS * 32) chunk_sum_rbq1_kernel(
    const uint32_t *__restrict__ codes, const int64_t *__restrict__ fqs, int d,
    const int32_t *__restrict__ perm, const int32_t *__restrict__ scl,
    const int64_t *__restrict__ offsets, int k, unsigned long long *__restrict__ T) {
    static_assert(CH_ROWS == 128, "pick4 covers 4 x 32 positions");
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t nval = offsets[k];
    const int64_t q0 = ((int64_t)blockIdx.x * CH_WARPS + warp) * CH_ROWS;
    if (q0 >= nval) return;
    const int cnt = (int)(nval - q0 < CH_ROWS ? nval - q0 : CH_ROWS);
    const int W = (d + 31) >> 5;
    const uint32_t lm = 1u << lane;
    int pp[4], cc[4];
    int64_t ff[4];
#pragma unroll
    for (int t = 0; t < 4; ++t) {
        const int i = lane + 32 * t;
        pp[t] = i < cnt ? perm[q0 + i] : 0;
        cc[t] = i < cnt ? scl[q0 + i] : -1;
        ff[t] = i < cnt ? fqs[q0 + i] : 0;
    }
    for (int w0 = 0; w0 < W; w0 += WM) {
        const int nw = min(WM, W - w0);
        // Fq = hi 2^20 + lo as two 32-bit sums (at most CH_ROWS rows between
        // flushes: sum lo < 2^27, sum hi <= 2^24)
        uint32_t alo[WM], ahi[WM];
#pragma unroll
        for (int t = 0; t < WM; ++t) alo[t] = ahi[t] = 0u;
        int64_t usum = 0;
        int cur = pick4(cc, 0);
        auto flush = [&](int c) {
#pragma unroll
            for (int t = 0; t < WM; ++t) {
                const int col = 32 * (w0 + t) + lane;
                const unsigned long long v = ((unsigned long long)ahi[t] << 20) + alo[t];
                if (t < nw && col < d && v) atomicAdd(T + (int64_t)c * (d + 1) + col, v);
                alo[t] = ahi[t] = 0u;
            }
            if (w0 == 0 && lane == 0 && usum) atomicAdd(T + (int64_t)c * (d + 1) + d, (unsigned long long)usum);
            usum = 0;
        };
        uint32_t buf[RB_DEPTH];
#pragma unroll
        for (int r = 0; r < RB_DEPTH; ++r) {
            const int p = pick4(pp, r);
            buf[r] = (r < cnt && lane < nw) ? __ldg(codes + (int64_t)p * W + w0 + lane) : 0u;
        }
        for (int i0 = 0; i0 < cnt; i0 += RB_DEPTH) {
#pragma unroll
            for (int r = 0; r < RB_DEPTH; ++r) {
                const int i = i0 + r;
                const uint32_t mine = buf[r];
                const int in = i + RB_DEPTH;
                const int pn = pick4(pp, in < CH_ROWS ? in : 0);
                buf[r] = (in < cnt && lane < nw) ? __ldg(codes + (int64_t)pn * W + w0 + lane) : 0u;
                if (i < cnt) {  // warp-uniform
                    const int c = pick4(cc, i);
                    const int64_t fq = pick4(ff, i);
                    if (c != cur) {
                        flush(cur);
                        cur = c;
                    }
                    usum += fq;
                    const uint32_t flo = (uint32_t)fq & 0xfffffu, fhi = (uint32_t)(fq >> 20);
#pragma unroll
                    for (int t = 0; t < WM; ++t) {
                        if (t < nw) {
                            add_if_bit2(alo[t], ahi[t], __shfl_sync(0xffffffffu, mine, t), lm, flo, fhi);
                        }
                    }
                }
            }
        }
        flush(cur);
    }
}

static unsigned chunk_blocks(int64_t n) {
    const int64_t per = (int64_t)CH_WARPS * CH_ROWS;
    int64_t b = (n + per - 1) / per;
    return (unsigned)(b < 1 ? 1 : b);
}

cudaError_t launch_chunk_sum_float(const void *X, int x_is_bf16, int64_t n, int d,
                                   const int32_t *perm, const int32_t *scl,
                                   const int64_t *offsets, int k, float *S_f, double *S_d,
                                   cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    const unsigned g = chunk_blocks(n);
    if (S_d) {
        if (x_is_bf16)
            chunk_sum_float_kernel<true, double><<<g, CH_WARPS * 32, 0, st>>>(X, d, perm, scl, offsets, k, S_d, d);
        else
            chunk_sum_float_kernel<false, double><<<g, CH_WARPS * 32, 0, st>>>(X, d, perm, scl, offsets, k, S_d, d);
    } else {
        if (x_is_bf16)
            chunk_sum_float_kernel<true, float><<<g, CH_WARPS * 32, 0, st>>>(X, d, perm, scl, offsets, k, S_f, d);
        else
            chunk_sum_float_kernel<false, float><<<g, CH_WARPS * 32, 0, st>>>(X, d, perm, scl, offsets, k, S_f, d);
    }
    return launched();
}

cudaError_t launch_chunk_sum_rbq1(const uint32_t *codes, const int64_t *fq, int64_t n, int d,
                                  const int32_t *perm, const int32_t *scl, const int64_t *offsets,
                                  int k, int64_t *T, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    const int W = (d + 31) >> 5;
    auto T64 = reinterpret_cast<unsigned long long *>(T);
    const unsigned g = chunk_blocks(n);
    if (W <= 8)
        chunk_sum_rbq1_kernel<8><<<g, CH_WARPS * 32, 0, st>>>(codes, fq, d, perm, scl, offsets, k, T64);
    else if (W <= 16)
        chunk_sum_rbq1_kernel<16><<<g, CH_WARPS * 32, 0, st>>>(codes, fq, d, perm, scl, offsets, k, T64);
    else if (W <= 24)
        chunk_sum_rbq1_kernel<24><<<g, CH_WARPS * 32, 0, st>>>(codes, fq, d, perm, scl, offsets, k, T64);
    else
        chunk_sum_rbq1_kernel<32><<<g, CH_WARPS * 32, 0, st>>>(codes, fq, d, perm, scl, offsets, k, T64);
    return launched();
}

// fp32 sums -> centroids (clusters without members keep theirs)
__global__ void finalize_float32_kernel(const float *__restrict__ S,
                                        const int64_t *__restrict__ counts, int k, int d,
                                        float *__restrict__ C) {
    const int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
    if (t >= (int64_t)k * d) return;
    const int64_t c = counts[t / d];
    if (c > 0) C[t] = __fdiv_rn(S[t], (float)c);
}

cudaError_t launch_finalize_float32(const float *S, const int64_t *counts, int k, int d,
                                    float *C_inout, cudaStream_t st) {
    const int64_t tot = (int64_t)k * d;
    finalize_float32_kernel<<<(unsigned)((tot + 255) / 256), 256, 0, st>>>(S, counts, k, d, C_inout);
    return launched();
}

// --------------------------------------------------------------- finalizers
__global__ void finalize_float_kernel(const double *__restrict__ partial,
                                      const int64_t *__restrict__ counts, int k, int d,
                                      float *__restrict__ C) {
    const int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
    if (t >= (int64_t)k * d) return;
    const int j = (int)(t / d);
    const int64_t c = counts[j];
    if (c > 0) C[t] = __double2float_rn(__ddiv_rn(partial[t], (double)c));
}

cudaError_t launch_finalize_float(const double *partial, const int64_t *counts, int k, int d,
                                  float *C_inout, cudaStream_t st) {
    const int64_t tot = (int64_t)k * d;
    finalize_float_kernel<<<(unsigned)((tot + 255) / 256), 256, 0, st>>>(partial, counts, k, d,
                                                                         C_inout);
    return launched();
}

__global__ void finalize_sq8_kernel(const int64_t *__restrict__ partial,
                                    const int64_t *__restrict__ counts, int k, int d,
                                    uint8_t *__restrict__ C) {
    const int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
    if (t >= (int64_t)k * d) return;
    const int j = (int)(t / d);
    const int64_t c = counts[j];
    if (c > 0) C[t] = round_half_even_div(partial[t], c);
}

cudaError_t launch_finalize_sq8(const int64_t *partial, const int64_t *counts, int k, int d,
                                uint8_t *C_inout, cudaStream_t st) {
    const int64_t tot = (int64_t)k * d;
    finalize_sq8_kernel<<<(unsigned)((tot + 255) / 256), 256, 0, st>>>(partial, counts, k, d,
                                                                       C_inout);
    return launched();
}

// One block per cluster: the factor f (one fp64 square root and division) is
// formed once and shared; GB300's fp64 rate makes per-element divisions the
// cost of this step otherwise.
__global__ void finalize_rbq1_kernel(const int64_t *__restrict__ partial,
                                     const int64_t *__restrict__ counts, int k, int d,
                                     const float *__restrict__ m, int e, float *__restrict__ C) {
    __shared__ double fs;
    const int j = blockIdx.x;
    const int64_t c = counts[j];
    if (c <= 0) return;  // block-uniform
    if (threadIdx.x == 0) {
        const double isd = __ddiv_rn(1.0, __dsqrt_rn((double)d));
        fs = __ddiv_rn(__dmul_rn(isd, ldexp(1.0, -e)), (double)c);
    }
    __syncthreads();
    const double f = fs;
    const int64_t *T = partial + (int64_t)j * (d + 1);
    const int64_t U = T[d];
    for (int i = threadIdx.x; i < d; i += blockDim.x) C[(int64_t)j * d + i] = rbq1_finish(T[i], U, m[i], f);
}

cudaError_t launch_finalize_rbq1(const int64_t *partial, const int64_t *counts, int k, int d,
                                 const float *m, int e, float *C_inout, cudaStream_t st) {
    finalize_rbq1_kernel<<<k, 256, 0, st>>>(partial, counts, k, d, m, e, C_inout);
    return launched();
}

__global__ void merge_kernel(void *__restrict__ dst, const void *__restrict__ src, int64_t count,
                             int elem_type) {
    for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < count;
         t += (int64_t)gridDim.x * blockDim.x) {
        if (elem_type == 0)
            reinterpret_cast<double *>(dst)[t] += reinterpret_cast<const double *>(src)[t];
        else
            reinterpret_cast<int64_t *>(dst)[t] += reinterpret_cast<const int64_t *>(src)[t];
    }
}

cudaError_t launch_merge(void *dst, const void *src, int64_t count, int elem_type,
                         cudaStream_t st) {
    if (count == 0) return cudaSuccess;
    int64_t blocks = (count + 255) / 256;
    if (blocks > 152 * 8) blocks = 152 * 8;
    merge_kernel<<<(unsigned)blocks, 256, 0, st>>>(dst, src, count, elem_type);
    return launched();
}

}  // namespace skm

namespace skm {

// ------------------------------------------------------- empty-cluster split
// Section 2.3 STEP 3 (splitting large clusters): clusters left empty by an
// update, in increasing index order, each take the current largest cluster L
// (most members, ties to the lowest index; stop once L has fewer than 2) and
// the two become L's centroid moved by a relative 2^-10 in opposite
// directions, the sign alternating per dimension (fp32), or by one code step
// (SQ8, clipped).  L keeps ceil(n_L/2) members for later choices.  One block.
constexpr int SPLIT_THREADS = 1024;

template <typename T>
__global__ void __launch_bounds__(SPLIT_THREADS) split_empty_kernel(T *__restrict__ C,
                                                                    const int64_t *__restrict__ counts,
                                                                    int k, int d, int64_t *__restrict__ w) {
    __shared__ int64_t sv[SPLIT_THREADS / 32];
    __shared__ int si[SPLIT_THREADS / 32];
    __shared__ int sL;
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    for (int j = tid; j < k; j += SPLIT_THREADS) w[j] = counts[j];
    __syncthreads();
    for (int j = 0; j < k; ++j) {
        if (counts[j] != 0) continue;  // the same for every thread
        // argmax of w, ties to the lowest index
        int64_t bv = -1;
        int bi = 0x7fffffff;
        for (int t = tid; t < k; t += SPLIT_THREADS)
            if (w[t] > bv) {
                bv = w[t];
                bi = t;
            }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const int64_t ov = __shfl_xor_sync(0xffffffffu, bv, o);
            const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
            if (ov > bv || (ov == bv && oi < bi)) {
                bv = ov;
                bi = oi;
            }
        }
        if (lane == 0) {
            sv[wid] = bv;
            si[wid] = bi;
        }
        __syncthreads();
        if (tid == 0) {
            int64_t v = sv[0];
            int L = si[0];
            for (int t = 1; t < SPLIT_THREADS / 32; ++t)
                if (sv[t] > v || (sv[t] == v && si[t] < L)) {
                    v = sv[t];
                    L = si[t];
                }
            sL = v >= 2 ? L : -1;
        }
        __syncthreads();
        const int L = sL;
        if (L < 0) break;  // the same for every thread
        for (int i = tid; i < d; i += SPLIT_THREADS) {
            const T c = C[(int64_t)L * d + i];
            const bool even = (i & 1) == 0;
            if constexpr (sizeof(T) == 1) {
                const int s = even ? 1 : -1;
                const int a = (int)c + s, b = (int)c - s;
                C[(int64_t)j * d + i] = (T)(a < 0 ? 0 : (a > 255 ? 255 : a));
                C[(int64_t)L * d + i] = (T)(b < 0 ? 0 : (b > 255 ? 255 : b));
            } else {
                const float up = 1.0f + 0x1p-10f, dn = 1.0f - 0x1p-10f;
                C[(int64_t)j * d + i] = __fmul_rn(c, even ? up : dn);
                C[(int64_t)L * d + i] = __fmul_rn(c, even ? dn : up);
            }
        }
        if (tid == 0) {
            w[j] = w[L] / 2;
            w[L] -= w[j];
        }
        __syncthreads();
    }
}

cudaError_t launch_split_empty(void *C, int code_bytes, const int64_t *counts, int k, int d,
                               int64_t *w, cudaStream_t st) {
    if (code_bytes == 1)
        split_empty_kernel<uint8_t><<<1, SPLIT_THREADS, 0, st>>>(static_cast<uint8_t *>(C), counts, k, d, w);
    else
        split_empty_kernel<float><<<1, SPLIT_THREADS, 0, st>>>(static_cast<float *>(C), counts, k, d, w);
    return launched();
}

}  // namespace skm

namespace skm {

// ---------------------------------------------------- stable sort by group
// Rows ordered by group, increasing row index within a group (hierarchical
// k-means' fine phase works on the meso clusters in this order, and its
// initial fine centroids are positions inside each group).  Blocks own
// SS_CHUNK consecutive rows: per-block group counts, a column scan over the
// blocks, then each block (one warp, 32 rows at a time in order) places its
// rows with __match_any_sync ranks, so the order is deterministic.
constexpr int SS_CHUNK = 4096;

static __device__ __forceinline__ int clamp_key(int g, int m) { return g < 0 ? 0 : (g >= m ? m - 1 : g); }

__global__ void ss_hist_kernel(const int32_t *__restrict__ key, int64_t n, int m, int32_t *__restrict__ hist) {
    extern __shared__ int32_t h[];
    for (int j = threadIdx.x; j < m; j += blockDim.x) h[j] = 0;
    __syncthreads();
    const int64_t r0 = (int64_t)blockIdx.x * SS_CHUNK, r1 = min(n, r0 + SS_CHUNK);
    for (int64_t r = r0 + threadIdx.x; r < r1; r += blockDim.x) atomicAdd(&h[clamp_key(key[r], m)], 1);
    __syncthreads();
    for (int j = threadIdx.x; j < m; j += blockDim.x) hist[(int64_t)blockIdx.x * m + j] = h[j];
}

// hist[b][j] (counts) -> first sorted position of block b's rows of group j;
// sizes[j] = rows in group j.  One block.
__global__ void ss_scan_kernel(int32_t *__restrict__ hist, int nblk, int m, int32_t *__restrict__ sizes) {
    extern __shared__ int32_t goff[];
    for (int j = threadIdx.x; j < m; j += blockDim.x) {
        int32_t run = 0;
        for (int b = 0; b < nblk; ++b) {
            const int32_t t = hist[(int64_t)b * m + j];
            hist[(int64_t)b * m + j] = run;
            run += t;
        }
        sizes[j] = run;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        int32_t run = 0;
        for (int j = 0; j < m; ++j) {
            goff[j] = run;
            run += sizes[j];
        }
    }
    __syncthreads();
    for (int j = threadIdx.x; j < m; j += blockDim.x)
        for (int b = 0; b < nblk; ++b) hist[(int64_t)b * m + j] += goff[j];
}

__global__ void ss_place_kernel(const int32_t *__restrict__ key, int64_t n, int m,
                                const int32_t *__restrict__ starts, int32_t *__restrict__ perm,
                                int32_t *__restrict__ skey) {
    extern __shared__ int32_t cnt[];
    const int lane = threadIdx.x;  // one warp
    for (int j = lane; j < m; j += 32) cnt[j] = starts[(int64_t)blockIdx.x * m + j];
    __syncwarp();
    const int64_t r0 = (int64_t)blockIdx.x * SS_CHUNK, r1 = min(n, r0 + SS_CHUNK);
    const unsigned lt = (1u << lane) - 1u;
    for (int64_t s = r0; s < r1; s += 32) {
        const int64_t r = s + lane;
        const int g = r < r1 ? clamp_key(key[r], m) : -1;
        const unsigned peers = __match_any_sync(0xffffffffu, g);
        int pos = 0;
        if (g >= 0) pos = cnt[g] + __popc(peers & lt);
        __syncwarp();
        if (g >= 0 && (peers & lt) == 0) cnt[g] += __popc(peers);  // the group's lowest lane
        __syncwarp();
        if (g >= 0) {
            perm[pos] = (int32_t)r;
            skey[pos] = g;
        }
    }
}

cudaError_t launch_stable_sort(const int32_t *key, int64_t n, int m, int32_t *hist, int32_t *sizes,
                               int32_t *perm, int32_t *skey, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    const int nblk = (int)((n + SS_CHUNK - 1) / SS_CHUNK);
    const size_t sm = sizeof(int32_t) * (size_t)m;
    ss_hist_kernel<<<nblk, 256, sm, st>>>(key, n, m, hist);
    cudaError_t e = launched();
    if (e != cudaSuccess) return e;
    ss_scan_kernel<<<1, 1024, sm, st>>>(hist, nblk, m, sizes);
    e = launched();
    if (e != cudaSuccess) return e;
    ss_place_kernel<<<nblk, 32, sm, st>>>(key, n, m, hist, perm, skey);
    return launched();
}

// dst row q = src row perm[q] (rowbytes per row); one warp per row
__global__ void gather_rows_bytes_kernel(const uint8_t *__restrict__ src, int64_t rowbytes,
                                         const int32_t *__restrict__ perm, int64_t n, uint8_t *__restrict__ dst,
                                         int vec16) {
    const int lane = threadIdx.x & 31;
    const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    for (int64_t q = warp; q < n; q += nw) {
        const uint8_t *s = src + (int64_t)perm[q] * rowbytes;
        uint8_t *t = dst + q * rowbytes;
        if (vec16) {
            for (int64_t i = lane; i < rowbytes / 16; i += 32)
                reinterpret_cast<uint4 *>(t)[i] = __ldg(reinterpret_cast<const uint4 *>(s) + i);
        } else {
            for (int64_t i = lane; i < rowbytes; i += 32) t[i] = s[i];
        }
    }
}

cudaError_t launch_gather_rows_bytes(const void *src, int64_t rowbytes, const int32_t *perm, int64_t n,
                                     void *dst, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    const int vec16 = rowbytes % 16 == 0 && ((reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(dst)) & 15) == 0;
    int64_t blocks = (n * 32 + 255) / 256;
    if (blocks > 152 * 16) blocks = 152 * 16;
    gather_rows_bytes_kernel<<<(int)blocks, 256, 0, st>>>(static_cast<const uint8_t *>(src), rowbytes, perm, n,
                                                         static_cast<uint8_t *>(dst), vec16);
    return launched();
}

// out[perm[q]] = in[q] (4-byte values)
__global__ void unpermute_kernel(const int32_t *__restrict__ in, const int32_t *__restrict__ perm, int64_t n,
                                 int32_t *__restrict__ out) {
    for (int64_t q = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; q < n; q += (int64_t)gridDim.x * blockDim.x)
        out[perm[q]] = in[q];
}

cudaError_t launch_unpermute(const void *in, const int32_t *perm, int64_t n, void *out, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    int64_t blocks = (n + 255) / 256;
    if (blocks > 152 * 16) blocks = 152 * 16;
    unpermute_kernel<<<(int)blocks, 256, 0, st>>>(static_cast<const int32_t *>(in), perm, n,
                                                  static_cast<int32_t *>(out));
    return launched();
}

}  // namespace skm
