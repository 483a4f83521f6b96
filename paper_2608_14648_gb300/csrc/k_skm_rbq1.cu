// SuperKMeans with RabitQ codes (Section 3.1 "SuperKMeans"): the squared
// distance splits over dimension segments [0, d1), [d1, d2), [d2, d)
// (d1 = d/8 in whole 32-dimension words, d2 = 2 d1), each estimated with the
// RabitQ estimator of Eq. rabitq_l2 / Eq. final:rabitq and factors of its own;
// after the first and second segment (12.5% and 25% of d) a centroid is
// dropped when its partial estimate D_t exceeds fl32(beta g_t), where beta is
// the full estimate to the row's previous centroid and g_t ADSampling's
// scaled threshold (e_t / d) (1 + eps0 / sqrt(e_t))^2; the survivors' full
// estimates D3 give the argmin (ties to the lowest index).  Every estimate is
// evaluated in the same fp32 operation order as the oracle, so the result is
// the oracle's bit for bit.  CUDA cores: AND + popcount over bit planes.
//
// Assignment kernel: a CTA takes 128 points (16 per warp) and walks the
// centroids in chunks of 128 staged in shared memory (bit planes with a
// padded row stride, so that lanes reading different centroids hit
// different banks).  Per point and chunk, lane l evaluates D1 of centroids
// l, l + 32, l + 64, l + 96; the survivors are gathered across the warp
// (ballots, __fns) into dense passes of 32 in which each lane evaluates D2
// and, if it survives, D3 of one centroid; the warp then keeps the smallest
// (D3, index).
#include "skm_internal.cuh"

namespace skm {
namespace {

constexpr int SEG_PTS = 128;   // points per CTA (16 per warp)
constexpr int SEG_KC = 128;    // centroids per staged chunk
constexpr int SEG_MAXW = 32;   // d <= 1024
constexpr int SEG_WARPS = 8;

__device__ __forceinline__ int seg_of_word(int w, int w1, int w2) { return w < w1 ? 0 : (w < w2 ? 1 : 2); }

// ---------------------------------------------------------------- encode
// One warp per point: per segment ||r_t||^2, ||r_t||_1 (fp64 lane sums, xor
// tree), F_t = fl32(sqrt(d_t) ||r_t||^2 / ||r_t||_1), popx_t.
__global__ void rbq1_seg_encode_kernel(const float *__restrict__ X, int64_t n, int d, const float *__restrict__ m,
                                       int d1, int d2, float *__restrict__ nx2s, float *__restrict__ Fs,
                                       int32_t *__restrict__ popxs) {
    const int lane = threadIdx.x & 31;
    const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    for (int64_t row = warp; row < n; row += nw) {
        double s2[3] = {0.0, 0.0, 0.0}, s1[3] = {0.0, 0.0, 0.0};
        int pc[3] = {0, 0, 0};
        for (int i = lane; i < d; i += 32) {
            const float r = __fsub_rn(X[row * d + i], m[i]);
            const int t = i < d1 ? 0 : (i < d2 ? 1 : 2);
            const double rd = (double)r;
#pragma unroll
            for (int u = 0; u < 3; ++u)
                if (u == t) {
                    s2[u] = __dadd_rn(s2[u], __dmul_rn(rd, rd));
                    s1[u] = __dadd_rn(s1[u], fabs(rd));
                    pc[u] += r > 0.0f;
                }
        }
#pragma unroll
        for (int u = 0; u < 3; ++u)
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                s2[u] = __dadd_rn(s2[u], __shfl_xor_sync(0xffffffffu, s2[u], o));
                s1[u] = __dadd_rn(s1[u], __shfl_xor_sync(0xffffffffu, s1[u], o));
                pc[u] += __shfl_xor_sync(0xffffffffu, pc[u], o);
            }
        if (lane < 3) {
            const int t = lane;
            const int dt = t == 0 ? d1 : (t == 1 ? d2 - d1 : d - d2);
            const double a2 = t == 0 ? s2[0] : (t == 1 ? s2[1] : s2[2]);
            const double a1 = t == 0 ? s1[0] : (t == 1 ? s1[1] : s1[2]);
            nx2s[row * 3 + t] = __double2float_rn(a2);
            Fs[row * 3 + t] = a1 > 0.0 ? __double2float_rn(__ddiv_rn(__dmul_rn(__dsqrt_rn((double)dt), a2), a1)) : 0.0f;
            popxs[row * 3 + t] = t == 0 ? pc[0] : (t == 1 ? pc[1] : pc[2]);
        }
    }
}

// ----------------------------------------------------------- centroid prep
// One warp per centroid: SQ4 codes of rho = c - m as four bit planes per
// word (the codes of launch_rbq1_cprep), and per segment the code sum and
// ||rho_t||^2 (pairwise inside each 32-dimension block, blocks in order).
constexpr int SEG_CPREP_WARPS = 4;
__global__ void __launch_bounds__(SEG_CPREP_WARPS * 32) rbq1_seg_cprep_kernel(
    const float *__restrict__ C, int k, int d, const float *__restrict__ m, int d1, int d2, float isd0, float isd1,
    float isd2, uint4 *__restrict__ planes, Rbq1SegInfo *__restrict__ info) {
    extern __shared__ float seg_rho[];  // [SEG_CPREP_WARPS][d]
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int j = blockIdx.x * SEG_CPREP_WARPS + warp;
    if (j >= k) return;  // warp-uniform
    float *rho = seg_rho + (size_t)warp * d;
    const float *c = C + (int64_t)j * d;
    float lo = INFINITY, hi = -INFINITY;
    for (int i = lane; i < d; i += 32) {
        const float r = __fsub_rn(c[i], m[i]);
        rho[i] = r;
        lo = fminf(lo, r);
        hi = fmaxf(hi, r);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, o));
        hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, o));
    }
    __syncwarp();
    float sc = __fdiv_rn(__fsub_rn(hi, lo), 15.0f);
    if (!(sc > 0.0f)) sc = 1.0f;
    const int W = (d + 31) >> 5, w1 = d1 >> 5, w2 = d2 >> 5;
    int32_t sy[3] = {0, 0, 0};
    double q2[3] = {0.0, 0.0, 0.0};
    for (int w = 0; w < W; ++w) {
        const int i = 32 * w + lane;
        const int t = seg_of_word(w, w1, w2);
        double sq = (i < d) ? __dmul_rn((double)rho[i], (double)rho[i]) : 0.0;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) sq = __dadd_rn(sq, __shfl_xor_sync(0xffffffffu, sq, o));
        uint32_t y = 0;
        if (i < d) {
            float q = rintf(__fdiv_rn(__fsub_rn(rho[i], lo), sc));
            q = (q >= 0.0f) ? q : 0.0f;
            q = fminf(q, 15.0f);
            y = (uint32_t)q;
        }
#pragma unroll
        for (int u = 0; u < 3; ++u)
            if (u == t) {
                q2[u] = __dadd_rn(q2[u], sq);
                sy[u] += (int32_t)y;
            }
        const uint32_t p0 = __ballot_sync(0xffffffffu, y & 1u);
        const uint32_t p1 = __ballot_sync(0xffffffffu, y & 2u);
        const uint32_t p2 = __ballot_sync(0xffffffffu, y & 4u);
        const uint32_t p3 = __ballot_sync(0xffffffffu, y & 8u);
        if (lane == 0) planes[(int64_t)j * W + w] = make_uint4(p0, p1, p2, p3);
    }
#pragma unroll
    for (int u = 0; u < 3; ++u)
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) sy[u] += __shfl_xor_sync(0xffffffffu, sy[u], o);
    if (lane == 0) {
        Rbq1SegInfo in;
        const float isd[3] = {isd0, isd1, isd2};
#pragma unroll
        for (int u = 0; u < 3; ++u) {
            in.bd[u] = __fmul_rn(lo, isd[u]);
            in.sd[u] = __fmul_rn(sc, isd[u]);
            in.ny2[u] = __double2float_rn(q2[u]);
            in.sumy[u] = sy[u];
        }
        info[j] = in;
    }
}

// ------------------------------------------------------------- assignment
struct SegRow {  // one point's factors
    float nx2[3], f2[3], pc[3];
};

// Segment t's estimate from its integer P_t (the library's fp32 order).
__device__ __forceinline__ float seg_est(int P, const Rbq1SegInfo &ci, const SegRow &r, int t) {
    const float u = __fmaf_rn(ci.sd[t], __int2float_rn(2 * P - ci.sumy[t]), __fmul_rn(ci.bd[t], r.pc[t]));
    return __fmaf_rn(r.f2[t], u, __fadd_rn(r.nx2[t], ci.ny2[t]));
}

// P over words [w0, w1) of the point (xw, in registers) and one centroid's
// planes (shared memory, stride words).
__device__ __forceinline__ int seg_P(const uint32_t (&xw)[SEG_MAXW], const uint4 *pl, int w0, int w1) {
    int P = 0;
#pragma unroll
    for (int w = 0; w < SEG_MAXW; ++w) {
        if (w >= w0 && w < w1) {
            const uint4 y = pl[w];
            P += __popc(xw[w] & y.x) + 2 * __popc(xw[w] & y.y) + 4 * __popc(xw[w] & y.z) + 8 * __popc(xw[w] & y.w);
        }
    }
    return P;
}

__global__ void __launch_bounds__(SEG_WARPS * 32) assign_rbq1_seg_kernel(
    const uint32_t *__restrict__ codes, const float *__restrict__ nx2s, const float *__restrict__ Fs,
    const int32_t *__restrict__ popxs, int64_t n, int d, int d1, int d2, const uint4 *__restrict__ planes,
    const Rbq1SegInfo *__restrict__ info, int k, const int32_t *__restrict__ prev, float g0, float g1,
    int32_t *__restrict__ assign, float *__restrict__ dist, unsigned long long *__restrict__ counters) {
    extern __shared__ __align__(16) unsigned char seg_smem[];
    const int W = (d + 31) >> 5, w1 = d1 >> 5, w2 = d2 >> 5;
    const int PS = W + 1;  // padded plane row stride (uint4), conflict-free lane-varying rows
    uint4 *cpl = reinterpret_cast<uint4 *>(seg_smem);                           // [SEG_KC][PS]
    Rbq1SegInfo *cinf = reinterpret_cast<Rbq1SegInfo *>(cpl + (size_t)SEG_KC * PS);  // [SEG_KC]
    uint32_t *xs = reinterpret_cast<uint32_t *>(cinf + SEG_KC);                 // [SEG_PTS][W]
    float *s_beta = reinterpret_cast<float *>(xs + (size_t)SEG_PTS * W);        // [SEG_PTS]
    float *s_best = s_beta + SEG_PTS;
    int32_t *s_bi = reinterpret_cast<int32_t *>(s_best + SEG_PTS);
    int32_t *s_seed = s_bi + SEG_PTS;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t p0 = (int64_t)blockIdx.x * SEG_PTS;
    const int np = (int)min((int64_t)SEG_PTS, n - p0);
    unsigned long long alive1 = 0, alive2 = 0;
    for (int e = threadIdx.x; e < SEG_PTS * W; e += blockDim.x) {
        const int q = e / W, w = e - q * W;
        xs[e] = q < np ? codes[(p0 + q) * W + w] : 0u;
    }
    __syncthreads();
    // the bound: D3 of each point's seed centroid (lanes over words)
    for (int q = warp; q < np; q += SEG_WARPS) {
        const int64_t p = p0 + q;
        int seed = prev ? prev[p] : 0;
        if (seed < 0 || seed >= k) seed = 0;
        int P[3] = {0, 0, 0};
        if (lane < W) {
            const uint32_t x = xs[q * W + lane];
            const uint4 y = planes[(int64_t)seed * W + lane];
            const int v = __popc(x & y.x) + 2 * __popc(x & y.y) + 4 * __popc(x & y.z) + 8 * __popc(x & y.w);
            const int t = seg_of_word(lane, w1, w2);
            P[0] = t == 0 ? v : 0;
            P[1] = t == 1 ? v : 0;
            P[2] = t == 2 ? v : 0;
        }
#pragma unroll
        for (int u = 0; u < 3; ++u)
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) P[u] += __shfl_xor_sync(0xffffffffu, P[u], o);
        if (lane == 0) {
            SegRow r;
#pragma unroll
            for (int u = 0; u < 3; ++u) {
                r.nx2[u] = nx2s[p * 3 + u];
                r.f2[u] = __fmul_rn(-2.0f, Fs[p * 3 + u]);
                const int dt = u == 0 ? d1 : (u == 1 ? d2 - d1 : d - d2);
                r.pc[u] = __int2float_rn(2 * popxs[p * 3 + u] - dt);
            }
            const Rbq1SegInfo ci = info[seed];
            const float D1 = seg_est(P[0], ci, r, 0);
            const float D2 = __fadd_rn(D1, seg_est(P[1], ci, r, 1));
            const float D3 = __fadd_rn(D2, seg_est(P[2], ci, r, 2));
            s_beta[q] = D3;
            s_best[q] = INFINITY;
            s_bi[q] = 0x7fffffff;
            s_seed[q] = seed;
        }
    }
    for (int c0 = 0; c0 < k; c0 += SEG_KC) {
        const int kc = min(SEG_KC, k - c0);
        __syncthreads();  // the previous chunk's planes and the state writes are done
        for (int e = threadIdx.x; e < kc * W; e += blockDim.x) {
            const int c = e / W, w = e - c * W;
            cpl[c * PS + w] = planes[(int64_t)(c0 + c) * W + w];
        }
        for (int c = threadIdx.x; c < kc; c += blockDim.x) cinf[c] = info[c0 + c];
        __syncthreads();
        for (int q = warp; q < np; q += SEG_WARPS) {
            const int64_t p = p0 + q;
            uint32_t xw[SEG_MAXW];
#pragma unroll
            for (int w = 0; w < SEG_MAXW; ++w) xw[w] = w < W ? xs[q * W + w] : 0u;  // broadcast reads
            SegRow r;
#pragma unroll
            for (int u = 0; u < 3; ++u) {
                r.nx2[u] = nx2s[p * 3 + u];
                r.f2[u] = __fmul_rn(-2.0f, Fs[p * 3 + u]);
                const int dt = u == 0 ? d1 : (u == 1 ? d2 - d1 : d - d2);
                r.pc[u] = __int2float_rn(2 * popxs[p * 3 + u] - dt);
            }
            const float beta = s_beta[q];
            const float t0 = __fmul_rn(beta, g0), t1 = __fmul_rn(beta, g1);
            const int seed = s_seed[q];
            // checkpoint 1 for the chunk: lane owns centroids lane + 32 s
            float D1v[4];
            unsigned M[4];
#pragma unroll
            for (int s = 0; s < 4; ++s) {
                const int c = 32 * s + lane;
                bool keep = false;
                D1v[s] = 0.0f;
                if (c < kc) {
                    D1v[s] = seg_est(seg_P(xw, cpl + c * PS, 0, w1), cinf[c], r, 0);
                    keep = (c0 + c == seed) || !(D1v[s] > t0);
                }
                M[s] = __ballot_sync(0xffffffffu, keep);
            }
            const int n0 = __popc(M[0]), n1 = __popc(M[1]), n2 = __popc(M[2]), n3 = __popc(M[3]);
            const int total = n0 + n1 + n2 + n3;
            alive1 += lane == 0 ? (unsigned long long)total : 0ull;
            float best = INFINITY;
            int bi = 0x7fffffff;
            for (int base = 0; base < total; base += 32) {
                const int i = base + lane;
                // the i-th survivor: its slot, owner lane and D1
                int slot, rank;
                if (i < n0) {
                    slot = 0;
                    rank = i;
                } else if (i < n0 + n1) {
                    slot = 1;
                    rank = i - n0;
                } else if (i < n0 + n1 + n2) {
                    slot = 2;
                    rank = i - n0 - n1;
                } else {
                    slot = 3;
                    rank = i - n0 - n1 - n2;
                }
                const unsigned ms = slot == 0 ? M[0] : (slot == 1 ? M[1] : (slot == 2 ? M[2] : M[3]));
                const int owner = i < total ? (int)__fns(ms, 0, rank + 1) : 0;
                float d1v = 0.0f;
#pragma unroll
                for (int s = 0; s < 4; ++s) {
                    const float v = __shfl_sync(0xffffffffu, D1v[s], owner & 31);
                    d1v = s == slot ? v : d1v;
                }
                if (i < total) {
                    const int c = 32 * slot + owner;
                    const int j = c0 + c;
                    const uint4 *pl = cpl + c * PS;
                    const Rbq1SegInfo ci = cinf[c];
                    const float D2 = __fadd_rn(d1v, seg_est(seg_P(xw, pl, w1, w2), ci, r, 1));
                    if (j == seed || !(D2 > t1)) {
                        ++alive2;
                        const float D3 = __fadd_rn(D2, seg_est(seg_P(xw, pl, w2, W), ci, r, 2));
                        if (D3 < best || (D3 == best && j < bi)) {
                            best = D3;
                            bi = j;
                        }
                    }
                }
            }
            // the warp's smallest (D3, index), merged into the point's state
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                const float ob = __shfl_xor_sync(0xffffffffu, best, o);
                const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
                if (ob < best || (ob == best && oi < bi)) {
                    best = ob;
                    bi = oi;
                }
            }
            if (lane == 0 && (best < s_best[q] || (best == s_best[q] && bi < s_bi[q]))) {
                s_best[q] = best;
                s_bi[q] = bi;
            }
        }
    }
    __syncthreads();
    for (int q = threadIdx.x; q < np; q += blockDim.x) {
        assign[p0 + q] = s_bi[q];
        if (dist) dist[p0 + q] = s_best[q];
    }
    if (counters) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) alive2 += __shfl_xor_sync(0xffffffffu, alive2, o);
        if (lane == 0) {
            atomicAdd(&counters[0], alive1);
            atomicAdd(&counters[1], alive2);
        }
    }
}

}  // namespace

void rbq1_seg_bounds(int d, int *d1, int *d2) {
    int w = (d + 128) / 256;
    if (w < 1) w = 1;
    *d1 = 32 * w;
    *d2 = 2 * (*d1);
}

void rbq1_seg_factors(int d, int d1, int d2, float *g) {
    const int e[2] = {d1, d2};
    for (int t = 0; t < 2; ++t) {
        const double a = 1.0 + SEG_EPS0 / sqrt((double)e[t]);
        g[t] = (float)(((double)e[t] / (double)d) * a * a);
    }
}

cudaError_t launch_rbq1_seg_encode(const float *X, int64_t n, int d, const float *m, float *nx2s, float *Fs,
                                   int32_t *popxs, cudaStream_t st) {
    int d1, d2;
    rbq1_seg_bounds(d, &d1, &d2);
    int64_t blocks = (n * 32 + 255) / 256;
    blocks = blocks < 1 ? 1 : (blocks > 152 * 16 ? 152 * 16 : blocks);
    rbq1_seg_encode_kernel<<<(unsigned)blocks, 256, 0, st>>>(X, n, d, m, d1, d2, nx2s, Fs, popxs);
    return launched();
}

cudaError_t launch_rbq1_seg_cprep(const float *C, int k, int d, const float *m, uint4 *planes, Rbq1SegInfo *info,
                                  cudaStream_t st) {
    int d1, d2;
    rbq1_seg_bounds(d, &d1, &d2);
    const float i0 = (float)(1.0 / sqrt((double)d1)), i1 = (float)(1.0 / sqrt((double)(d2 - d1))),
                i2 = (float)(1.0 / sqrt((double)(d - d2)));
    const size_t smem = (size_t)SEG_CPREP_WARPS * d * sizeof(float);
    if (smem > 48 * 1024) {
        const cudaError_t e =
            cudaFuncSetAttribute(rbq1_seg_cprep_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
    }
    rbq1_seg_cprep_kernel<<<(k + SEG_CPREP_WARPS - 1) / SEG_CPREP_WARPS, SEG_CPREP_WARPS * 32, smem, st>>>(
        C, k, d, m, d1, d2, i0, i1, i2, planes, info);
    return launched();
}

cudaError_t launch_assign_rbq1_seg(const uint32_t *codes, const float *nx2s, const float *Fs, const int32_t *popxs,
                                   int64_t n, int d, const uint4 *planes, const Rbq1SegInfo *info, int k,
                                   const int32_t *prev, int32_t *assign, float *dist, unsigned long long *counters,
                                   cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    int d1, d2;
    rbq1_seg_bounds(d, &d1, &d2);
    float g[2];
    rbq1_seg_factors(d, d1, d2, g);
    const int W = (d + 31) >> 5;
    const size_t smem = (size_t)SEG_KC * (W + 1) * sizeof(uint4) + (size_t)SEG_KC * sizeof(Rbq1SegInfo) +
                        (size_t)SEG_PTS * W * sizeof(uint32_t) + (size_t)SEG_PTS * 16;
    const cudaError_t e =
        cudaFuncSetAttribute(assign_rbq1_seg_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int64_t blocks = (n + SEG_PTS - 1) / SEG_PTS;
    assign_rbq1_seg_kernel<<<(unsigned)blocks, SEG_WARPS * 32, smem, st>>>(
        codes, nx2s, Fs, popxs, n, d, d1, d2, planes, info, k, prev, g[0], g[1], assign, dist, counters);
    return launched();
}

}  // namespace skm
