// RabitQ 1-bit assignment (Section 3.1 "RabitQ", Eq. rabitq_l2 with
// Eq. final:rabitq): the highlighted sum P = sum_i xbar_i ybar_i of a 1-bit
// point code against a 4-bit centroid code is computed exactly as
// P = sum_w sum_j 2^j popc(xbar_w & plane_j,w) with AND + POPC on packed
// 32-bit words; the distance estimate follows in fp32 in the fixed order
//   u = fma(sd, 2P - sumy, bd (2 popx - d)),  est = fma(-2 F, u, nx2 + ny2)
// (sd, bd: the centroid's SQ4 scale and bias times fl(1/sqrt d)), and the
// argmin keeps the lowest index on ties.
//
// One thread per point; the point's code words live in shared memory
// (transposed, conflict-free), centroid bit planes are staged per chunk and
// read as warp-wide broadcasts.  Four centroids are evaluated per pass over
// the words so each x word is loaded once per four centroids.
#include "skm_internal.cuh"

namespace skm {

constexpr int RBQ1_THREADS = 128;

__device__ __forceinline__ int plane_dot(uint32_t x, uint4 y) {
    return __popc(x & y.x) + 2 * __popc(x & y.y) + 4 * __popc(x & y.z) + 8 * __popc(x & y.w);
}

__device__ __forceinline__ float rbq1_estimate(int P, const Rbq1CInfo &ci, float nx2, float f2,
                                               float pc) {
    const float u = __fmaf_rn(ci.sd, __int2float_rn(2 * P - ci.sumy), __fmul_rn(ci.bd, pc));
    return __fmaf_rn(f2, u, __fadd_rn(nx2, ci.ny2));
}

__global__ void __launch_bounds__(RBQ1_THREADS) assign_rbq1_kernel(
    const uint32_t *__restrict__ codes, const float *__restrict__ nx2, const float *__restrict__ F,
    const int32_t *__restrict__ popx, int64_t n, int d, const uint4 *__restrict__ planes,
    const Rbq1CInfo *__restrict__ info, int k, int kc, int32_t *__restrict__ assign,
    float *__restrict__ dist) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int W = (d + 31) >> 5;
    uint4 *ps = reinterpret_cast<uint4 *>(smem_raw);                     // [kc][W]
    Rbq1CInfo *is = reinterpret_cast<Rbq1CInfo *>(ps + (size_t)kc * W);  // [kc]
    uint32_t *xs = reinterpret_cast<uint32_t *>(is + kc);                 // [W][THREADS]

    const int tid = threadIdx.x;
    const int64_t p = (int64_t)blockIdx.x * RBQ1_THREADS + tid;
    const bool valid = p < n;
    // stage this block's point codes transposed: xs[w][t]
    for (int e = tid; e < W * RBQ1_THREADS; e += RBQ1_THREADS) {
        const int t = e / W, w = e - t * W;
        const int64_t q = (int64_t)blockIdx.x * RBQ1_THREADS + t;
        xs[w * RBQ1_THREADS + t] = (q < n) ? codes[q * W + w] : 0u;
    }
    const float my_nx2 = valid ? nx2[p] : 0.0f;
    const float my_f2 = valid ? __fmul_rn(-2.0f, F[p]) : 0.0f;  // exact
    const float my_pc = valid ? __int2float_rn(2 * popx[p] - d) : 0.0f;

    float best = INFINITY;
    int besti = 0;
    for (int c0 = 0; c0 < k; c0 += kc) {
        const int cn = min(kc, k - c0);
        __syncthreads();
        for (int e = tid; e < cn * W; e += RBQ1_THREADS) ps[e] = planes[(int64_t)c0 * W + e];
        for (int e = tid; e < cn; e += RBQ1_THREADS) is[e] = info[c0 + e];
        __syncthreads();
        int j = 0;
        for (; j + 4 <= cn; j += 4) {
            int P0 = 0, P1 = 0, P2 = 0, P3 = 0;
            const uint4 *p0 = ps + (size_t)j * W;
            for (int w = 0; w < W; ++w) {
                const uint32_t xw = xs[w * RBQ1_THREADS + tid];
                P0 += plane_dot(xw, p0[w]);
                P1 += plane_dot(xw, p0[W + w]);
                P2 += plane_dot(xw, p0[2 * W + w]);
                P3 += plane_dot(xw, p0[3 * W + w]);
            }
            const int Ps[4] = {P0, P1, P2, P3};
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const float est = rbq1_estimate(Ps[q], is[j + q], my_nx2, my_f2, my_pc);
                if (est < best) {
                    best = est;
                    besti = c0 + j + q;
                }
            }
        }
        for (; j < cn; ++j) {
            int P = 0;
            const uint4 *pj = ps + (size_t)j * W;
            for (int w = 0; w < W; ++w) P += plane_dot(xs[w * RBQ1_THREADS + tid], pj[w]);
            const float est = rbq1_estimate(P, is[j], my_nx2, my_f2, my_pc);
            if (est < best) {
                best = est;
                besti = c0 + j;
            }
        }
    }
    if (valid) {
        assign[p] = besti;
        if (dist) dist[p] = best;
    }
}

// Symmetric variant (binarized centroids): Hamming distance h by XOR + POPC,
// est = fma(-2 F, fy (d - 2h), nx2 + ny2) in that fp32 order.  One thread per
// point; tiles of SYM_KT centroids' sign words in shared memory (broadcast
// reads), the point's words from global memory (L1-resident across a tile).
constexpr int SYM_KT = 32;
__global__ void __launch_bounds__(RBQ1_THREADS) assign_rbq1_sym_kernel(
    const uint32_t *__restrict__ codes, const float *__restrict__ nx2, const float *__restrict__ F, int64_t n, int d,
    const uint32_t *__restrict__ yw, const Rbq1CInfo *__restrict__ info, int k, int32_t *__restrict__ assign,
    float *__restrict__ dist) {
    extern __shared__ uint32_t sy[];  // [SYM_KT][W]
    const int W = (d + 31) >> 5;
    const int64_t p = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
    const bool valid = p < n;
    const uint32_t *xr = codes + (valid ? p : 0) * W;
    const float f2 = valid ? __fmul_rn(-2.0f, F[p]) : 0.0f;
    const float xn = valid ? nx2[p] : 0.0f;
    float best = INFINITY;
    int32_t besti = 0;
    for (int j0 = 0; j0 < k; j0 += SYM_KT) {
        __syncthreads();
        for (int t = threadIdx.x; t < SYM_KT * W; t += blockDim.x) {
            const int c = t / W, w = t - c * W;
            sy[t] = (j0 + c < k) ? yw[(int64_t)(j0 + c) * W + w] : 0u;
        }
        __syncthreads();
        if (!valid) continue;
        int h[SYM_KT];
#pragma unroll
        for (int c = 0; c < SYM_KT; ++c) h[c] = 0;
        for (int w = 0; w < W; ++w) {
            const uint32_t xw = xr[w];
#pragma unroll
            for (int c = 0; c < SYM_KT; ++c) h[c] += __popc(xw ^ sy[c * W + w]);
        }
#pragma unroll
        for (int c = 0; c < SYM_KT; ++c) {
            const int j = j0 + c;
            if (j < k) {
                const Rbq1CInfo in = info[j];
                const float u = __fmul_rn(in.sd, __int2float_rn(d - 2 * h[c]));
                const float est = __fmaf_rn(f2, u, __fadd_rn(xn, in.ny2));
                if (est < best) {
                    best = est;
                    besti = j;
                }
            }
        }
    }
    if (valid) {
        assign[p] = besti;
        if (dist) dist[p] = best;
    }
}

cudaError_t launch_assign_rbq1_sym(const uint32_t *codes, const float *nx2, const float *F, int64_t n, int d,
                                   const uint32_t *yw, const Rbq1CInfo *info, int k, int32_t *assign, float *dist,
                                   cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    const size_t smem = (size_t)SYM_KT * ((d + 31) >> 5) * sizeof(uint32_t);
    if (smem > 48 * 1024) {
        const cudaError_t e =
            cudaFuncSetAttribute(assign_rbq1_sym_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
    }
    assign_rbq1_sym_kernel<<<(unsigned)((n + RBQ1_THREADS - 1) / RBQ1_THREADS), RBQ1_THREADS, smem, st>>>(
        codes, nx2, F, n, d, yw, info, k, assign, dist);
    return launched();
}

cudaError_t launch_assign_rbq1(const uint32_t *codes, const float *nx2, const float *F,
                               const int32_t *popx, int64_t n, int d, const uint4 *planes,
                               const Rbq1CInfo *info, int k, int32_t *assign, float *dist,
                               cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    const int W = (d + 31) >> 5;
    const size_t xs_bytes = (size_t)W * RBQ1_THREADS * 4;
    const size_t per_c = (size_t)W * 16 + sizeof(Rbq1CInfo);
    const size_t budget = 96 * 1024;
    int kc = (int)((budget > xs_bytes ? budget - xs_bytes : per_c) / per_c);
    kc = max(4, min(kc, 256));
    kc = min(kc, max(4, k));
    const size_t smem = (size_t)kc * per_c + xs_bytes + 16;
    cudaError_t e = cudaFuncSetAttribute(assign_rbq1_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    assign_rbq1_kernel<<<(unsigned)((n + RBQ1_THREADS - 1) / RBQ1_THREADS), RBQ1_THREADS, smem,
                         st>>>(codes, nx2, F, popx, n, d, planes, info, k, kc, assign, dist);
    return launched();
}

}  // namespace skm
