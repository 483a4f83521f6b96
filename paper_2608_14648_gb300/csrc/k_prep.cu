// Per-iteration centroid preparation.
//  RBQ1 (Section 3.1 "RabitQ"): the centroid residual rho = c - m is
//  re-encoded with per-centroid SQ4 (b = min rho, s = (max rho - b)/15,
//  s = 1 when flat, ybar = clip(rint((rho - b)/s), 0, 15)) and stored as four
//  bit planes per 32-dimension word, so that sum_i xbar_i ybar_i =
//  sum_j 2^j popc(xbar & plane_j).  One thread per centroid walks its row in
//  order, which fixes the fp64 summation order of ||rho||^2.
//  SQ8: per-row sums of squared codes (exact int32).
#include "skm_internal.cuh"

namespace skm {

__global__ void rbq1_cprep_kernel(const float *__restrict__ C, int k, int d,
                                  const float *__restrict__ m, uint4 *__restrict__ planes,
                                  Rbq1CInfo *__restrict__ info) {
    const int j = blockIdx.x * blockDim.x + threadIdx.x;
    if (j >= k) return;
    const float *c = C + (int64_t)j * d;
    float lo = INFINITY, hi = -INFINITY;
    double q2 = 0.0;
    for (int i = 0; i < d; ++i) {
        const float r = __fsub_rn(c[i], m[i]);
        lo = fminf(lo, r);
        hi = fmaxf(hi, r);
        q2 = __dadd_rn(q2, __dmul_rn((double)r, (double)r));
    }
    float sc = __fdiv_rn(__fsub_rn(hi, lo), 15.0f);
    if (!(sc > 0.0f)) sc = 1.0f;
    const int W = (d + 31) >> 5;
    int32_t sy = 0;
    for (int w = 0; w < W; ++w) {
        uint32_t p0 = 0, p1 = 0, p2 = 0, p3 = 0;
        for (int l = 0; l < 32; ++l) {
            const int i = 32 * w + l;
            if (i >= d) break;
            const float r = __fsub_rn(c[i], m[i]);
            float q = rintf(__fdiv_rn(__fsub_rn(r, lo), sc));
            q = (q >= 0.0f) ? q : 0.0f;
            q = fminf(q, 15.0f);
            const uint32_t y = (uint32_t)q;
            sy += (int32_t)y;
            p0 |= (y & 1u) << l;
            p1 |= ((y >> 1) & 1u) << l;
            p2 |= ((y >> 2) & 1u) << l;
            p3 |= ((y >> 3) & 1u) << l;
        }
        planes[(int64_t)j * W + w] = make_uint4(p0, p1, p2, p3);
    }
    Rbq1CInfo in;
    in.b = lo;
    in.s = sc;
    in.sumy = sy;
    in.ny2 = __double2float_rn(q2);
    info[j] = in;
}

cudaError_t launch_rbq1_cprep(const float *C, int k, int d, const float *m, uint4 *planes,
                              Rbq1CInfo *info, cudaStream_t st) {
    rbq1_cprep_kernel<<<(k + 63) / 64, 64, 0, st>>>(C, k, d, m, planes, info);
    return launched();
}

// sum_i code_i^2 per row (exact, fits int32 for d <= 4096); one warp per row.
__global__ void row_sqnorm_u8_kernel(const uint8_t *__restrict__ codes, int64_t n, int d,
                                     int32_t *__restrict__ out) {
    const int lane = threadIdx.x & 31;
    const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
    for (int64_t p = warp; p < n; p += nwarps) {
        int32_t s = 0;
        for (int i = lane; i < d; i += 32) {
            const int32_t v = codes[p * d + i];
            s += v * v;
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
        if (lane == 0) out[p] = s;
    }
}

cudaError_t launch_row_sqnorm_u8(const uint8_t *codes, int64_t n, int d, int32_t *out,
                                 cudaStream_t st) {
    int64_t blocks = (n * 32 + 255) / 256;
    if (blocks > 152 * 16) blocks = 152 * 16;
    if (blocks < 1) blocks = 1;
    row_sqnorm_u8_kernel<<<(int)blocks, 256, 0, st>>>(codes, n, d, out);
    return launched();
}

}  // namespace skm
