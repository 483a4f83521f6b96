// Per-iteration centroid preparation.
//  RBQ1 (Section 3.1 "RabitQ"): the centroid residual rho = c - m is
//  re-encoded with per-centroid SQ4 (b = min rho, s = (max rho - b)/15,
//  s = 1 when flat, ybar = clip(rint((rho - b)/s), 0, 15)) and stored as four
//  bit planes per 32-dimension word, so that sum_i xbar_i ybar_i =
//  sum_j 2^j popc(xbar & plane_j), and/or as e4m3 bytes for the tensor kernel.
//  ||rho||^2 is summed in fp64 in the library's blocked pairwise order.
//  SQ8: per-row sums of squared codes (exact int32).
#include "skm_internal.cuh"

namespace skm {

// One warp per centroid.  rho = c - m is kept in the warp's slice of shared
// memory; min/max and the code sum are exact warp reductions, the codes of
// 32 consecutive dimensions become four bit planes through __ballot_sync, and
// ||rho||^2 is summed in fp64 pairwise inside each 32-dimension block (xor
// butterfly 16, 8, 4, 2, 1) with the block sums added in order.
constexpr int CPREP_WARPS = 4;

// planes != nullptr: SQ4 codes as four bit planes per word (AND + popcount
// kernel); yq != nullptr: the same codes as e4m3 bytes, row stride dq (tensor
// kernel).
__global__ void __launch_bounds__(CPREP_WARPS * 32) rbq1_cprep_kernel(
    const float *__restrict__ C, int k, int d, const float *__restrict__ m,
    uint4 *__restrict__ planes, Rbq1CInfo *__restrict__ info, uint8_t *__restrict__ yq, int dq,
    float isd) {
    extern __shared__ float sh_rho[];  // [CPREP_WARPS][d]
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int j = blockIdx.x * CPREP_WARPS + warp;
    if (j >= k) return;  // warp-uniform
    float *rho = sh_rho + (size_t)warp * d;
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
    const int W = (d + 31) >> 5;
    int32_t sy = 0;
    double q2 = 0.0;  // ||rho||^2: pairwise within 32-dim blocks, blocks in order
    for (int w = 0; w < W; ++w) {
        const int i = 32 * w + lane;
        double sq = (i < d) ? __dmul_rn((double)rho[i], (double)rho[i]) : 0.0;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) sq = __dadd_rn(sq, __shfl_xor_sync(0xffffffffu, sq, o));
        q2 = __dadd_rn(q2, sq);
        uint32_t y = 0;
        if (i < d) {
            float q = rintf(__fdiv_rn(__fsub_rn(rho[i], lo), sc));
            q = (q >= 0.0f) ? q : 0.0f;
            q = fminf(q, 15.0f);
            y = (uint32_t)q;
            if (yq) yq[(int64_t)j * dq + i] = e4m3_of_code(y);
        }
        sy += (int32_t)y;
        const uint32_t p0 = __ballot_sync(0xffffffffu, y & 1u);
        const uint32_t p1 = __ballot_sync(0xffffffffu, y & 2u);
        const uint32_t p2 = __ballot_sync(0xffffffffu, y & 4u);
        const uint32_t p3 = __ballot_sync(0xffffffffu, y & 8u);
        if (planes && lane == 0) planes[(int64_t)j * W + w] = make_uint4(p0, p1, p2, p3);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sy += __shfl_xor_sync(0xffffffffu, sy, o);
    if (lane == 0) {
        Rbq1CInfo in;
        in.bd = __fmul_rn(lo, isd);
        in.sd = __fmul_rn(sc, isd);
        in.sumy = sy;
        in.ny2 = __double2float_rn(q2);
        info[j] = in;
    }
}

static cudaError_t launch_cprep_common(const float *C, int k, int d, const float *m, uint4 *planes,
                                       Rbq1CInfo *info, uint8_t *yq, int dq, cudaStream_t st) {
    const size_t smem = (size_t)CPREP_WARPS * d * sizeof(float);
    if (smem > 48 * 1024) {
        const cudaError_t e = cudaFuncSetAttribute(
            rbq1_cprep_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
    }
    rbq1_cprep_kernel<<<(k + CPREP_WARPS - 1) / CPREP_WARPS, CPREP_WARPS * 32, smem, st>>>(
        C, k, d, m, planes, info, yq, dq, rbq1_isd(d));
    return launched();
}

cudaError_t launch_rbq1_cprep(const float *C, int k, int d, const float *m, uint4 *planes,
                              Rbq1CInfo *info, cudaStream_t st) {
    return launch_cprep_common(C, k, d, m, planes, info, nullptr, 0, st);
}

cudaError_t launch_rbq1_cprep_tc(const float *C, int k, int d, const float *m, uint8_t *yq, int dq,
                                 Rbq1CInfo *info, cudaStream_t st) {
    return launch_cprep_common(C, k, d, m, nullptr, info, yq, dq, st);
}

// Symmetric 1-bit variant: the centroid residual rho = c - m binarized like a
// point (bit = rho_i > 0); ||rho||^2 and ||rho||_1 in fp64, pairwise inside
// 32-dimension blocks, blocks in order; fy = fl32((||rho||^2 / ||rho||_1) /
// sqrt(d)) = F_y / d (0 when rho = 0).  Outputs: e4m3 +-1 codes (yq, row
// stride dq) and/or sign words (yw), and info = (bd 0, sd fy, sumy 0, ny2), so
// the tensor epilogue's u = fma(sd, acc, bd pc) is fy (d - 2h).
__global__ void __launch_bounds__(CPREP_WARPS * 32) rbq1_cprep_sym_kernel(
    const float *__restrict__ C, int k, int d, const float *__restrict__ m, uint8_t *__restrict__ yq, int dq,
    uint32_t *__restrict__ yw, Rbq1CInfo *__restrict__ info) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int j = blockIdx.x * CPREP_WARPS + warp;
    if (j >= k) return;  // warp-uniform
    const float *c = C + (int64_t)j * d;
    const int W = (d + 31) >> 5;
    double q2 = 0.0, l1 = 0.0;
    for (int w = 0; w < W; ++w) {
        const int i = 32 * w + lane;
        const float r = (i < d) ? __fsub_rn(c[i], m[i]) : 0.0f;
        double sq = (i < d) ? __dmul_rn((double)r, (double)r) : 0.0;
        double ab = (i < d) ? fabs((double)r) : 0.0;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            sq = __dadd_rn(sq, __shfl_xor_sync(0xffffffffu, sq, o));
            ab = __dadd_rn(ab, __shfl_xor_sync(0xffffffffu, ab, o));
        }
        q2 = __dadd_rn(q2, sq);
        l1 = __dadd_rn(l1, ab);
        const bool bit = (i < d) && r > 0.0f;
        if (yq && i < d) yq[(int64_t)j * dq + i] = bit ? 0x38 : 0xB8;
        const uint32_t word = __ballot_sync(0xffffffffu, bit);
        if (yw && lane == 0) yw[(int64_t)j * W + w] = word;
    }
    if (lane == 0) {
        Rbq1CInfo in;
        in.bd = 0.0f;
        in.sd = (l1 > 0.0) ? __double2float_rn(__ddiv_rn(__ddiv_rn(q2, l1), __dsqrt_rn((double)d))) : 0.0f;
        in.sumy = 0;
        in.ny2 = __double2float_rn(q2);
        info[j] = in;
    }
}

cudaError_t launch_rbq1_cprep_sym(const float *C, int k, int d, const float *m, uint8_t *yq, int dq, uint32_t *yw,
                                  Rbq1CInfo *info, cudaStream_t st) {
    rbq1_cprep_sym_kernel<<<(k + CPREP_WARPS - 1) / CPREP_WARPS, CPREP_WARPS * 32, 0, st>>>(C, k, d, m, yq, dq, yw,
                                                                                        info);
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
