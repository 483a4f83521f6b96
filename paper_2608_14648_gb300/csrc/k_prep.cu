// Per-iteration centroid preparation.
//  RBQ1 (Section 3.1 "RabitQ"): the centroid residual rho = c - m is
//  re-encoded with per-centroid SQ4 (b = min rho, s = (max rho - b)/15,
//  s = 1 when flat, ybar = clip(rint((rho - b)/s), 0, 15)) and stored as four
//  bit planes per 32-dimension word, so that sum_i xbar_i ybar_i =
//  sum_j 2^j popc(xbar & plane_j).  One lane per centroid walks its row in
//  order, which fixes the fp64 summation order of ||rho||^2.
//  SQ8: per-row sums of squared codes (exact int32).
#include "skm_internal.cuh"

namespace skm {

// Each warp owns 32 centroids (one per lane).  The warp stages 32 x 32 tiles
// of rho = c - m through shared memory with coalesced loads; each lane then
// walks its own centroid's dimensions in increasing order.
constexpr int CPREP_WARPS = 4;

// e4m3 encodings of the integers 0..15 (sign 0, exponent bias 7, 3 mantissa
// bits): 0 -> 0x00, 1 -> 0x38, 2 -> 0x40, 3 -> 0x44, 4 -> 0x48, ... 15 -> 0x57.
__device__ __forceinline__ uint8_t e4m3_of_code(uint32_t y) {
    if (y == 0) return 0;
    const int e = 31 - __clz(y);                       // floor(log2 y), 0..3
    const uint32_t mant = (y << (3 - e)) & 7u;         // 3 bits below the leading one
    return (uint8_t)(((uint32_t)(e + 7) << 3) | mant);
}

// planes != nullptr: SQ4 codes as four bit planes per word (AND + popcount
// kernel); yq != nullptr: the same codes as e4m3 bytes, row stride dq (tensor
// kernel).
__global__ void __launch_bounds__(CPREP_WARPS * 32) rbq1_cprep_kernel(
    const float *__restrict__ C, int k, int d, const float *__restrict__ m,
    uint4 *__restrict__ planes, Rbq1CInfo *__restrict__ info, uint8_t *__restrict__ yq, int dq) {
    __shared__ float tile[CPREP_WARPS][32][33];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int j0 = (blockIdx.x * CPREP_WARPS + warp) * 32;
    if (j0 >= k) return;  // warp-uniform
    const int j = j0 + lane;
    const bool valid = j < k;
    float(*t)[33] = tile[warp];
    auto stage = [&](int i0) {
        const int i = i0 + lane;
        const float mi = (i < d) ? m[i] : 0.0f;
#pragma unroll 4
        for (int r = 0; r < 32; ++r) {
            const int row = j0 + r;
            t[r][lane] = (row < k && i < d) ? __fsub_rn(C[(int64_t)row * d + i], mi) : 0.0f;
        }
        __syncwarp();
    };
    float lo = INFINITY, hi = -INFINITY;
    double q2 = 0.0;
    for (int i0 = 0; i0 < d; i0 += 32) {
        stage(i0);
        const int n = min(32, d - i0);
        for (int l = 0; l < n; ++l) {
            const float r = t[lane][l];
            lo = fminf(lo, r);
            hi = fmaxf(hi, r);
            q2 = __dadd_rn(q2, __dmul_rn((double)r, (double)r));
        }
        __syncwarp();
    }
    float sc = __fdiv_rn(__fsub_rn(hi, lo), 15.0f);
    if (!(sc > 0.0f)) sc = 1.0f;
    const int W = (d + 31) >> 5;
    int32_t sy = 0;
    for (int w = 0; w < W; ++w) {
        stage(32 * w);
        uint32_t p0 = 0, p1 = 0, p2 = 0, p3 = 0;
        const int n = min(32, d - 32 * w);
        for (int l = 0; l < n; ++l) {
            float q = rintf(__fdiv_rn(__fsub_rn(t[lane][l], lo), sc));
            q = (q >= 0.0f) ? q : 0.0f;
            q = fminf(q, 15.0f);
            const uint32_t y = (uint32_t)q;
            sy += (int32_t)y;
            if (yq && valid) yq[(int64_t)j * dq + 32 * w + l] = e4m3_of_code(y);
            p0 |= (y & 1u) << l;
            p1 |= ((y >> 1) & 1u) << l;
            p2 |= ((y >> 2) & 1u) << l;
            p3 |= ((y >> 3) & 1u) << l;
        }
        if (valid && planes) planes[(int64_t)j * W + w] = make_uint4(p0, p1, p2, p3);
        __syncwarp();
    }
    if (valid) {
        Rbq1CInfo in;
        in.b = lo;
        in.s = sc;
        in.sumy = sy;
        in.ny2 = __double2float_rn(q2);
        info[j] = in;
    }
}

cudaError_t launch_rbq1_cprep(const float *C, int k, int d, const float *m, uint4 *planes,
                              Rbq1CInfo *info, cudaStream_t st) {
    const int per_block = CPREP_WARPS * 32;
    rbq1_cprep_kernel<<<(k + per_block - 1) / per_block, per_block, 0, st>>>(C, k, d, m, planes,
                                                                            info, nullptr, 0);
    return launched();
}

cudaError_t launch_rbq1_cprep_tc(const float *C, int k, int d, const float *m, uint8_t *yq, int dq,
                                 Rbq1CInfo *info, cudaStream_t st) {
    const int per_block = CPREP_WARPS * 32;
    rbq1_cprep_kernel<<<(k + per_block - 1) / per_block, per_block, 0, st>>>(C, k, d, m, nullptr,
                                                                            info, yq, dq);
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
