// SQ8 assignment in the code domain (Section 3.1 "SQ8 and SQ4"):
// dist = sum_i (xbar_i - cbar_i)^2 = nx + nc - 2 sum_i xbar_i cbar_i, exact in
// int32 (d <= 4096), argmin with ties to the lowest index.
//
// CUDA-core kernel: 64 points x 64 centroids per tile, 64 dimensions (16 code
// words) per shared-memory slice, each thread a 4 x 4 block of pairs using
// __dp4a (four u8 x u8 products per instruction, exact).
#include "skm_internal.cuh"

namespace skm {

__device__ __forceinline__ uint32_t load_code_word(const uint8_t *__restrict__ row, int d, int w,
                                                   bool aligned4) {
    const int i = 4 * w;
    if (aligned4 && i + 3 < d) return __ldg(reinterpret_cast<const uint32_t *>(row + i));
    uint32_t v = 0;
#pragma unroll
    for (int q = 0; q < 4; ++q)
        if (i + q < d) v |= ((uint32_t)__ldg(row + i + q)) << (8 * q);
    return v;
}

__global__ void __launch_bounds__(256) assign_sq8_simt_kernel(
    const uint8_t *__restrict__ X, int64_t n, int d, const uint8_t *__restrict__ C, int k,
    const int32_t *__restrict__ nx, const int32_t *__restrict__ nc, int32_t *__restrict__ assign,
    float *__restrict__ dist) {
    __shared__ __align__(16) uint32_t xs[16][68];
    __shared__ __align__(16) uint32_t cs[16][68];
    const int tid = threadIdx.x;
    const int ty = tid >> 4, tx = tid & 15;
    const int64_t row0 = (int64_t)blockIdx.x * 64;
    const bool aligned4 = (d % 4) == 0;
    const int W4 = (d + 3) / 4;
    const int lw = tid & 15, lr0 = tid >> 4;  // loader: word lw of rows lr0 + 16q

    int32_t best[4];
    int besti[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        best[i] = 0x7fffffff;
        besti[i] = 0x7fffffff;
    }
    int32_t nxr[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int64_t r = row0 + ty * 4 + i;
        nxr[i] = (r < n) ? nx[r] : 0;
    }

    for (int c0 = 0; c0 < k; c0 += 64) {
        int32_t acc[4][4];
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int j = 0; j < 4; ++j) acc[i][j] = 0;
        for (int w0 = 0; w0 < W4; w0 += 16) {
            __syncthreads();
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int r = lr0 + 16 * q;
                const int w = w0 + lw;
                uint32_t xv = 0, cv = 0;
                if (w < W4) {
                    if (row0 + r < n) xv = load_code_word(X + (row0 + r) * d, d, w, aligned4);
                    if (c0 + r < k) cv = load_code_word(C + (int64_t)(c0 + r) * d, d, w, aligned4);
                }
                xs[lw][r] = xv;
                cs[lw][r] = cv;
            }
            __syncthreads();
            const int wmax = min(16, W4 - w0);
            for (int ww = 0; ww < wmax; ++ww) {
                const uint4 xv = *reinterpret_cast<const uint4 *>(&xs[ww][ty * 4]);
                const uint4 cv = *reinterpret_cast<const uint4 *>(&cs[ww][tx * 4]);
                const uint32_t xa[4] = {xv.x, xv.y, xv.z, xv.w};
                const uint32_t ca[4] = {cv.x, cv.y, cv.z, cv.w};
#pragma unroll
                for (int i = 0; i < 4; ++i)
#pragma unroll
                    for (int j = 0; j < 4; ++j)
                        acc[i][j] = (int32_t)__dp4a(xa[i], ca[j], (uint32_t)acc[i][j]);
            }
        }
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            int32_t bd = 0x7fffffff;
            int bi = 0x7fffffff;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int cj = c0 + tx * 4 + j;
                if (cj < k) {
                    const int32_t dd = nxr[i] + nc[cj] - 2 * acc[i][j];
                    if (dd < bd) {
                        bd = dd;
                        bi = cj;
                    }
                }
            }
#pragma unroll
            for (int o = 8; o > 0; o >>= 1) {
                const int32_t od = __shfl_xor_sync(0xffffffffu, bd, o);
                const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
                if (od < bd || (od == bd && oi < bi)) {
                    bd = od;
                    bi = oi;
                }
            }
            if (bd < best[i] || (bd == best[i] && bi < besti[i])) {
                best[i] = bd;
                besti[i] = bi;
            }
        }
    }
    if (tx == 0) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int64_t r = row0 + ty * 4 + i;
            if (r < n) {
                assign[r] = besti[i];
                if (dist) dist[r] = (float)best[i];
            }
        }
    }
}

cudaError_t launch_assign_sq8_simt(const uint8_t *X, int64_t n, int d, const uint8_t *C, int k,
                                   const int32_t *nx, const int32_t *nc, int32_t *assign,
                                   float *dist, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    assign_sq8_simt_kernel<<<(unsigned)((n + 63) / 64), 256, 0, st>>>(X, n, d, C, k, nx, nc,
                                                                      assign, dist);
    return launched();
}

}  // namespace skm
