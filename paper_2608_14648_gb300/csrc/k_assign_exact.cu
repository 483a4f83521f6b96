// Exact fp32 nearest-centroid scan (Section 2.3 STEP 2) on CUDA cores:
// dist = sum_i (x_i - c_i)^2 accumulated in fp32 per pair, argmin with ties
// to the lowest index, the N x K matrix never leaves registers.
//
// Tile: 64 points x 64 centroids per step, 32 dimensions staged in shared
// memory per k-slice; each of 256 threads owns a 4 x 4 block of pairs.  The 16
// threads that share a point sit in one half-warp, so the per-tile argmin is a
// 4-step shuffle reduction.  This kernel is the full-scan fallback of the
// tensor-core screen (rows listed in `rows`) and the BF16 pruning path's
// dense reference scan.
#include "skm_internal.cuh"

namespace skm {

template <typename TX>
__device__ __forceinline__ float load_x(const TX *p);
template <>
__device__ __forceinline__ float load_x<float>(const float *p) {
    return __ldg(p);
}
template <>
__device__ __forceinline__ float load_x<uint16_t>(const uint16_t *p) {
    return __uint_as_float(((uint32_t)__ldg(p)) << 16);
}

__device__ __forceinline__ void argmin_merge(float &bd, int &bi, float d, int i) {
    if (d < bd || (d == bd && i < bi)) {
        bd = d;
        bi = i;
    }
}

// rows == nullptr: rows 0..nrows-1.  Otherwise the rows are rows[0..count)
// with count = *nrows_dev (a device-side list, e.g. the rows a screen could
// not decide).  Blocks stride over work items of 64 rows.  With `keys` (one
// per listed row, preset to ~0) the centroids are also split across the grid
// when the list is short (a handful of rows against thousands of centroids
// would otherwise run on a few SMs): each work item covers a range of
// centroid tiles and merges (dist bits << 32 | index) into its rows' keys with
// atomicMin — non-negative distances order like their bit patterns, so the
// smallest key is the nearest centroid with ties to the lowest index.
template <typename TX>
__global__ void __launch_bounds__(256) assign_exact_kernel(const TX *__restrict__ X,
                                                           const int32_t *__restrict__ rows,
                                                           const int32_t *__restrict__ nrows_dev,
                                                           int64_t nrows_arg, int d,
                                                           const float *__restrict__ C, int k,
                                                           int32_t *__restrict__ assign,
                                                           float *__restrict__ dist,
                                                           unsigned long long *__restrict__ keys) {
    __shared__ __align__(16) float xs[32][68];
    __shared__ __align__(16) float cs[32][68];
    const int tid = threadIdx.x;
    const int ty = tid >> 4, tx = tid & 15;
    const int64_t nrows = nrows_dev ? (int64_t)*nrows_dev : nrows_arg;
    const int64_t rtiles = (nrows + 63) / 64;
    const int ktiles = (k + 63) / 64;
    int nsplit = 1;
    if (keys && rtiles > 0) nsplit = (int)max((int64_t)1, min((int64_t)ktiles, (int64_t)gridDim.x / rtiles));
    const int tps = (ktiles + nsplit - 1) / nsplit;  // centroid tiles per split
    const int64_t nwork = rtiles * nsplit;
    for (int64_t w = blockIdx.x; w < nwork; w += gridDim.x) {
        const int64_t row0 = (w / nsplit) * 64;
        const int cbeg = (int)(w % nsplit) * tps * 64;
        const int cend = min(k, cbeg + tps * 64);
        __syncthreads();

        // the point rows this block owns (indirect when `rows` is given)
        int64_t prow[4];
        bool pval[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int64_t r = row0 + ty * 4 + i;
            pval[i] = r < nrows;
            prow[i] = pval[i] ? (rows ? (int64_t)rows[r] : r) : 0;
        }
        // loader mapping: thread loads rows lr0 + 8q (q = 0..7) at dim ld
        const int ld = tid & 31, lr0 = tid >> 5;
        int64_t lrow[8];
        bool lval[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            const int64_t r = row0 + lr0 + 8 * q;
            lval[q] = r < nrows;
            lrow[q] = lval[q] ? (rows ? (int64_t)rows[r] : r) : 0;
        }

        float best[4];
        int besti[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            best[i] = INFINITY;
            besti[i] = 0x7fffffff;
        }

        for (int c0 = cbeg; c0 < cend; c0 += 64) {
            float acc[4][4];
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = 0.0f;

            for (int k0 = 0; k0 < d; k0 += 32) {
                const int dim = k0 + ld;
                __syncthreads();
#pragma unroll
                for (int q = 0; q < 8; ++q) {
                    const int r = lr0 + 8 * q;
                    float xv = 0.0f, cv = 0.0f;
                    if (dim < d) {
                        if (lval[q]) xv = load_x<TX>(X + lrow[q] * d + dim);
                        if (c0 + r < cend) cv = __ldg(C + (int64_t)(c0 + r) * d + dim);
                    }
                    xs[ld][r] = xv;
                    cs[ld][r] = cv;
                }
                __syncthreads();
                const int kmax = min(32, d - k0);
                for (int kk = 0; kk < kmax; ++kk) {
                    const float4 xv = *reinterpret_cast<const float4 *>(&xs[kk][ty * 4]);
                    const float4 cv = *reinterpret_cast<const float4 *>(&cs[kk][tx * 4]);
                    const float xa[4] = {xv.x, xv.y, xv.z, xv.w};
                    const float ca[4] = {cv.x, cv.y, cv.z, cv.w};
#pragma unroll
                    for (int i = 0; i < 4; ++i)
#pragma unroll
                        for (int j = 0; j < 4; ++j) {
                            const float t = __fsub_rn(xa[i], ca[j]);
                            acc[i][j] = __fmaf_rn(t, t, acc[i][j]);
                        }
                }
            }
            // per-row argmin over this centroid tile, then merge into the running best
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                float bd = INFINITY;
                int bi = 0x7fffffff;
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const int cj = c0 + tx * 4 + j;
                    if (cj < cend) argmin_merge(bd, bi, acc[i][j], cj);
                }
#pragma unroll
                for (int o = 8; o > 0; o >>= 1) {
                    const float od = __shfl_xor_sync(0xffffffffu, bd, o);
                    const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
                    argmin_merge(bd, bi, od, oi);
                }
                argmin_merge(best[i], besti[i], bd, bi);
            }
        }
        if (tx == 0) {
#pragma unroll
            for (int i = 0; i < 4; ++i)
                if (pval[i]) {
                    if (keys) {
                        if (besti[i] != 0x7fffffff)
                            atomicMin(keys + row0 + ty * 4 + i,
                                      ((unsigned long long)__float_as_uint(best[i]) << 32) | (uint32_t)besti[i]);
                    } else {
                        assign[prow[i]] = besti[i];
                        if (dist) dist[prow[i]] = best[i];
                    }
                }
        }
    }  // work items
}

__global__ void keys_init_kernel(const int32_t *__restrict__ count, unsigned long long *__restrict__ keys) {
    const int64_t c = *count;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < c; i += (int64_t)gridDim.x * blockDim.x)
        keys[i] = ~0ull;
}

__global__ void keys_finish_kernel(const int32_t *__restrict__ rows, const int32_t *__restrict__ count,
                                   const unsigned long long *__restrict__ keys, int32_t *__restrict__ assign,
                                   float *__restrict__ dist) {
    const int64_t c = *count;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < c; i += (int64_t)gridDim.x * blockDim.x) {
        const unsigned long long key = keys[i];
        if (key == ~0ull) continue;  // no centroid (k == 0 cannot happen on this path)
        assign[rows[i]] = (int32_t)(key & 0xffffffffull);
        if (dist) dist[rows[i]] = __uint_as_float((uint32_t)(key >> 32));
    }
}

static unsigned blocks_for_rows(int64_t nrows) {
    int64_t b = (nrows + 63) / 64;
    const int64_t cap = 152LL * 8;  // 8 resident 256-thread blocks per SM
    return (unsigned)(b < 1 ? 1 : (b > cap ? cap : b));
}

cudaError_t launch_assign_exact_f32(const float *X, int64_t n, int d, const float *C, int k,
                                    int32_t *assign, float *dist, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    assign_exact_kernel<float><<<blocks_for_rows(n), 256, 0, st>>>(X, nullptr, nullptr, n, d, C,
                                                                   k, assign, dist, nullptr);
    return launched();
}

cudaError_t launch_assign_exact_bf16(const uint16_t *X, int64_t n, int d, const float *C, int k,
                                     int32_t *assign, float *dist, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    assign_exact_kernel<uint16_t><<<blocks_for_rows(n), 256, 0, st>>>(X, nullptr, nullptr, n, d,
                                                                      C, k, assign, dist, nullptr);
    return launched();
}

cudaError_t launch_assign_exact_rows(const void *X, int x_is_bf16, const int32_t *rows,
                                     const int32_t *count_dev, int64_t max_rows, int d,
                                     const float *C, int k, int32_t *assign, float *dist,
                                     unsigned long long *keys, cudaStream_t st) {
    if (max_rows == 0) return cudaSuccess;
    // enough blocks to split the centroids when only a few rows are listed
    const unsigned g = keys ? 152u * 4u : blocks_for_rows(max_rows);
    if (keys) {
        keys_init_kernel<<<152, 256, 0, st>>>(count_dev, keys);
        cudaError_t e = launched();
        if (e != cudaSuccess) return e;
    }
    if (x_is_bf16)
        assign_exact_kernel<uint16_t><<<g, 256, 0, st>>>(static_cast<const uint16_t *>(X), rows,
                                                         count_dev, 0, d, C, k, assign, dist, keys);
    else
        assign_exact_kernel<float><<<g, 256, 0, st>>>(static_cast<const float *>(X), rows,
                                                      count_dev, 0, d, C, k, assign, dist, keys);
    cudaError_t e = launched();
    if (e != cudaSuccess || !keys) return e;
    keys_finish_kernel<<<152, 256, 0, st>>>(rows, count_dev, keys, assign, dist);
    return launched();
}

}  // namespace skm
