// Initialisation gathers, the WCSS objective, the projection Y = (X - mu) P
// (rotation / JLT / PCA, Section 3.1) and the PCA covariance.
#include "skm_internal.cuh"

namespace skm {

// ------------------------------------------------------------ init gathers
__global__ void gather_rows_kernel(const unsigned char *__restrict__ X, int64_t n,
                                   int64_t row_bytes, const int64_t *__restrict__ idx, int k,
                                   unsigned char *__restrict__ out, int *__restrict__ status) {
    const int j = blockIdx.x;
    if (j >= k) return;
    const int64_t p = idx[j];
    if (p < 0 || p >= n) {  // invalid index: row left untouched, status flagged
        if (threadIdx.x == 0) atomicExch(status, 1);
        return;
    }
    const unsigned char *src = X + p * row_bytes;
    unsigned char *dst = out + (int64_t)j * row_bytes;
    for (int64_t b = threadIdx.x; b < row_bytes; b += blockDim.x) dst[b] = src[b];
}

cudaError_t launch_gather_rows(const void *X, int64_t n, int elem_bytes, int64_t row_elems,
                               const int64_t *idx, int k, void *out, int *status,
                               cudaStream_t st) {
    gather_rows_kernel<<<k, 256, 0, st>>>(static_cast<const unsigned char *>(X), n,
                                          row_elems * elem_bytes, idx, k,
                                          static_cast<unsigned char *>(out), status);
    return launched();
}

// Decode of single points: the decode-average of a one-member cluster, in
// exactly the operation order of the RBQ1 update (count = 1).
__global__ void rbq1_decode_rows_kernel(const uint32_t *__restrict__ codes,
                                        const float *__restrict__ F, int64_t n, int d,
                                        const float *__restrict__ m, int e,
                                        const int64_t *__restrict__ idx, int k,
                                        float *__restrict__ out, int *__restrict__ status) {
    const int j = blockIdx.x;
    if (j >= k) return;
    const int W = (d + 31) >> 5;
    const int64_t p = idx[j];
    if (p < 0 || p >= n) {
        if (threadIdx.x == 0) atomicExch(status, 1);
        return;
    }
    const int64_t fq = __double2ll_rn(__dmul_rn((double)F[p], ldexp(1.0, e)));
    // the update's factor for a cluster of one member: fl(1/sqrt(d)) 2^-e
    const double f = __dmul_rn(__ddiv_rn(1.0, __dsqrt_rn((double)d)), ldexp(1.0, -e));
    for (int i = threadIdx.x; i < d; i += blockDim.x) {
        const int64_t T = ((codes[p * W + (i >> 5)] >> (i & 31)) & 1u) ? fq : 0;
        const double v = __dmul_rn(__ll2double_rn(2 * T - fq), f);
        out[(int64_t)j * d + i] = __double2float_rn(__dadd_rn((double)m[i], v));
    }
}

cudaError_t launch_rbq1_decode_rows(const uint32_t *codes, const float *F, int64_t n, int d,
                                    const float *m, int e, const int64_t *idx, int k,
                                    float *out, int *status, cudaStream_t st) {
    rbq1_decode_rows_kernel<<<k, 256, 0, st>>>(codes, F, n, d, m, e, idx, k, out, status);
    return launched();
}

// ---------------------------------------------------------------- objective
// One warp per point: fp32 sum of squared differences to its centroid, then
// fp64 per-block partials (fixed order), reduced by launch_sum_double.
__global__ void objective_kernel(const void *__restrict__ Xv, int x_is_bf16, int64_t n, int d,
                                 const float *__restrict__ C, const int32_t *__restrict__ assign,
                                 double *__restrict__ partials) {
    __shared__ double wsum[32];
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
    double acc = 0.0;
    for (int64_t p = warp; p < n; p += nwarps) {
        const float *c = C + (int64_t)assign[p] * d;
        float s = 0.0f;
        for (int i = lane; i < d; i += 32) {
            float x;
            if (x_is_bf16)
                x = __uint_as_float(((uint32_t) reinterpret_cast<const uint16_t *>(Xv)[p * d + i])
                                    << 16);
            else
                x = reinterpret_cast<const float *>(Xv)[p * d + i];
            const float t = __fsub_rn(x, c[i]);
            s = __fmaf_rn(t, t, s);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
        acc += (double)s;
    }
    if (lane == 0) wsum[wid] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
        double t = 0.0;
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w) t += wsum[w];
        partials[blockIdx.x] = t;
    }
}

cudaError_t launch_objective(const void *X, int x_is_bf16, int64_t n, int d, const float *C,
                             const int32_t *assign, double *partials, int nblk,
                             cudaStream_t st) {
    objective_kernel<<<nblk, 256, 0, st>>>(X, x_is_bf16, n, d, C, assign, partials);
    return launched();
}

__global__ void sum_double_kernel(const double *__restrict__ in, int64_t count,
                                  double *__restrict__ out) {
    __shared__ double sh[256];
    double s = 0.0;
    for (int64_t i = threadIdx.x; i < count; i += blockDim.x) s += in[i];
    sh[threadIdx.x] = s;
    __syncthreads();
    if (threadIdx.x == 0) {
        double t = 0.0;
        for (int i = 0; i < (int)blockDim.x; ++i) t += sh[i];
        *out = t;
    }
}

cudaError_t launch_sum_double(const double *in, int64_t count, double *out, cudaStream_t st) {
    sum_double_kernel<<<1, 256, 0, st>>>(in, count, out);
    return launched();
}

__global__ void sum_float_partial_kernel(const float *__restrict__ in, int64_t count,
                                         double *__restrict__ partials) {
    __shared__ double sh[256];
    double s = 0.0;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < count;
         i += (int64_t)gridDim.x * blockDim.x)
        s += (double)in[i];
    sh[threadIdx.x] = s;
    __syncthreads();
    if (threadIdx.x == 0) {
        double t = 0.0;
        for (int i = 0; i < (int)blockDim.x; ++i) t += sh[i];
        partials[blockIdx.x] = t;
    }
}

cudaError_t launch_sum_float_to_double(const float *in, int64_t count, double *partials,
                                       int nblk, cudaStream_t st) {
    sum_float_partial_kernel<<<nblk, 256, 0, st>>>(in, count, partials);
    return launched();
}

// --------------------------------------------------------------- projection
// Y = (X - mu) P, fp32 FMA accumulation; 64 x 64 output tile per block,
// 32-deep k-slices in shared memory, 4 x 4 outputs per thread.
__global__ void __launch_bounds__(256) project_kernel(const float *__restrict__ X, int64_t n,
                                                      int d, const float *__restrict__ mu,
                                                      const float *__restrict__ P, int dout,
                                                      int out_bf16, void *__restrict__ Yv) {
    __shared__ __align__(16) float xs[32][68];
    __shared__ __align__(16) float ps[32][68];
    const int tid = threadIdx.x, ty = tid >> 4, tx = tid & 15;
    const int64_t row0 = (int64_t)blockIdx.x * 64;
    const int col0 = blockIdx.y * 64;
    float acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = 0.0f;
    const int ld = tid & 31, lr0 = tid >> 5;
    for (int k0 = 0; k0 < d; k0 += 32) {
        __syncthreads();
        // X tile: rows row0.., dims k0..; P tile: dims k0.., cols col0..
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            const int r = lr0 + 8 * q;
            const int dim = k0 + ld;
            float xv = 0.0f;
            if (dim < d && row0 + r < n) {
                xv = X[(row0 + r) * d + dim];
                if (mu) xv = __fsub_rn(xv, mu[dim]);
            }
            xs[ld][r] = xv;
        }
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            const int kr = tid / 64 + 4 * q;  // 0..31
            const int c = tid & 63;
            float pv = 0.0f;
            if (k0 + kr < d && col0 + c < dout) pv = P[(int64_t)(k0 + kr) * dout + col0 + c];
            ps[kr][c] = pv;
        }
        __syncthreads();
        const int kmax = min(32, d - k0);
        for (int kk = 0; kk < kmax; ++kk) {
            const float4 xv = *reinterpret_cast<const float4 *>(&xs[kk][ty * 4]);
            const float4 pv = *reinterpret_cast<const float4 *>(&ps[kk][tx * 4]);
            const float xa[4] = {xv.x, xv.y, xv.z, xv.w};
            const float pa[4] = {pv.x, pv.y, pv.z, pv.w};
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = __fmaf_rn(xa[i], pa[j], acc[i][j]);
        }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int64_t r = row0 + ty * 4 + i;
        if (r >= n) continue;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int c = col0 + tx * 4 + j;
            if (c >= dout) continue;
            if (out_bf16)
                reinterpret_cast<__nv_bfloat16 *>(Yv)[r * dout + c] = __float2bfloat16_rn(acc[i][j]);
            else
                reinterpret_cast<float *>(Yv)[r * dout + c] = acc[i][j];
        }
    }
}

cudaError_t launch_project(const float *X, int64_t n, int d, const float *mean, const float *P,
                           int d_out, int out_bf16, void *Y, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    dim3 grid((unsigned)((n + 63) / 64), (unsigned)((d_out + 63) / 64));
    project_kernel<<<grid, 256, 0, st>>>(X, n, d, mean, P, d_out, out_bf16, Y);
    return launched();
}

// --------------------------------------------------------------- covariance
// partial[s][i][j] = sum over row-split s of (x_i - mu_i)(x_j - mu_j): fp32
// products accumulated in fp32 over 256-row blocks, then folded into fp64.
__global__ void __launch_bounds__(256) cov_partial_kernel(const float *__restrict__ X, int64_t n,
                                                          int d, const float *__restrict__ mu,
                                                          double *__restrict__ partial) {
    __shared__ __align__(16) float as[32][68];
    __shared__ __align__(16) float bs[32][68];
    const int tid = threadIdx.x, ty = tid >> 4, tx = tid & 15;
    const int i0 = blockIdx.x * 64, j0 = blockIdx.y * 64;
    const int s = blockIdx.z, S = gridDim.z;
    const int64_t rows_per = (n + S - 1) / S;
    const int64_t r_lo = (int64_t)s * rows_per, r_hi = min(n, r_lo + rows_per);
    double accd[4][4];
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int b = 0; b < 4; ++b) accd[a][b] = 0.0;
    const int lc = tid & 63, lr0 = tid >> 6;  // loader: column lc, rows lr0 + 4q
    for (int64_t rb = r_lo; rb < r_hi; rb += 256) {
        float acc[4][4];
#pragma unroll
        for (int a = 0; a < 4; ++a)
#pragma unroll
            for (int b = 0; b < 4; ++b) acc[a][b] = 0.0f;
        const int64_t rend = min(r_hi, rb + 256);
        for (int64_t r0 = rb; r0 < rend; r0 += 32) {
            __syncthreads();
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                const int rr = lr0 + 4 * q;  // 0..31
                const int64_t r = r0 + rr;
                float av = 0.0f, bv = 0.0f;
                if (r < rend) {
                    if (i0 + lc < d) av = __fsub_rn(X[r * d + i0 + lc], mu[i0 + lc]);
                    if (j0 + lc < d) bv = __fsub_rn(X[r * d + j0 + lc], mu[j0 + lc]);
                }
                as[rr][lc] = av;
                bs[rr][lc] = bv;
            }
            __syncthreads();
#pragma unroll 4
            for (int kk = 0; kk < 32; ++kk) {
                const float4 av = *reinterpret_cast<const float4 *>(&as[kk][ty * 4]);
                const float4 bv = *reinterpret_cast<const float4 *>(&bs[kk][tx * 4]);
                const float aa[4] = {av.x, av.y, av.z, av.w};
                const float ba[4] = {bv.x, bv.y, bv.z, bv.w};
#pragma unroll
                for (int a = 0; a < 4; ++a)
#pragma unroll
                    for (int b = 0; b < 4; ++b) acc[a][b] = __fmaf_rn(aa[a], ba[b], acc[a][b]);
            }
        }
#pragma unroll
        for (int a = 0; a < 4; ++a)
#pragma unroll
            for (int b = 0; b < 4; ++b) accd[a][b] += (double)acc[a][b];
    }
#pragma unroll
    for (int a = 0; a < 4; ++a) {
        const int i = i0 + ty * 4 + a;
        if (i >= d) continue;
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            const int j = j0 + tx * 4 + b;
            if (j < d) partial[((int64_t)s * d + i) * d + j] = accd[a][b];
        }
    }
}

cudaError_t launch_cov_partial(const float *X, int64_t n, int d, const float *mean,
                               double *partial, int splits, cudaStream_t st) {
    dim3 grid((unsigned)((d + 63) / 64), (unsigned)((d + 63) / 64), (unsigned)splits);
    cov_partial_kernel<<<grid, 256, 0, st>>>(X, n, d, mean, partial);
    return launched();
}

__global__ void cov_reduce_kernel(const double *__restrict__ partial, int splits, int d,
                                  double *__restrict__ cov) {
    const int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
    const int64_t dd = (int64_t)d * d;
    if (t >= dd) return;
    double s = 0.0;
    for (int q = 0; q < splits; ++q) s += partial[(int64_t)q * dd + t];
    cov[t] = s;
}

cudaError_t launch_cov_reduce(const double *partial, int splits, int d, double *cov,
                              cudaStream_t st) {
    const int64_t dd = (int64_t)d * d;
    cov_reduce_kernel<<<(unsigned)((dd + 255) / 256), 256, 0, st>>>(partial, splits, d, cov);
    return launched();
}

}  // namespace skm

namespace skm {

// -------------------------------------------------- randomized Hadamard rotation
// y = (1/sqrt(D)) H_D diag(sigma) [x - mean; 0] (a structured random
// orthogonal transform, Section 3.1's rotation before RabitQ / SuperKMeans,
// O(D log D) per row instead of a D x D product).  Element i of the padded
// row lives in lane i % 32, register i / 32 of one warp; the Walsh-Hadamard
// butterflies over the register bits run inside each lane and those over the
// lane bits through __shfl_xor_sync.  The transform is a product of
// independent per-bit butterflies, so their order does not change the
// result beyond rounding.  D <= 1024 here; 2048 and 4096 use shared memory.
template <int J>
__global__ void __launch_bounds__(256) hadamard_warp_kernel(const float *__restrict__ X, int64_t n, int d,
                                                            const float *__restrict__ mean,
                                                            const float *__restrict__ sigma, float scale,
                                                            int out_bf16, void *__restrict__ Y) {
    constexpr int D = 32 * J;
    const int lane = threadIdx.x & 31;
    const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    float sg[J], mu[J];
#pragma unroll
    for (int j = 0; j < J; ++j) {
        const int i = lane + 32 * j;
        sg[j] = __ldg(sigma + i);
        mu[j] = (mean && i < d) ? __ldg(mean + i) : 0.0f;
    }
    for (int64_t r = warp; r < n; r += nw) {
        float v[J];
#pragma unroll
        for (int j = 0; j < J; ++j) {
            const int i = lane + 32 * j;
            const float x = i < d ? __ldg(X + r * d + i) : 0.0f;
            v[j] = __fmul_rn(__fsub_rn(x, mu[j]), sg[j]);
        }
#pragma unroll
        for (int h = 1; h < J; h <<= 1)
#pragma unroll
            for (int j = 0; j < J; ++j)
                if ((j & h) == 0) {
                    const float a = v[j], b = v[j + h];
                    v[j] = __fadd_rn(a, b);
                    v[j + h] = __fsub_rn(a, b);
                }
#pragma unroll
        for (int o = 1; o < 32; o <<= 1)
#pragma unroll
            for (int j = 0; j < J; ++j) {
                const float p = __shfl_xor_sync(0xffffffffu, v[j], o);
                v[j] = (lane & o) ? __fsub_rn(p, v[j]) : __fadd_rn(v[j], p);
            }
#pragma unroll
        for (int j = 0; j < J; ++j) {
            const int i = lane + 32 * j;
            const float y = __fmul_rn(v[j], scale);
            if (out_bf16)
                reinterpret_cast<__nv_bfloat16 *>(Y)[r * D + i] = __float2bfloat16_rn(y);
            else
                reinterpret_cast<float *>(Y)[r * D + i] = y;
        }
    }
}

// D = 2048 or 4096: one block per row, the row in shared memory.
__global__ void __launch_bounds__(512) hadamard_block_kernel(const float *__restrict__ X, int64_t n, int d, int D,
                                                             const float *__restrict__ mean,
                                                             const float *__restrict__ sigma, float scale,
                                                             int out_bf16, void *__restrict__ Y) {
    __shared__ float v[4096];
    for (int64_t r = blockIdx.x; r < n; r += gridDim.x) {
        __syncthreads();
        for (int i = threadIdx.x; i < D; i += blockDim.x) {
            const float x = i < d ? __ldg(X + r * d + i) : 0.0f;
            const float m = (mean && i < d) ? __ldg(mean + i) : 0.0f;
            v[i] = __fmul_rn(__fsub_rn(x, m), __ldg(sigma + i));
        }
        for (int h = 1; h < D; h <<= 1) {
            __syncthreads();
            for (int t = threadIdx.x; t < D / 2; t += blockDim.x) {
                const int j = (t / h) * 2 * h + (t % h);
                const float a = v[j], b = v[j + h];
                v[j] = __fadd_rn(a, b);
                v[j + h] = __fsub_rn(a, b);
            }
        }
        __syncthreads();
        for (int i = threadIdx.x; i < D; i += blockDim.x) {
            const float y = __fmul_rn(v[i], scale);
            if (out_bf16)
                reinterpret_cast<__nv_bfloat16 *>(Y)[r * D + i] = __float2bfloat16_rn(y);
            else
                reinterpret_cast<float *>(Y)[r * D + i] = y;
        }
    }
}

cudaError_t launch_hadamard(const float *X, int64_t n, int d, const float *mean, const float *sigma, int D,
                            int out_bf16, void *Y, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    const float scale = (float)(1.0 / sqrt((double)D));
    if (D <= 1024) {
        int64_t blocks = (n * 32 + 255) / 256;
        if (blocks > 152 * 8) blocks = 152 * 8;
        const int g = (int)blocks;
        switch (D) {
        case 32: hadamard_warp_kernel<1><<<g, 256, 0, st>>>(X, n, d, mean, sigma, scale, out_bf16, Y); break;
        case 64: hadamard_warp_kernel<2><<<g, 256, 0, st>>>(X, n, d, mean, sigma, scale, out_bf16, Y); break;
        case 128: hadamard_warp_kernel<4><<<g, 256, 0, st>>>(X, n, d, mean, sigma, scale, out_bf16, Y); break;
        case 256: hadamard_warp_kernel<8><<<g, 256, 0, st>>>(X, n, d, mean, sigma, scale, out_bf16, Y); break;
        case 512: hadamard_warp_kernel<16><<<g, 256, 0, st>>>(X, n, d, mean, sigma, scale, out_bf16, Y); break;
        case 1024: hadamard_warp_kernel<32><<<g, 256, 0, st>>>(X, n, d, mean, sigma, scale, out_bf16, Y); break;
        default: return cudaErrorInvalidValue;
        }
        return launched();
    }
    int64_t blocks = n < 152 * 4 ? n : 152 * 4;
    hadamard_block_kernel<<<(int)blocks, 512, 0, st>>>(X, n, d, D, mean, sigma, scale, out_bf16, Y);
    return launched();
}

}  // namespace skm

namespace skm {

// x = y P^T + mu (unprojection of projected centroids, Section 4 "Dimensionality
// Reduction and Vector Search"): 16 x 64 output tiles, y rows and P rows staged
// through shared memory in 32-wide slices; fp32 FMA.
__global__ void __launch_bounds__(256) unproject_kernel(const float *__restrict__ Y, int64_t n, int dout,
                                                        const float *__restrict__ P, const float *__restrict__ mu,
                                                        int d, float *__restrict__ X) {
    __shared__ float ys[16][33];
    __shared__ float ps[64][33];
    const int tx = threadIdx.x & 63, ty = threadIdx.x >> 6;  // 64 x 4 threads, 4 rows each
    const int64_t r0 = (int64_t)blockIdx.y * 16;
    const int c0 = blockIdx.x * 64;
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
    for (int j0 = 0; j0 < dout; j0 += 32) {
        __syncthreads();
        for (int t = threadIdx.x; t < 16 * 32; t += 256) {
            const int rr = t >> 5, jj = t & 31;
            ys[rr][jj] = (r0 + rr < n && j0 + jj < dout) ? Y[(r0 + rr) * dout + j0 + jj] : 0.f;
        }
        for (int t = threadIdx.x; t < 64 * 32; t += 256) {
            const int cc = t >> 5, jj = t & 31;
            ps[cc][jj] = (c0 + cc < d && j0 + jj < dout) ? P[(int64_t)(c0 + cc) * dout + j0 + jj] : 0.f;
        }
        __syncthreads();
#pragma unroll 8
        for (int jj = 0; jj < 32; ++jj) {
            const float pv = ps[tx][jj];
#pragma unroll
            for (int q = 0; q < 4; ++q) acc[q] = __fmaf_rn(ys[ty * 4 + q][jj], pv, acc[q]);
        }
    }
    const int c = c0 + tx;
    if (c < d)
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int64_t r = r0 + ty * 4 + q;
            if (r < n) X[r * d + c] = __fadd_rn(acc[q], mu ? mu[c] : 0.f);
        }
}

cudaError_t launch_unproject(const float *Y, int64_t n, int dout, const float *P, const float *mu, int d,
                             float *X, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    const dim3 grid((unsigned)((d + 63) / 64), (unsigned)((n + 15) / 16));
    if (grid.y > 65535u) return cudaErrorInvalidValue;
    unproject_kernel<<<grid, 256, 0, st>>>(Y, n, dout, P, mu, d, X);
    return launched();
}

// Host-to-device copy by the SMs (skm_copy_from_host): 16-byte loads from the
// mapped host buffer, four in flight per thread, when both ends are 16-byte
// aligned; bytes otherwise and for the tail.  A few dozen blocks fill the host
// link.
__global__ void copy_from_host_kernel(const uint8_t *__restrict__ src, uint8_t *__restrict__ dst, size_t bytes,
                                      size_t n16) {
    const size_t stride = (size_t)gridDim.x * blockDim.x;
    size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x;
    const uint4 *s4 = reinterpret_cast<const uint4 *>(src);
    uint4 *d4 = reinterpret_cast<uint4 *>(dst);
    for (; i + 3 * stride < n16; i += 4 * stride) {
        const uint4 a = s4[i], b = s4[i + stride], c = s4[i + 2 * stride], e = s4[i + 3 * stride];
        d4[i] = a;
        d4[i + stride] = b;
        d4[i + 2 * stride] = c;
        d4[i + 3 * stride] = e;
    }
    for (; i < n16; i += stride) d4[i] = s4[i];
    for (size_t j = 16 * n16 + blockIdx.x * (size_t)blockDim.x + threadIdx.x; j < bytes; j += stride) dst[j] = src[j];
}

cudaError_t launch_copy_from_host(const void *src, void *dst, size_t bytes, cudaStream_t st) {
    if (bytes == 0) return cudaSuccess;
    const bool al = (((uintptr_t)src | (uintptr_t)dst) & 15) == 0;
    const size_t n16 = al ? bytes / 16 : 0;
    const size_t units = al ? n16 : bytes;
    const size_t blocks = (units + 255) / 256;
    copy_from_host_kernel<<<(unsigned)(blocks < 32 ? (blocks < 1 ? 1 : blocks) : 32), 256, 0, st>>>(
        static_cast<const uint8_t *>(src), static_cast<uint8_t *>(dst), bytes, n16);
    return launched();
}

}  // namespace skm
