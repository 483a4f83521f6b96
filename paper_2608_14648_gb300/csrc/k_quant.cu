// Quantization of the points before clustering (Section 3.1): per-dimension
// SQ8 and RabitQ 1-bit codes.  All kernels stream the fp32 points once with
// 128-bit loads where the row length allows it; every float step that decides
// a code is an explicit IEEE fp32 operation (no contraction).
#include "skm_internal.cuh"

namespace skm {

// ---------------------------------------------------------------------------
// Column min/max and column sums: blocks take a contiguous slab of rows; each
// thread owns columns (strided by blockDim.x).  Partial results per slab are
// reduced in a second, fixed-order pass, so the results are deterministic.
// ---------------------------------------------------------------------------
__global__ void colminmax_partial_kernel(const float *__restrict__ X, int64_t n, int d,
                                         float *__restrict__ pmin, float *__restrict__ pmax) {
    const int64_t rows_per = (n + gridDim.x - 1) / gridDim.x;
    const int64_t r0 = (int64_t)blockIdx.x * rows_per;
    const int64_t r1 = min(n, r0 + rows_per);
    for (int c = threadIdx.x; c < d; c += blockDim.x) {
        float lo = INFINITY, hi = -INFINITY;
        for (int64_t r = r0; r < r1; ++r) {
            float v = X[r * d + c];
            lo = fminf(lo, v);
            hi = fmaxf(hi, v);
        }
        pmin[(int64_t)blockIdx.x * d + c] = lo;
        pmax[(int64_t)blockIdx.x * d + c] = hi;
    }
}

cudaError_t launch_colminmax_partial(const float *X, int64_t n, int d, float *pmin, float *pmax,
                                     int nblk, cudaStream_t st) {
    colminmax_partial_kernel<<<nblk, 256, 0, st>>>(X, n, d, pmin, pmax);
    return launched();
}

__global__ void sq8_params_kernel(const float *__restrict__ pmin, const float *__restrict__ pmax,
                                  int nblk, int d, float levels, float *__restrict__ b,
                                  float *__restrict__ s) {
    int c = blockIdx.x * blockDim.x + threadIdx.x;
    if (c >= d) return;
    float lo = INFINITY, hi = -INFINITY;
    for (int i = 0; i < nblk; ++i) {
        lo = fminf(lo, pmin[(int64_t)i * d + c]);
        hi = fmaxf(hi, pmax[(int64_t)i * d + c]);
    }
    float sc = __fdiv_rn(__fsub_rn(hi, lo), levels);
    if (!(sc > 0.0f)) sc = 1.0f;
    b[c] = lo;
    s[c] = sc;
}

cudaError_t launch_sq8_params(const float *pmin, const float *pmax, int nblk, int d, int levels,
                              float *b, float *s, cudaStream_t st) {
    sq8_params_kernel<<<(d + 127) / 128, 128, 0, st>>>(pmin, pmax, nblk, d, (float)levels, b, s);
    return launched();
}

// code = clip(rint((x - b) / s), 0, L) (L = 255 for 8-bit, 15 for 4-bit
// codes, one code per byte); 16 elements per thread per step.
__device__ __forceinline__ uint32_t sq8_code(float x, float b, float s, float top) {
    float q = rintf(__fdiv_rn(__fsub_rn(x, b), s));
    q = (q >= 0.0f) ? q : 0.0f;
    q = fminf(q, top);
    return (uint32_t)q;
}

__global__ void sq8_encode_vec_kernel(const float4 *__restrict__ X, int64_t n16, int d,
                                      const float *__restrict__ b, const float *__restrict__ s,
                                      float top, uint4 *__restrict__ out) {
    // requires d % 16 == 0: a 16-element chunk never crosses a row
    for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < n16;
         t += (int64_t)gridDim.x * blockDim.x) {
        const int c0 = (int)((t * 16) % d);
        float4 v[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) v[q] = X[t * 4 + q];
        uint32_t w[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int c = c0 + 4 * q;
            w[q] = sq8_code(v[q].x, b[c], s[c], top) | (sq8_code(v[q].y, b[c + 1], s[c + 1], top) << 8) |
                   (sq8_code(v[q].z, b[c + 2], s[c + 2], top) << 16) |
                   (sq8_code(v[q].w, b[c + 3], s[c + 3], top) << 24);
        }
        out[t] = make_uint4(w[0], w[1], w[2], w[3]);
    }
}

__global__ void sq8_encode_scalar_kernel(const float *__restrict__ X, int64_t total, int d,
                                         const float *__restrict__ b, const float *__restrict__ s,
                                         float top, uint8_t *__restrict__ out) {
    for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < total;
         t += (int64_t)gridDim.x * blockDim.x) {
        const int c = (int)(t % d);
        out[t] = (uint8_t)sq8_code(X[t], b[c], s[c], top);
    }
}

static int grid_for(int64_t work, int threads) {
    int64_t g = (work + threads - 1) / threads;
    const int64_t cap = 152LL * 16;  // 16 resident blocks per SM on 152 SMs
    if (g > cap) g = cap;
    if (g < 1) g = 1;
    return (int)g;
}

cudaError_t launch_sq8_encode(const float *X, int64_t n, int d, const float *b, const float *s,
                              int levels, uint8_t *codes, cudaStream_t st) {
    const int64_t total = n * d;
    const float top = (float)levels;
    if (d % 16 == 0 && (((uintptr_t)X | (uintptr_t)codes) & 15) == 0) {
        const int64_t n16 = total / 16;
        sq8_encode_vec_kernel<<<grid_for(n16, 256), 256, 0, st>>>(
            reinterpret_cast<const float4 *>(X), n16, d, b, s, top, reinterpret_cast<uint4 *>(codes));
    } else {
        sq8_encode_scalar_kernel<<<grid_for(total, 256), 256, 0, st>>>(X, total, d, b, s, top, codes);
    }
    return launched();
}

__global__ void sq8_decode_kernel(const uint8_t *__restrict__ codes, int64_t total, int d,
                                  const float *__restrict__ b, const float *__restrict__ s,
                                  float *__restrict__ Y) {
    for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < total;
         t += (int64_t)gridDim.x * blockDim.x) {
        const int c = (int)(t % d);
        Y[t] = __fadd_rn(__fmul_rn((float)codes[t], s[c]), b[c]);
    }
}

cudaError_t launch_sq8_decode(const uint8_t *codes, int64_t n, int d, const float *b,
                              const float *s, float *Y, cudaStream_t st) {
    const int64_t total = n * d;
    sq8_decode_kernel<<<grid_for(total, 256), 256, 0, st>>>(codes, total, d, b, s, Y);
    return launched();
}

// Column sums: each block sums a contiguous run of rows; a thread owns
// columns c, c + 256, ... and keeps a Kahan-compensated fp32 sum per column
// (error about 2^-23 of the sum of magnitudes), written out as fp64.
__global__ void colsum_partial_kernel(const float *__restrict__ X, int64_t n, int d,
                                      double *__restrict__ psum) {
    const int64_t rows_per = (n + gridDim.x - 1) / gridDim.x;
    const int64_t r0 = (int64_t)blockIdx.x * rows_per;
    const int64_t r1 = min(n, r0 + rows_per);
    for (int c = threadIdx.x; c < d; c += blockDim.x) {
        float s = 0.0f, comp = 0.0f;
        int64_t r = r0;
        for (; r + 4 <= r1; r += 4) {
            float v[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) v[u] = __ldg(X + (r + u) * d + c);
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const float y = __fsub_rn(v[u], comp);
                const float t = __fadd_rn(s, y);
                comp = __fsub_rn(__fsub_rn(t, s), y);
                s = t;
            }
        }
        for (; r < r1; ++r) {
            const float y = __fsub_rn(__ldg(X + r * d + c), comp);
            const float t = __fadd_rn(s, y);
            comp = __fsub_rn(__fsub_rn(t, s), y);
            s = t;
        }
        psum[(int64_t)blockIdx.x * d + c] = (double)s - (double)comp;
    }
}

cudaError_t launch_colsum_partial(const float *X, int64_t n, int d, double *psum, int nblk,
                                  cudaStream_t st) {
    colsum_partial_kernel<<<nblk, 256, 0, st>>>(X, n, d, psum);
    return launched();
}

__global__ void colmean_finish_kernel(const double *__restrict__ psum, int nblk, int d, int64_t n,
                                      float *__restrict__ m, double *__restrict__ mean_d) {
    int c = blockIdx.x * blockDim.x + threadIdx.x;
    if (c >= d) return;
    double acc = 0.0;
    for (int i = 0; i < nblk; ++i) acc += psum[(int64_t)i * d + c];
    const double mu = __ddiv_rn(acc, (double)n);
    if (m) m[c] = __double2float_rn(mu);
    if (mean_d) mean_d[c] = mu;
}

cudaError_t launch_colmean_finish(const double *psum, int nblk, int d, int64_t n, float *m,
                                  double *mean_d, cudaStream_t st) {
    colmean_finish_kernel<<<(d + 127) / 128, 128, 0, st>>>(psum, nblk, d, n, m, mean_d);
    return launched();
}

// ---------------------------------------------------------------------------
// RabitQ 1-bit encode: one warp per point.  Lane l handles dimensions
// 32w + l; the sign bits of a 32-dimension group are one __ballot_sync.
// ||r||^2 and ||r||_1: Kahan-compensated fp32 lane sums (relative error about
// 2^-23), then an fp64 xor-tree across lanes; F = sqrt(d) ||r||^2 / ||r||_1
// is evaluated in fp64 and rounded once.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void kahan_add(float &s, float &c, float v) {
    const float y = __fsub_rn(v, c);
    const float t = __fadd_rn(s, y);
    c = __fsub_rn(__fsub_rn(t, s), y);
    s = t;
}

constexpr int ENC_UNROLL = 8;

__global__ void rbq1_encode_kernel(const float *__restrict__ X, int64_t n, int d,
                                   const float *__restrict__ m, uint32_t *__restrict__ codes,
                                   float *__restrict__ nx2, float *__restrict__ F,
                                   int32_t *__restrict__ popx) {
    const int lane = threadIdx.x & 31;
    const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int W = (d + 31) >> 5;
    const double sqrt_d = sqrt((double)d);
    for (int64_t p = warp; p < n; p += nwarps) {
        const float *x = X + p * d;
        float s2 = 0.0f, c2 = 0.0f, s1 = 0.0f, c1 = 0.0f;
        int pc = 0;
        for (int w0 = 0; w0 < W; w0 += ENC_UNROLL) {
            float v[ENC_UNROLL];
#pragma unroll
            for (int u = 0; u < ENC_UNROLL; ++u) {
                const int i = 32 * (w0 + u) + lane;
                v[u] = (w0 + u < W && i < d) ? __ldg(x + i) : 0.0f;
            }
#pragma unroll
            for (int u = 0; u < ENC_UNROLL; ++u) {
                const int w = w0 + u;
                if (w < W) {  // warp-uniform
                    const int i = 32 * w + lane;
                    const float r = i < d ? __fsub_rn(v[u], __ldg(m + i)) : 0.0f;
                    const unsigned bits = __ballot_sync(0xffffffffu, r > 0.0f);
                    kahan_add(s2, c2, __fmul_rn(r, r));
                    kahan_add(s1, c1, fabsf(r));
                    if (lane == 0) {
                        codes[p * W + w] = bits;
                        pc += __popc(bits);
                    }
                }
            }
        }
        double t2 = (double)s2 - (double)c2, t1 = (double)s1 - (double)c1;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            t2 += __shfl_xor_sync(0xffffffffu, t2, o);
            t1 += __shfl_xor_sync(0xffffffffu, t1, o);
        }
        if (lane == 0) {
            nx2[p] = __double2float_rn(t2);
            F[p] = (t1 > 0.0) ? __double2float_rn(__ddiv_rn(__dmul_rn(sqrt_d, t2), t1)) : 0.0f;
            popx[p] = pc;
        }
    }
}

cudaError_t launch_rbq1_encode(const float *X, int64_t n, int d, const float *m, uint32_t *codes,
                               float *nx2, float *F, int32_t *popx, cudaStream_t st) {
    const int threads = 256;
    rbq1_encode_kernel<<<grid_for(n * 32, threads), threads, 0, st>>>(X, n, d, m, codes, nx2, F,
                                                                      popx);
    return launched();
}

// max F (F >= 0, so the IEEE bit pattern orders like an unsigned integer),
// then e = 24 - ceil(log2 max F), e = 0 when max F == 0.
__global__ void rbq1_maxbits_kernel(const float *__restrict__ F, int64_t n,
                                    unsigned int *__restrict__ maxbits) {
    unsigned int mx = 0;
    for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < n;
         t += (int64_t)gridDim.x * blockDim.x) {
        const float f = F[t];
        if (f > 0.0f) mx = max(mx, __float_as_uint(f));
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = max(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    if ((threadIdx.x & 31) == 0 && mx) atomicMax(maxbits, mx);
}

__global__ void rbq1_exponent_kernel(const unsigned int *__restrict__ maxbits, int *__restrict__ e) {
    const float mx = __uint_as_float(*maxbits);
    if (!(mx > 0.0f)) {
        *e = 0;
        return;
    }
    int ex;
    const double fr = frexp((double)mx, &ex);
    const int c = (fr == 0.5) ? ex - 1 : ex;
    *e = 24 - c;
}

cudaError_t launch_rbq1_exponent(const float *F, int64_t n, unsigned int *maxbits, int *e_dev,
                                 cudaStream_t st) {
    cudaError_t err = cudaMemsetAsync(maxbits, 0, sizeof(unsigned int), st);
    if (err != cudaSuccess) return err;
    rbq1_maxbits_kernel<<<grid_for(n, 256), 256, 0, st>>>(F, n, maxbits);
    rbq1_exponent_kernel<<<1, 1, 0, st>>>(maxbits, e_dev);
    return launched(2);
}

}  // namespace skm
