// Quantization of the points before clustering (Section 3.1): per-dimension
// SQ8 and RabitQ 1-bit codes.  All kernels stream the fp32 points once with
// 128-bit loads where the row length allows it; every float step that decides
// a code is an explicit IEEE fp32 operation (no contraction).
#include <string.h>

#include "skm_internal.cuh"

namespace skm {

static int grid_for(int64_t work, int threads) {
    int64_t g = (work + threads - 1) / threads;
    const int64_t cap = 152LL * 16;  // grid-stride kernels: at most 16 blocks per SM of 152
    if (g > cap) g = cap;
    if (g < 1) g = 1;
    return (int)g;
}


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

// d % 4 == 0: 512-thread blocks split into P row phases of G = min(d/4, 512)
// threads; a thread owns float4 column groups g, g + G, ... over its phase's
// contiguous part of the block's rows (four rows of loads in flight), and the
// phases are folded in phase order through shared memory.  With the grid of
// two blocks per SM, the bytes in flight come from 32 resident warps per SM.
constexpr int COL_THREADS = 512;
constexpr int COL_ROWS = 4;

struct ColPhase {
    int G, P, ph, g0;
    int64_t a, b;  // the phase's rows [a, b)
};

__device__ __forceinline__ ColPhase col_phase(int64_t n, int d4) {
    ColPhase c;
    c.G = min(d4, (int)blockDim.x);
    c.P = blockDim.x / c.G;
    c.ph = threadIdx.x / c.G;
    c.g0 = threadIdx.x % c.G;
    const int64_t rows_per = (n + gridDim.x - 1) / gridDim.x;
    const int64_t r0 = min(n, (int64_t)blockIdx.x * rows_per), r1 = min(n, r0 + rows_per);
    const int64_t sub = (r1 - r0 + c.P - 1) / c.P;
    c.a = min(r1, r0 + c.ph * sub);
    c.b = min(r1, c.a + sub);
    return c;
}

__global__ void __launch_bounds__(COL_THREADS, 2)
    colminmax_partial_v4_kernel(const float4 *__restrict__ X, int64_t n, int d, float *__restrict__ pmin,
                                float *__restrict__ pmax) {
    extern __shared__ float4 col_sh[];
    const int d4 = d >> 2;
    const ColPhase cp = col_phase(n, d4);
    float4 *shlo = col_sh, *shhi = col_sh + (int64_t)cp.P * d4;
    if (cp.ph < cp.P) {
        for (int g = cp.g0; g < d4; g += cp.G) {
            float4 lo = make_float4(INFINITY, INFINITY, INFINITY, INFINITY);
            float4 hi = make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
            auto take = [&](const float4 &v) {
                lo = make_float4(fminf(lo.x, v.x), fminf(lo.y, v.y), fminf(lo.z, v.z), fminf(lo.w, v.w));
                hi = make_float4(fmaxf(hi.x, v.x), fmaxf(hi.y, v.y), fmaxf(hi.z, v.z), fmaxf(hi.w, v.w));
            };
            int64_t r = cp.a;
            for (; r + COL_ROWS <= cp.b; r += COL_ROWS) {
                float4 v[COL_ROWS];
#pragma unroll
                for (int u = 0; u < COL_ROWS; ++u) v[u] = __ldg(X + (r + u) * d4 + g);
#pragma unroll
                for (int u = 0; u < COL_ROWS; ++u) take(v[u]);
            }
            for (; r < cp.b; ++r) take(__ldg(X + r * d4 + g));
            if (cp.P == 1) {
                reinterpret_cast<float4 *>(pmin + (int64_t)blockIdx.x * d)[g] = lo;
                reinterpret_cast<float4 *>(pmax + (int64_t)blockIdx.x * d)[g] = hi;
            } else {
                shlo[cp.ph * d4 + g] = lo;
                shhi[cp.ph * d4 + g] = hi;
            }
        }
    }
    if (cp.P == 1) return;
    __syncthreads();
    for (int g = threadIdx.x; g < d4; g += blockDim.x) {
        float4 lo = shlo[g], hi = shhi[g];
        for (int q = 1; q < cp.P; ++q) {
            const float4 l = shlo[q * d4 + g], h = shhi[q * d4 + g];
            lo = make_float4(fminf(lo.x, l.x), fminf(lo.y, l.y), fminf(lo.z, l.z), fminf(lo.w, l.w));
            hi = make_float4(fmaxf(hi.x, h.x), fmaxf(hi.y, h.y), fmaxf(hi.z, h.z), fmaxf(hi.w, h.w));
        }
        reinterpret_cast<float4 *>(pmin + (int64_t)blockIdx.x * d)[g] = lo;
        reinterpret_cast<float4 *>(pmax + (int64_t)blockIdx.x * d)[g] = hi;
    }
}

// shared memory of the two phase-split column kernels: P * d4 <= 512 when
// P > 1, so P * d <= 2048 values
static size_t col_smem(int d, size_t per_col) {
    const int d4 = d / 4;
    const int G = d4 < COL_THREADS ? d4 : COL_THREADS;
    const int P = COL_THREADS / G;
    return P > 1 ? (size_t)P * d * per_col : 0;
}

cudaError_t launch_colminmax_partial(const float *X, int64_t n, int d, float *pmin, float *pmax,
                                     int nblk, cudaStream_t st) {
    if (d % 4 == 0 && (((uintptr_t)X | (uintptr_t)pmin | (uintptr_t)pmax) & 15) == 0) {
        const size_t sh = 2 * col_smem(d, sizeof(float));  // at most 16 KB
        colminmax_partial_v4_kernel<<<nblk, COL_THREADS, sh, st>>>(reinterpret_cast<const float4 *>(X), n, d,
                                                                   pmin, pmax);
    } else {
        colminmax_partial_kernel<<<nblk, 256, 0, st>>>(X, n, d, pmin, pmax);
    }
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
// codes, one code per byte).
__device__ __forceinline__ uint32_t sq8_code(float x, float b, float s, float top) {
    float q = rintf(__fdiv_rn(__fsub_rn(x, b), s));
    q = (q >= 0.0f) ? q : 0.0f;
    q = fminf(q, top);
    return (uint32_t)q;
}

// The same code with one multiplication in place of the division: with
// rs = fl(1/s) a normal number, q' = fl(a rs) (a = fl(x - b)) is within
// (2^-23 + 2^-24 + 2^-48) |a/s| of the correctly rounded quotient q.  Only
// quotients in [-0.5, L + 0.5] decide a code, and there |a/s| <= 256, so the two
// are within 2^-14.4: when q' is more than 2^-13 away from every half-integer
// they round to the same integer (quotients beyond that range clip to the same
// end on both sides); otherwise (and for inf / NaN, including rs = NaN passed
// for a subnormal 1/s) the quotient is taken by the IEEE division.
__device__ __forceinline__ uint32_t sq8_code_rs(float x, float b, float s, float rs, float top) {
    const float a = __fsub_rn(x, b);
    const float q = __fmul_rn(a, rs);
    float t = rintf(q);
    if (!(fabsf(__fsub_rn(q, t)) < 0.5f - 0x1p-13f)) t = rintf(__fdiv_rn(a, s));
    t = (t >= 0.0f) ? t : 0.0f;
    t = fminf(t, top);
    return (uint32_t)t;
}

// d % 4 == 0: one warp per row, lane l takes the float4 at dimensions
// 128t + 4l .. + 3 and writes their four codes as one 32-bit word, so the
// (b, s) loads and the code stores are contiguous across the warp; a row's
// loads (up to SQ_V4 float4 per lane) are issued before use.  The block keeps
// fl(1/s) per column in shared memory (sq8_code_rs).
constexpr int SQ_V4 = 8;
constexpr int SQ_RS_MAX_D = 8192;  // 32 KB of reciprocals

__global__ void sq8_encode_rows_kernel(const float4 *__restrict__ X, int64_t n, int d,
                                       const float4 *__restrict__ b, const float4 *__restrict__ s,
                                       float top, uint32_t *__restrict__ out) {
    extern __shared__ float4 sq_rs[];
    for (int c = threadIdx.x; c < (d >> 2); c += blockDim.x) {
        const float4 sv = __ldg(s + c);
        auto rcp = [](float v) {
            const float r = __frcp_rn(v);
            return fabsf(r) >= 0x1p-126f ? r : __int_as_float(0x7fffffff);
        };
        sq_rs[c] = make_float4(rcp(sv.x), rcp(sv.y), rcp(sv.z), rcp(sv.w));
    }
    __syncthreads();
    const int lane = threadIdx.x & 31;
    const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int d4 = d >> 2;
    for (int64_t p = warp; p < n; p += nwarps) {
        const float4 *x = X + p * d4;
        uint32_t *o = out + p * d4;
        for (int t0 = 0; 32 * t0 < d4; t0 += SQ_V4) {
            float4 v[SQ_V4];
#pragma unroll
            for (int u = 0; u < SQ_V4; ++u) {
                const int j = 32 * (t0 + u) + lane;
                if (j < d4) v[u] = __ldg(x + j);
            }
#pragma unroll
            for (int u = 0; u < SQ_V4; ++u) {
                const int j = 32 * (t0 + u) + lane;
                if (j < d4) {
                    const float4 bb = __ldg(b + j), ss = __ldg(s + j), rr = sq_rs[j];
                    o[j] = sq8_code_rs(v[u].x, bb.x, ss.x, rr.x, top) |
                           (sq8_code_rs(v[u].y, bb.y, ss.y, rr.y, top) << 8) |
                           (sq8_code_rs(v[u].z, bb.z, ss.z, rr.z, top) << 16) |
                           (sq8_code_rs(v[u].w, bb.w, ss.w, rr.w, top) << 24);
                }
            }
        }
    }
}

// d % 4 == 0 and d <= 1024: the layout of sq8_encode_rows_kernel with
// NV = ceil(d / 128) float4 per lane and the next row's loads in flight while
// the current row is coded.
template <int NV>
__global__ void __launch_bounds__(256) sq8_encode_pf_kernel(const float4 *__restrict__ X, int64_t n, int d,
                                                            const float4 *__restrict__ b,
                                                            const float4 *__restrict__ s, float top,
                                                            uint32_t *__restrict__ out) {
    __shared__ float4 rs_sh[256];
    for (int c = threadIdx.x; c < (d >> 2); c += blockDim.x) {
        const float4 sv = __ldg(s + c);
        auto rcp = [](float v) {
            const float r = __frcp_rn(v);
            return fabsf(r) >= 0x1p-126f ? r : __int_as_float(0x7fffffff);
        };
        rs_sh[c] = make_float4(rcp(sv.x), rcp(sv.y), rcp(sv.z), rcp(sv.w));
    }
    __syncthreads();
    const int lane = threadIdx.x & 31;
    const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int d4 = d >> 2;
    auto load_row = [&](int64_t p, float4(&v)[NV]) {
        const float4 *x = X + p * d4;
#pragma unroll
        for (int u = 0; u < NV; ++u) {
            const int j = 32 * u + lane;
            if (j < d4) v[u] = __ldg(x + j);
        }
    };
    float4 v[NV];
    if (warp < n) load_row(warp, v);
    for (int64_t p = warp; p < n; p += nwarps) {
        float4 nxt[NV];
        if (p + nwarps < n) load_row(p + nwarps, nxt);
        uint32_t *o = out + p * d4;
#pragma unroll
        for (int u = 0; u < NV; ++u) {
            const int j = 32 * u + lane;
            if (j < d4) {
                const float4 bb = __ldg(b + j), rr = rs_sh[j];
                const float ax = __fsub_rn(v[u].x, bb.x), ay = __fsub_rn(v[u].y, bb.y);
                const float az = __fsub_rn(v[u].z, bb.z), aw = __fsub_rn(v[u].w, bb.w);
                const float qx = __fmul_rn(ax, rr.x), qy = __fmul_rn(ay, rr.y);
                const float qz = __fmul_rn(az, rr.z), qw = __fmul_rn(aw, rr.w);
                float tx = rintf(qx), ty = rintf(qy), tz = rintf(qz), tw = rintf(qw);
                // any quotient near a half-integer (or not finite): the divisions decide
                constexpr float lim = 0.5f - 0x1p-13f;
                if (!(fmaxf(fmaxf(fabsf(__fsub_rn(qx, tx)), fabsf(__fsub_rn(qy, ty))),
                            fmaxf(fabsf(__fsub_rn(qz, tz)), fabsf(__fsub_rn(qw, tw)))) < lim) ||
                    !(fabsf(qx) + fabsf(qy) + fabsf(qz) + fabsf(qw) < INFINITY)) {
                    const float4 ss = __ldg(s + j);
                    if (!(fabsf(__fsub_rn(qx, tx)) < lim)) tx = rintf(__fdiv_rn(ax, ss.x));
                    if (!(fabsf(__fsub_rn(qy, ty)) < lim)) ty = rintf(__fdiv_rn(ay, ss.y));
                    if (!(fabsf(__fsub_rn(qz, tz)) < lim)) tz = rintf(__fdiv_rn(az, ss.z));
                    if (!(fabsf(__fsub_rn(qw, tw)) < lim)) tw = rintf(__fdiv_rn(aw, ss.w));
                }
                auto clip = [top](float t) { return (uint32_t)fminf(t >= 0.0f ? t : 0.0f, top); };
                o[j] = clip(tx) | (clip(ty) << 8) | (clip(tz) << 16) | (clip(tw) << 24);
            }
        }
#pragma unroll
        for (int u = 0; u < NV; ++u) v[u] = nxt[u];
    }
}

template <int NV>
static void sq8_pf_launch(const float *X, int64_t n, int d, const float *b, const float *s, float top,
                          uint8_t *codes, cudaStream_t st) {
    sq8_encode_pf_kernel<NV><<<grid_for(n * 32, 256), 256, 0, st>>>(
        reinterpret_cast<const float4 *>(X), n, d, reinterpret_cast<const float4 *>(b),
        reinterpret_cast<const float4 *>(s), top, reinterpret_cast<uint32_t *>(codes));
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

cudaError_t launch_sq8_encode(const float *X, int64_t n, int d, const float *b, const float *s,
                              int levels, uint8_t *codes, cudaStream_t st) {
    const int64_t total = n * d;
    const float top = (float)levels;
    const bool v4 = d % 4 == 0 && (((uintptr_t)X | (uintptr_t)b | (uintptr_t)s) & 15) == 0 &&
                    ((uintptr_t)codes & 3) == 0;
    if (v4 && d <= 1024) {
        switch ((d + 127) / 128) {
        case 1: sq8_pf_launch<1>(X, n, d, b, s, top, codes, st); break;
        case 2: sq8_pf_launch<2>(X, n, d, b, s, top, codes, st); break;
        case 3: sq8_pf_launch<3>(X, n, d, b, s, top, codes, st); break;
        case 4: sq8_pf_launch<4>(X, n, d, b, s, top, codes, st); break;
        case 5: sq8_pf_launch<5>(X, n, d, b, s, top, codes, st); break;
        case 6: sq8_pf_launch<6>(X, n, d, b, s, top, codes, st); break;
        case 7: sq8_pf_launch<7>(X, n, d, b, s, top, codes, st); break;
        default: sq8_pf_launch<8>(X, n, d, b, s, top, codes, st); break;
        }
    } else if (v4 && d <= SQ_RS_MAX_D) {
        sq8_encode_rows_kernel<<<grid_for(n * 32, 256), 256, (size_t)d * sizeof(float), st>>>(
            reinterpret_cast<const float4 *>(X), n, d, reinterpret_cast<const float4 *>(b),
            reinterpret_cast<const float4 *>(s), top, reinterpret_cast<uint32_t *>(codes));
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

// d % 4 == 0: the phase split of colminmax_partial_v4_kernel; each phase keeps
// the Kahan recurrence per column in row order over its rows, and the phases'
// compensated sums are added in fp64 in phase order.
__device__ __forceinline__ void kahan_col(float &s, float &comp, float v) {
    const float y = __fsub_rn(v, comp);
    const float t = __fadd_rn(s, y);
    comp = __fsub_rn(__fsub_rn(t, s), y);
    s = t;
}

__global__ void __launch_bounds__(COL_THREADS, 2)
    colsum_partial_v4_kernel(const float4 *__restrict__ X, int64_t n, int d, double *__restrict__ psum) {
    extern __shared__ double col_shd[];
    const int d4 = d >> 2;
    const ColPhase cp = col_phase(n, d4);
    if (cp.ph < cp.P) {
        for (int g = cp.g0; g < d4; g += cp.G) {
            float4 s = make_float4(0.0f, 0.0f, 0.0f, 0.0f), c = s;
            auto take = [&](const float4 &v) {
                kahan_col(s.x, c.x, v.x);
                kahan_col(s.y, c.y, v.y);
                kahan_col(s.z, c.z, v.z);
                kahan_col(s.w, c.w, v.w);
            };
            int64_t r = cp.a;
            for (; r + COL_ROWS <= cp.b; r += COL_ROWS) {
                float4 v[COL_ROWS];
#pragma unroll
                for (int u = 0; u < COL_ROWS; ++u) v[u] = __ldg(X + (r + u) * d4 + g);
#pragma unroll
                for (int u = 0; u < COL_ROWS; ++u) take(v[u]);
            }
            for (; r < cp.b; ++r) take(__ldg(X + r * d4 + g));
            double *o = cp.P == 1 ? psum + (int64_t)blockIdx.x * d + 4 * g : col_shd + (int64_t)cp.ph * d + 4 * g;
            o[0] = (double)s.x - (double)c.x;
            o[1] = (double)s.y - (double)c.y;
            o[2] = (double)s.z - (double)c.z;
            o[3] = (double)s.w - (double)c.w;
        }
    }
    if (cp.P == 1) return;
    __syncthreads();
    for (int c = threadIdx.x; c < d; c += blockDim.x) {
        double acc = col_shd[c];
        for (int q = 1; q < cp.P; ++q) acc = __dadd_rn(acc, col_shd[(int64_t)q * d + c]);
        psum[(int64_t)blockIdx.x * d + c] = acc;
    }
}

cudaError_t launch_colsum_partial(const float *X, int64_t n, int d, double *psum, int nblk,
                                  cudaStream_t st) {
    if (d % 4 == 0 && ((uintptr_t)X & 15) == 0) {
        const size_t sh = col_smem(d, sizeof(double));  // at most 16 KB
        colsum_partial_v4_kernel<<<nblk, COL_THREADS, sh, st>>>(reinterpret_cast<const float4 *>(X), n, d, psum);
    } else {
        colsum_partial_kernel<<<nblk, 256, 0, st>>>(X, n, d, psum);
    }
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

// ---------------------------------------------------------------------------
// The RabitQ dataset mean in exact fixed point: with 2^(E-1) <= max |x| < 2^E
// over all points and L = ceil(log2 n), s = 61 - L - E; every coordinate
// enters as rint(x 2^s) (an integer below 2^(61-L) in magnitude, formed from
// the fp32 significand by fixed_rint), the column sums are exact int64 sums
// (at most 2^61 in magnitude, order-independent), and m = fl32(S / (n 2^s))
// with one fp64 division.  Row shards that use the same s and n add up to
// exactly the single-process sums.
// ---------------------------------------------------------------------------
__host__ __device__ inline int mean_scale_of(unsigned amax_bits, int64_t n) {
    if (amax_bits == 0) return 0;
    const unsigned ef = (amax_bits >> 23) & 0xffu;
    int E;
    if (ef == 0) {  // subnormal maximum: mantissa m 2^-149, m < 2^23
        unsigned mm = amax_bits & 0x7fffffu;
        int hb = 0;
        while (mm >> (hb + 1)) ++hb;
        E = hb + 1 - 149;
    } else {
        E = (int)ef - 127 + 1;
    }
    int lg = 0;
    while ((int64_t(1) << lg) < n) ++lg;
    return 61 - lg - E;
}

__global__ void absmax_bits_kernel(const float *__restrict__ X, int64_t count, unsigned *__restrict__ bits) {
    unsigned mx = 0;
    const int64_t t0 = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
    const int64_t st = (int64_t)gridDim.x * blockDim.x;
    if (((uintptr_t)X & 15) == 0) {
        const int64_t c4 = count >> 2;
        const uint4 *X4 = reinterpret_cast<const uint4 *>(X);
        for (int64_t i = t0; i < c4; i += st) {
            const uint4 v = __ldg(X4 + i);
            mx = max(mx, max(max(v.x & 0x7fffffffu, v.y & 0x7fffffffu), max(v.z & 0x7fffffffu, v.w & 0x7fffffffu)));
        }
        for (int64_t i = 4 * c4 + t0; i < count; i += st) mx = max(mx, __float_as_uint(X[i]) & 0x7fffffffu);
    } else {
        for (int64_t i = t0; i < count; i += st) mx = max(mx, __float_as_uint(X[i]) & 0x7fffffffu);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = max(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    if ((threadIdx.x & 31) == 0 && mx) atomicMax(bits, mx);
}

__global__ void mean_scale_kernel(const unsigned *__restrict__ bits, int64_t n, int *__restrict__ s_out) {
    *s_out = mean_scale_of(*bits, n);
}

// S[c] += sum over this launch's rows of rint(x_rc 2^s); blocks take row
// ranges, threads columns (four at a time when rows are 16-byte aligned).
__global__ void colsum_fixed_kernel(const float *__restrict__ X, int64_t n, int d, const int *__restrict__ s_dev,
                                    int s_host, unsigned long long *__restrict__ S) {
    const int s = s_dev ? *s_dev : s_host;
    const int64_t per = (n + gridDim.x - 1) / gridDim.x;
    const int64_t r0 = (int64_t)blockIdx.x * per, r1 = min(n, r0 + per);
    if (r0 >= r1) return;
    if ((d & 3) == 0 && ((uintptr_t)X & 15) == 0) {
        const int d4 = d >> 2;
        const float4 *X4 = reinterpret_cast<const float4 *>(X);
        for (int g = threadIdx.x; g < d4; g += blockDim.x) {
            int64_t a0 = 0, a1 = 0, a2 = 0, a3 = 0;
            int64_t r = r0;
            for (; r + 4 <= r1; r += 4) {
                float4 v[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) v[u] = __ldg(X4 + (r + u) * d4 + g);
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    a0 += fixed_rint(v[u].x, s);
                    a1 += fixed_rint(v[u].y, s);
                    a2 += fixed_rint(v[u].z, s);
                    a3 += fixed_rint(v[u].w, s);
                }
            }
            for (; r < r1; ++r) {
                const float4 v = __ldg(X4 + r * d4 + g);
                a0 += fixed_rint(v.x, s);
                a1 += fixed_rint(v.y, s);
                a2 += fixed_rint(v.z, s);
                a3 += fixed_rint(v.w, s);
            }
            atomicAdd(S + 4 * g, (unsigned long long)a0);
            atomicAdd(S + 4 * g + 1, (unsigned long long)a1);
            atomicAdd(S + 4 * g + 2, (unsigned long long)a2);
            atomicAdd(S + 4 * g + 3, (unsigned long long)a3);
        }
    } else {
        for (int c = threadIdx.x; c < d; c += blockDim.x) {
            int64_t a = 0;
            for (int64_t r = r0; r < r1; ++r) a += fixed_rint(__ldg(X + r * d + c), s);
            atomicAdd(S + c, (unsigned long long)a);
        }
    }
}

__global__ void mean_fixed_finish_kernel(const unsigned long long *__restrict__ S, int d, int64_t n,
                                         const int *__restrict__ s_dev, int s_host, float *__restrict__ m) {
    const int c = blockIdx.x * blockDim.x + threadIdx.x;
    if (c >= d) return;
    const int s = s_dev ? *s_dev : s_host;
    const double q = __ddiv_rn(__ll2double_rn((long long)S[c]), scalbn((double)n, s));
    m[c] = __double2float_rn(q);
}

int host_mean_scale(float amax, int64_t n) {
    uint32_t b;
    memcpy(&b, &amax, sizeof(b));
    return mean_scale_of(b & 0x7fffffffu, n);
}

cudaError_t launch_absmax_bits(const float *X, int64_t count, unsigned *bits, cudaStream_t st) {
    cudaError_t e = cudaMemsetAsync(bits, 0, sizeof(unsigned), st);
    if (e != cudaSuccess) return e;
    int64_t blocks = (count / 4 + 255) / 256;
    blocks = blocks < 1 ? 1 : (blocks > 152 * 8 ? 152 * 8 : blocks);
    absmax_bits_kernel<<<(unsigned)blocks, 256, 0, st>>>(X, count, bits);
    return launched();
}

cudaError_t launch_mean_fixed(const float *X, int64_t n, int d, unsigned *bits, int *s_dev, unsigned long long *S,
                              float *m, cudaStream_t st) {
    cudaError_t e = launch_absmax_bits(X, n * (int64_t)d, bits, st);
    if (e != cudaSuccess) return e;
    mean_scale_kernel<<<1, 1, 0, st>>>(bits, n, s_dev);
    if ((e = launched()) != cudaSuccess) return e;
    if ((e = launch_colsum_fixed(X, n, d, s_dev, 0, S, true, st)) != cudaSuccess) return e;
    return launch_mean_fixed_finish(S, d, n, s_dev, 0, m, st);
}

cudaError_t launch_colsum_fixed(const float *X, int64_t n, int d, const int *s_dev, int s_host,
                                unsigned long long *S, bool zero_first, cudaStream_t st) {
    if (zero_first) {
        const cudaError_t e = cudaMemsetAsync(S, 0, sizeof(unsigned long long) * (size_t)d, st);
        if (e != cudaSuccess) return e;
    }
    int64_t blocks = (n + 1023) / 1024;
    blocks = blocks < 1 ? 1 : (blocks > 152 * 8 ? 152 * 8 : blocks);
    colsum_fixed_kernel<<<(unsigned)blocks, 256, 0, st>>>(X, n, d, s_dev, s_host, S);
    return launched();
}

cudaError_t launch_mean_fixed_finish(const unsigned long long *S, int d, int64_t n, const int *s_dev, int s_host,
                                     float *m, cudaStream_t st) {
    mean_fixed_finish_kernel<<<(d + 127) / 128, 128, 0, st>>>(S, d, n, s_dev, s_host, m);
    return launched();
}

cudaError_t launch_colmean_finish(const double *psum, int nblk, int d, int64_t n, float *m,
                                  double *mean_d, cudaStream_t st) {
    colmean_finish_kernel<<<(d + 127) / 128, 128, 0, st>>>(psum, nblk, d, n, m, mean_d);
    return launched();
}

// ---------------------------------------------------------------------------
// RabitQ 1-bit encode: one warp per point, r = x - m.  ||r||^2 and ||r||_1 are
// Kahan-compensated fp32 lane sums (relative error about 2^-23); the 32 lane
// pairs (s, -c) are folded across the warp as double-float numbers (error-free
// TwoSum of the leading parts, trailing parts added), so the row total keeps
// about 40 bits before its single rounding to fp32.  F = sqrt(d) ||r||^2 /
// ||r||_1 then takes three fp32 roundings (relative error below 2^-22).  No
// fp64 instruction runs per point: GB300 issues fp64 at a small fraction of the
// fp32 rate, and a per-row fp64 tail bounded the former version.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void kahan_add(float &s, float &c, float v) {
    const float y = __fsub_rn(v, c);
    const float t = __fadd_rn(s, y);
    c = __fsub_rn(__fsub_rn(t, s), y);
    s = t;
}

// (hi, lo) += (h2, l2) for double-float numbers: TwoSum of the leading parts,
// trailing parts added to the error, renormalised by FastTwoSum.
__device__ __forceinline__ void df_add(float &hi, float &lo, float h2, float l2) {
    const float s = __fadd_rn(hi, h2);
    const float bb = __fsub_rn(s, hi);
    const float e = __fadd_rn(__fsub_rn(hi, __fsub_rn(s, bb)), __fsub_rn(h2, bb));
    const float t = __fadd_rn(e, __fadd_rn(lo, l2));
    hi = __fadd_rn(s, t);
    lo = __fsub_rn(t, __fsub_rn(hi, s));
}

// Folds the lane sums of one point and writes ||r||^2, F and popcount(code).
__device__ __forceinline__ void rbq1_row_finish(float s2, float c2, float s1, float c1, int pc, int lane,
                                                float sqrt_d, float *nx2, float *F, int32_t *popx) {
    float h2 = s2, l2 = -c2, h1 = s1, l1 = -c1;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float a = __shfl_xor_sync(0xffffffffu, h2, o), b = __shfl_xor_sync(0xffffffffu, l2, o);
        const float e = __shfl_xor_sync(0xffffffffu, h1, o), f = __shfl_xor_sync(0xffffffffu, l1, o);
        df_add(h2, l2, a, b);
        df_add(h1, l1, e, f);
    }
    pc = __reduce_add_sync(0xffffffffu, pc);
    if (lane == 0) {
        const float t2 = __fadd_rn(h2, l2), t1 = __fadd_rn(h1, l1);
        *nx2 = t2;
        *F = t1 > 0.0f ? __fdiv_rn(__fmul_rn(sqrt_d, t2), t1) : 0.0f;
        *popx = pc;
    }
}

constexpr int ENC_UNROLL = 8;

// Any d: lane l takes dimensions 32w + l, the sign bits of a 32-dimension
// group are one __ballot_sync.
__global__ void rbq1_encode_kernel(const float *__restrict__ X, int64_t n, int d,
                                   const float *__restrict__ m, uint32_t *__restrict__ codes,
                                   float *__restrict__ nx2, float *__restrict__ F,
                                   int32_t *__restrict__ popx) {
    const int lane = threadIdx.x & 31;
    const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int W = (d + 31) >> 5;
    const float sqrt_d = __fsqrt_rn((float)d);
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
        rbq1_row_finish(s2, c2, s1, c1, pc, lane, sqrt_d, nx2 + p, F + p, popx + p);
    }
}

// d % 4 == 0: lane l takes the float4 at dimensions 128t + 4l .. 128t + 4l + 3,
// so its four sign bits are bits 4(l mod 8) .. 4(l mod 8) + 3 of code word
// 4t + l/8; an OR butterfly over each group of 8 lanes assembles the words.
// All of a row's loads (up to ENC_V4 float4 per lane) are issued before use.
constexpr int ENC_V4 = 8;

__global__ void rbq1_encode_v4_kernel(const float4 *__restrict__ X, int64_t n, int d,
                                      const float4 *__restrict__ m, uint32_t *__restrict__ codes,
                                      float *__restrict__ nx2, float *__restrict__ F,
                                      int32_t *__restrict__ popx) {
    const int lane = threadIdx.x & 31;
    const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int W = (d + 31) >> 5, d4 = d >> 2;
    const float sqrt_d = __fsqrt_rn((float)d);
    for (int64_t p = warp; p < n; p += nwarps) {
        const float4 *x = X + p * d4;
        float s2 = 0.0f, c2 = 0.0f, s1 = 0.0f, c1 = 0.0f;
        int pc = 0;
        for (int t0 = 0; 32 * t0 < d4; t0 += ENC_V4) {
            float4 v[ENC_V4];
#pragma unroll
            for (int u = 0; u < ENC_V4; ++u) {
                const int j = 32 * (t0 + u) + lane;
                v[u] = j < d4 ? __ldg(x + j) : make_float4(0.0f, 0.0f, 0.0f, 0.0f);
            }
#pragma unroll
            for (int u = 0; u < ENC_V4; ++u) {
                const int t = t0 + u;
                if (32 * t < d4) {  // warp-uniform
                    const int j = 32 * t + lane;
                    float4 r = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
                    if (j < d4) {
                        const float4 mm = __ldg(m + j);
                        r = make_float4(__fsub_rn(v[u].x, mm.x), __fsub_rn(v[u].y, mm.y),
                                        __fsub_rn(v[u].z, mm.z), __fsub_rn(v[u].w, mm.w));
                    }
                    kahan_add(s2, c2, __fmul_rn(r.x, r.x));
                    kahan_add(s2, c2, __fmul_rn(r.y, r.y));
                    kahan_add(s2, c2, __fmul_rn(r.z, r.z));
                    kahan_add(s2, c2, __fmul_rn(r.w, r.w));
                    kahan_add(s1, c1, fabsf(r.x));
                    kahan_add(s1, c1, fabsf(r.y));
                    kahan_add(s1, c1, fabsf(r.z));
                    kahan_add(s1, c1, fabsf(r.w));
                    uint32_t nib = (r.x > 0.0f ? 1u : 0u) | (r.y > 0.0f ? 2u : 0u) | (r.z > 0.0f ? 4u : 0u) |
                                   (r.w > 0.0f ? 8u : 0u);
                    nib <<= 4 * (lane & 7);
                    nib |= __shfl_xor_sync(0xffffffffu, nib, 1);
                    nib |= __shfl_xor_sync(0xffffffffu, nib, 2);
                    nib |= __shfl_xor_sync(0xffffffffu, nib, 4);
                    const int wi = 4 * t + (lane >> 3);
                    if ((lane & 7) == 0 && wi < W) {
                        codes[p * W + wi] = nib;
                        pc += __popc(nib);
                    }
                }
            }
        }
        rbq1_row_finish(s2, c2, s1, c1, pc, lane, sqrt_d, nx2 + p, F + p, popx + p);
    }
}

// d % 4 == 0 and d <= 1024, NV = ceil(d / 128) float4 per lane, with the next
// row's loads issued before the current row is evaluated, so every warp always
// has a row in flight.  Per float4 the four terms of each sum are added plainly
// and the partial enters the compensated lane sum, so ||r||^2 and ||r||_1 are
// within about 5 * 2^-24 relative and F within about 12 * 2^-24.
template <int NV>
__global__ void __launch_bounds__(256) rbq1_encode_pf_kernel(const float4 *__restrict__ X, int64_t n, int d,
                                                             const float4 *__restrict__ m,
                                                             uint32_t *__restrict__ codes, float *__restrict__ nx2,
                                                             float *__restrict__ F, int32_t *__restrict__ popx) {
    const int lane = threadIdx.x & 31;
    const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int W = (d + 31) >> 5, d4 = d >> 2;
    const float sqrt_d = __fsqrt_rn((float)d);
    const float4 zero = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
    float4 cur[NV];
    auto load_row = [&](int64_t p, float4(&v)[NV]) {
        const float4 *x = X + p * d4;
#pragma unroll
        for (int u = 0; u < NV; ++u) {
            const int j = 32 * u + lane;
            v[u] = j < d4 ? __ldg(x + j) : zero;
        }
    };
    if (warp < n) load_row(warp, cur);
    for (int64_t p = warp; p < n; p += nwarps) {
        float4 nxt[NV];
        if (p + nwarps < n) load_row(p + nwarps, nxt);
        float s2 = 0.0f, c2 = 0.0f, s1 = 0.0f, c1 = 0.0f;
        int pc = 0;
#pragma unroll
        for (int u = 0; u < NV; ++u) {
            const int j = 32 * u + lane;
            float4 r = zero;
            if (j < d4) {
                const float4 mm = __ldg(m + j);
                r = make_float4(__fsub_rn(cur[u].x, mm.x), __fsub_rn(cur[u].y, mm.y), __fsub_rn(cur[u].z, mm.z),
                                __fsub_rn(cur[u].w, mm.w));
            }
            // the float4's four terms summed plainly (non-negative terms: relative
            // error <= 3 * 2^-24), the partial added with compensation
            kahan_add(s2, c2, __fadd_rn(__fadd_rn(__fmul_rn(r.x, r.x), __fmul_rn(r.y, r.y)),
                                        __fadd_rn(__fmul_rn(r.z, r.z), __fmul_rn(r.w, r.w))));
            kahan_add(s1, c1, __fadd_rn(__fadd_rn(fabsf(r.x), fabsf(r.y)), __fadd_rn(fabsf(r.z), fabsf(r.w))));
            uint32_t nib = (r.x > 0.0f ? 1u : 0u) | (r.y > 0.0f ? 2u : 0u) | (r.z > 0.0f ? 4u : 0u) |
                           (r.w > 0.0f ? 8u : 0u);
            nib <<= 4 * (lane & 7);
            nib |= __shfl_xor_sync(0xffffffffu, nib, 1);
            nib |= __shfl_xor_sync(0xffffffffu, nib, 2);
            nib |= __shfl_xor_sync(0xffffffffu, nib, 4);
            const int wi = 4 * u + (lane >> 3);
            if ((lane & 7) == 0 && wi < W) {
                codes[p * W + wi] = nib;
                pc += __popc(nib);
            }
        }
        rbq1_row_finish(s2, c2, s1, c1, pc, lane, sqrt_d, nx2 + p, F + p, popx + p);
#pragma unroll
        for (int u = 0; u < NV; ++u) cur[u] = nxt[u];
    }
}

template <int NV>
static void rbq1_pf_launch(const float *X, int64_t n, int d, const float *m, uint32_t *codes, float *nx2, float *F,
                           int32_t *popx, cudaStream_t st) {
    rbq1_encode_pf_kernel<NV><<<grid_for(n * 32, 256), 256, 0, st>>>(
        reinterpret_cast<const float4 *>(X), n, d, reinterpret_cast<const float4 *>(m), codes, nx2, F, popx);
}

cudaError_t launch_rbq1_encode(const float *X, int64_t n, int d, const float *m, uint32_t *codes,
                               float *nx2, float *F, int32_t *popx, cudaStream_t st) {
    const int threads = 256;
    if (d % 4 == 0 && d <= 1024 && ((uintptr_t)X & 15) == 0 && ((uintptr_t)m & 15) == 0) {
        switch ((d + 127) / 128) {
        case 1: rbq1_pf_launch<1>(X, n, d, m, codes, nx2, F, popx, st); break;
        case 2: rbq1_pf_launch<2>(X, n, d, m, codes, nx2, F, popx, st); break;
        case 3: rbq1_pf_launch<3>(X, n, d, m, codes, nx2, F, popx, st); break;
        case 4: rbq1_pf_launch<4>(X, n, d, m, codes, nx2, F, popx, st); break;
        case 5: rbq1_pf_launch<5>(X, n, d, m, codes, nx2, F, popx, st); break;
        case 6: rbq1_pf_launch<6>(X, n, d, m, codes, nx2, F, popx, st); break;
        case 7: rbq1_pf_launch<7>(X, n, d, m, codes, nx2, F, popx, st); break;
        default: rbq1_pf_launch<8>(X, n, d, m, codes, nx2, F, popx, st); break;
        }
    } else if (d % 4 == 0 && ((uintptr_t)X & 15) == 0 && ((uintptr_t)m & 15) == 0) {
        rbq1_encode_v4_kernel<<<grid_for(n * 32, threads), threads, 0, st>>>(
            reinterpret_cast<const float4 *>(X), n, d, reinterpret_cast<const float4 *>(m), codes, nx2, F,
            popx);
    } else {
        rbq1_encode_kernel<<<grid_for(n * 32, threads), threads, 0, st>>>(X, n, d, m, codes, nx2, F,
                                                                          popx);
    }
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
