// LVQ4 (Section 3.1 "LVQ4"): every vector gets its own bias b = min and scale
// s = (max - b) / 15 and 4-bit codes; distances follow Eq. final:lvq from the
// integer code dot product P = <xbar, ybar> and per-vector terms, and the
// centroid update is the fused decode-average of the members' codes.
//
//   encode   one warp per vector: min / max, s, codes packed 8 nibbles per
//            uint32 word through 8-lane OR butterflies, N and A in fp64 from
//            the exact integer sums S = sum code, Q = sum code^2
//   cprep    the same encoding of every centroid once per assignment, as
//            e4m3 bytes for the tensor-core kernel (0..15 are exact in e4m3)
//            or as nibble words for the __dp4a kernel (d > 1024)
//   update   fixed-point weights Sq = round(s 2^e), Bq = round(b 2^e) in the
//            cluster-sorted order; the sums T = sum Sq xbar, U = sum Bq are
//            exact int64 (streamed in k_ringsum.cu, or the chunk kernel here),
//            then c = (T + U) f in fp64 with one factor f = 2^-e / count per
//            cluster
//
// Every float step that decides a code or a key is an explicit IEEE operation
// (no contraction), in the order the oracle takes it.
#include "skm_internal.cuh"

namespace skm {
namespace {

constexpr unsigned FULL = 0xffffffffu;

int grid_warps_rows(int64_t rows) {
    int64_t b = (rows * 32 + 255) / 256;
    const int64_t cap = 152LL * 16;
    return (int)(b < 1 ? 1 : (b > cap ? cap : b));
}

struct Lvq4Vec {
    float lo, s;
    int32_t S, Q;
};

// One warp encodes the vector v[0..d): every lane calls emit(base, lane, code)
// for each 32-dimension chunk (code 0 past d), so emit may use warp shuffles.
template <typename Emit>
__device__ __forceinline__ Lvq4Vec lvq4_encode_warp(const float *__restrict__ v, int d, int lane, Emit emit) {
    float lo = INFINITY, hi = -INFINITY;
    for (int i = lane; i < d; i += 32) {
        const float x = v[i];
        lo = fminf(lo, x);
        hi = fmaxf(hi, x);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        lo = fminf(lo, __shfl_xor_sync(FULL, lo, o));
        hi = fmaxf(hi, __shfl_xor_sync(FULL, hi, o));
    }
    float s = __fdiv_rn(__fsub_rn(hi, lo), 15.0f);
    if (!(s > 0.0f)) s = 1.0f;
    int32_t S = 0, Q = 0;
    for (int base = 0; base < d; base += 32) {
        const int i = base + lane;
        uint32_t c = 0;
        if (i < d) {
            float q = rintf(__fdiv_rn(__fsub_rn(v[i], lo), s));
            q = (q >= 0.0f) ? q : 0.0f;
            q = fminf(q, 15.0f);
            c = (uint32_t)q;
        }
        S += (int32_t)c;
        Q += (int32_t)(c * c);
        emit(base, lane, c);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        S += __shfl_xor_sync(FULL, S, o);
        Q += __shfl_xor_sync(FULL, Q, o);
    }
    return Lvq4Vec{lo, s, S, Q};
}

// N = s*s*Q + 2*b*s*S + d*b*b and A = s*S + d*b, fp64 left to right.
__device__ __forceinline__ double lvq4_norm(const Lvq4Vec &r, int d) {
    const double sd = (double)r.s, bd = (double)r.lo, dd = (double)d;
    const double t1 = __dmul_rn(__dmul_rn(sd, sd), (double)r.Q);
    const double t2 = __dmul_rn(__dmul_rn(__dmul_rn(2.0, bd), sd), (double)r.S);
    const double t3 = __dmul_rn(__dmul_rn(dd, bd), bd);
    return __dadd_rn(__dadd_rn(t1, t2), t3);
}
__device__ __forceinline__ double lvq4_sum(const Lvq4Vec &r, int d) {
    return __dadd_rn(__dmul_rn((double)r.s, (double)r.S), __dmul_rn((double)d, (double)r.lo));
}

// 8 lanes' codes -> one nibble word held by lane 8g of each group g
__device__ __forceinline__ uint32_t pack_nibbles(uint32_t c, int lane) {
    uint32_t v = c << (4 * (lane & 7));
    v |= __shfl_xor_sync(FULL, v, 1);
    v |= __shfl_xor_sync(FULL, v, 2);
    v |= __shfl_xor_sync(FULL, v, 4);
    return v;
}

// N and A (R25) take fp64 arithmetic, which GB300 issues at a small fraction
// of its fp32 rate, and a warp instruction costs the same with one lane active
// as with 32: a warp therefore parks the (s, b, S, Q) of 32 consecutive rows of
// its loop in lanes 0..31 and evaluates the 32 fp64 tails together.
struct FacBatch {
    Lvq4Vec r{0.0f, 0.0f, 0, 0};
    int64_t row = -1;
    int cnt = 0;
    __device__ __forceinline__ void put(const Lvq4Vec &v, int64_t p, int lane, float4 *fac, int d) {
        if (lane == cnt) {
            r = v;
            row = p;
        }
        if (++cnt == 32) flush(fac, d);
    }
    __device__ __forceinline__ void flush(float4 *fac, int d) {
        if (row >= 0)
            fac[row] = make_float4(r.s, r.lo, __double2float_rn(lvq4_norm(r, d)), __double2float_rn(lvq4_sum(r, d)));
        row = -1;
        cnt = 0;
    }
};

__global__ void lvq4_encode_kernel(const float *__restrict__ X, int64_t n, int d, uint32_t *__restrict__ codes,
                                   float4 *__restrict__ fac) {
    const int lane = threadIdx.x & 31;
    const int64_t w0 = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int W = lvq4_words(d);
    FacBatch fb;
    for (int64_t p = w0; p < n; p += nw) {
        uint32_t *cw = codes + p * W;
        const Lvq4Vec r = lvq4_encode_warp(X + p * d, d, lane, [&](int base, int ln, uint32_t c) {
            const uint32_t v = pack_nibbles(c, ln);
            const int wi = (base >> 3) + (ln >> 3);
            if ((ln & 7) == 0 && wi < W) cw[wi] = v;
        });
        fb.put(r, p, lane, fac, d);
    }
    fb.flush(fac, d);
}

// d % 4 == 0 and d <= 1024: the row stays in registers (lane l holds the
// float4 at dimensions 128u + 4l .. + 3 for u < NV = ceil(d / 128), the next
// row's loads in flight while this one is encoded), so the points are read
// once; the two lanes of a pair assemble one nibble word (8 dimensions), the
// even lane stores it.  Same code arithmetic as lvq4_encode_warp.

// clip(rint(fl((x - lo) / s)), 0, 15) with one multiplication in place of the
// division: with rs = fl(1/s), q' = fl(a rs) (a = fl(x - lo)) is within
// (2^-23 + 2^-24 + 2^-48) |a/s| of the correctly rounded quotient q, i.e. within
// 2^-18.5 since a/s <= 15 / (1 - 2^-24) here (a <= fl(hi - lo), s rounded from
// fl(hi - lo) / 15).  When q' is more than
// 2^-17 away from every half-integer, q and q' round to the same integer;
// otherwise (and for inf / NaN) the quotient is taken by the IEEE division.
// The bound needs a normal rs: callers pass NaN instead of a subnormal one.
// Four codes at once: one combined test sends the float4 to the divisions
// when any of its quotients is near a half-integer or not finite (fmaxf drops
// NaN, hence the separate finiteness test).
__device__ __forceinline__ void lvq4_code4(const float4 &x, float lo, float s, float rs, uint32_t &c0, uint32_t &c1,
                                           uint32_t &c2, uint32_t &c3) {
    const float ax = __fsub_rn(x.x, lo), ay = __fsub_rn(x.y, lo), az = __fsub_rn(x.z, lo), aw = __fsub_rn(x.w, lo);
    const float qx = __fmul_rn(ax, rs), qy = __fmul_rn(ay, rs), qz = __fmul_rn(az, rs), qw = __fmul_rn(aw, rs);
    float tx = rintf(qx), ty = rintf(qy), tz = rintf(qz), tw = rintf(qw);
    constexpr float lim = 0.5f - 0x1p-17f;
    if (!(fmaxf(fmaxf(fabsf(__fsub_rn(qx, tx)), fabsf(__fsub_rn(qy, ty))),
                fmaxf(fabsf(__fsub_rn(qz, tz)), fabsf(__fsub_rn(qw, tw)))) < lim) ||
        !(fabsf(qx) + fabsf(qy) + fabsf(qz) + fabsf(qw) < INFINITY)) {
        if (!(fabsf(__fsub_rn(qx, tx)) < lim)) tx = rintf(__fdiv_rn(ax, s));
        if (!(fabsf(__fsub_rn(qy, ty)) < lim)) ty = rintf(__fdiv_rn(ay, s));
        if (!(fabsf(__fsub_rn(qz, tz)) < lim)) tz = rintf(__fdiv_rn(az, s));
        if (!(fabsf(__fsub_rn(qw, tw)) < lim)) tw = rintf(__fdiv_rn(aw, s));
    }
    auto clip = [](float t) { return (uint32_t)fminf(t >= 0.0f ? t : 0.0f, 15.0f); };
    c0 = clip(tx);
    c1 = clip(ty);
    c2 = clip(tz);
    c3 = clip(tw);
}


template <int NV>
__global__ void __launch_bounds__(256, 2) lvq4_encode_v4_kernel(const float4 *__restrict__ X, int64_t n, int d,
                                                                uint32_t *__restrict__ codes, float4 *__restrict__ fac) {
    const int lane = threadIdx.x & 31;
    const int64_t w0 = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int W = lvq4_words(d), d4 = d >> 2;
    auto load_row = [&](int64_t p, float4(&v)[NV]) {
        const float4 *x = X + p * d4;
#pragma unroll
        for (int u = 0; u < NV; ++u) {
            const int j = 32 * u + lane;
            if (j < d4) v[u] = __ldg(x + j);
        }
    };
    FacBatch fb;
    float4 v[NV];
    if (w0 < n) load_row(w0, v);
    for (int64_t p = w0; p < n; p += nw) {
        float4 nxt[NV];
        if (p + nw < n) load_row(p + nw, nxt);  // the next row in flight while this one is encoded
        float lo = INFINITY, hi = -INFINITY;
#pragma unroll
        for (int u = 0; u < NV; ++u) {
            if (32 * u + lane < d4) {
                lo = fminf(lo, fminf(fminf(v[u].x, v[u].y), fminf(v[u].z, v[u].w)));
                hi = fmaxf(hi, fmaxf(fmaxf(v[u].x, v[u].y), fmaxf(v[u].z, v[u].w)));
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            lo = fminf(lo, __shfl_xor_sync(FULL, lo, o));
            hi = fmaxf(hi, __shfl_xor_sync(FULL, hi, o));
        }
        float s = __fdiv_rn(__fsub_rn(hi, lo), 15.0f);
        if (!(s > 0.0f)) s = 1.0f;
        float rs = __frcp_rn(s);
        if (!(fabsf(rs) >= 0x1p-126f)) rs = __int_as_float(0x7fffffff);  // subnormal: divide every code
        int32_t S = 0, Q = 0;
        uint32_t *cw = codes + p * W;
#pragma unroll
        for (int u = 0; u < NV; ++u) {
            const int j = 32 * u + lane;
            uint32_t h = 0;
            if (j < d4) {
                uint32_t c0, c1, c2, c3;
                lvq4_code4(v[u], lo, s, rs, c0, c1, c2, c3);
                S += (int32_t)(c0 + c1 + c2 + c3);
                Q += (int32_t)(c0 * c0 + c1 * c1 + c2 * c2 + c3 * c3);
                h = (c0 | (c1 << 4) | (c2 << 8) | (c3 << 12)) << (16 * (lane & 1));
            }
            h |= __shfl_xor_sync(FULL, h, 1);
            const int wi = j >> 1;
            if ((lane & 1) == 0 && wi < W) cw[wi] = h;
        }
        S = __reduce_add_sync(FULL, S);
        Q = __reduce_add_sync(FULL, Q);
        fb.put(Lvq4Vec{lo, s, S, Q}, p, lane, fac, d);
#pragma unroll
        for (int u = 0; u < NV; ++u) v[u] = nxt[u];
    }
    fb.flush(fac, d);
}

// M = max over points of max(s, |b|) (positive floats order like their bits),
// then e = 31 - ceil(log2 M), 0 when M == 0.
__global__ void lvq4_maxbits_kernel(const float4 *__restrict__ fac, int64_t n, unsigned int *__restrict__ maxbits) {
    unsigned int mx = 0;
    for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < n; t += (int64_t)gridDim.x * blockDim.x) {
        const float4 f = fac[t];
        const float m = fmaxf(f.x, fabsf(f.y));
        if (m > 0.0f) mx = max(mx, __float_as_uint(m));
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = max(mx, __shfl_xor_sync(FULL, mx, o));
    if ((threadIdx.x & 31) == 0 && mx) atomicMax(maxbits, mx);
}

__global__ void lvq4_exponent_kernel(const unsigned int *__restrict__ maxbits, int *__restrict__ e) {
    const float mx = __uint_as_float(*maxbits);
    if (!(mx > 0.0f)) {
        *e = 0;
        return;
    }
    int ex;
    const double fr = frexp((double)mx, &ex);
    const int c = (fr == 0.5) ? ex - 1 : ex;  // ceil(log2 mx)
    *e = 31 - c;
}

// One warp per centroid; info[j] = (s, b, N, G = s * sum ybar).
__global__ void lvq4_cprep_kernel(const float *__restrict__ C, int k, int d, uint8_t *__restrict__ yq, int dq,
                                  uint32_t *__restrict__ yw, float4 *__restrict__ info) {
    const int lane = threadIdx.x & 31;
    const int j = (int)((blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5);
    if (j >= k) return;  // warp-uniform
    const int W = lvq4_words(d);
    const Lvq4Vec r = lvq4_encode_warp(C + (int64_t)j * d, d, lane, [&](int base, int ln, uint32_t c) {
        const int i = base + ln;
        if (yq && i < d) yq[(int64_t)j * dq + i] = e4m3_of_code(c);
        if (yw) {
            const uint32_t v = pack_nibbles(c, ln);
            const int wi = (base >> 3) + (ln >> 3);
            if ((ln & 7) == 0 && wi < W) yw[(int64_t)j * W + wi] = v;
        }
    });
    if (lane == 0)
        info[j] = make_float4(r.s, r.lo, __double2float_rn(lvq4_norm(r, d)),
                              __double2float_rn(__dmul_rn((double)r.s, (double)r.S)));
}

// nibble words -> e4m3 bytes (8 per word, one 8-byte store)
__global__ void lvq4_expand_kernel(const uint32_t *__restrict__ codes, int64_t n, int d, uint8_t *__restrict__ xs,
                                   int dq) {
    const int W = lvq4_words(d);
    const int64_t total = n * W;
    for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < total; t += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = t / W;
        const int w = (int)(t - r * W);
        const uint32_t v = codes[t];
        uint32_t lo = 0, hi = 0;
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            lo |= (uint32_t)e4m3_of_code((v >> (4 * u)) & 15u) << (8 * u);
            hi |= (uint32_t)e4m3_of_code((v >> (16 + 4 * u)) & 15u) << (8 * u);
        }
        *reinterpret_cast<uint2 *>(xs + r * dq + 8 * w) = make_uint2(lo, hi);
    }
}

// Column-pair records of the tensor epilogue; columns past k get N = +inf.
__global__ void lvq4_pack_pairs_kernel(const float4 *__restrict__ info, int k, int kp, float4 *__restrict__ bg,
                                      float4 *__restrict__ sn) {
    const int pp = blockIdx.x * blockDim.x + threadIdx.x;
    if (2 * pp >= kp) return;
    float b[2], g[2], s[2], nn[2];
#pragma unroll
    for (int o = 0; o < 2; ++o) {
        const int j = 2 * pp + o;
        if (j < k) {
            const float4 in = info[j];
            s[o] = in.x;
            b[o] = in.y;
            nn[o] = in.z;
            g[o] = in.w;
        } else {
            s[o] = b[o] = g[o] = 0.0f;
            nn[o] = INFINITY;
        }
    }
    bg[pp] = make_float4(b[0], b[1], g[0], g[1]);
    sn[pp] = make_float4(s[0], s[1], nn[0], nn[1]);
}

// d > 1024: one thread per point, tiles of SA_KT centroids in shared memory as
// even / odd nibble bytes, P by __dp4a; the key of Eq. final:lvq in the same
// fp32 order as the tensor epilogue.
constexpr int SA_KT = 16;
__global__ void __launch_bounds__(256) assign_lvq4_simt_kernel(const uint32_t *__restrict__ codes,
                                                               const float4 *__restrict__ fac, int64_t n, int d,
                                                               const uint32_t *__restrict__ yw,
                                                               const float4 *__restrict__ info, int k,
                                                               int32_t *__restrict__ assign, float *__restrict__ dist) {
    extern __shared__ uint32_t sy[];  // [SA_KT][2][W]
    const int W = lvq4_words(d);
    const int64_t row = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
    const bool valid = row < n;
    const float4 f = valid ? fac[row] : make_float4(0.f, 0.f, 0.f, 0.f);
    const float sx2 = __fmul_rn(-2.0f, f.x), bx2 = __fmul_rn(-2.0f, f.y), ax2 = __fmul_rn(-2.0f, f.w);
    const uint32_t *xr = codes + (valid ? row : 0) * W;
    float best = INFINITY;
    int32_t besti = 0;
    for (int j0 = 0; j0 < k; j0 += SA_KT) {
        __syncthreads();
        for (int t = threadIdx.x; t < SA_KT * W; t += blockDim.x) {
            const int c = t / W, w = t - c * W;
            const uint32_t v = (j0 + c < k) ? yw[(int64_t)(j0 + c) * W + w] : 0u;
            sy[(2 * c) * W + w] = v & 0x0F0F0F0Fu;
            sy[(2 * c + 1) * W + w] = (v >> 4) & 0x0F0F0F0Fu;
        }
        __syncthreads();
        if (!valid) continue;
        uint32_t P[SA_KT];
#pragma unroll
        for (int c = 0; c < SA_KT; ++c) P[c] = 0;
        for (int w = 0; w < W; ++w) {
            const uint32_t xw = xr[w];
            const uint32_t xe = xw & 0x0F0F0F0Fu, xo = (xw >> 4) & 0x0F0F0F0Fu;
#pragma unroll
            for (int c = 0; c < SA_KT; ++c) {
                P[c] = __dp4a(xe, sy[(2 * c) * W + w], P[c]);
                P[c] = __dp4a(xo, sy[(2 * c + 1) * W + w], P[c]);
            }
        }
#pragma unroll
        for (int c = 0; c < SA_KT; ++c) {
            const int j = j0 + c;
            if (j < k) {
                const float4 in = info[j];
                float key = __fmaf_rn(in.y, ax2, in.z);
                key = __fmaf_rn(in.w, bx2, key);
                const float t = __fmul_rn(in.x, __uint2float_rn(P[c]));
                key = __fmaf_rn(sx2, t, key);
                if (key < best) {
                    best = key;
                    besti = j;
                }
            }
        }
    }
    if (valid) {
        assign[row] = besti;
        if (dist) dist[row] = __fadd_rn(f.z, best);
    }
}

// Fixed-point weights in the cluster-sorted order (position q: member perm[q]).
__global__ void lvq4_q_kernel(const float4 *__restrict__ fac, const int32_t *__restrict__ perm,
                              const int64_t *__restrict__ offsets, int k, int e, uint32_t *__restrict__ sq,
                              int64_t *__restrict__ bq) {
    const int64_t nval = offsets[k];
    for (int64_t q = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; q < nval; q += (int64_t)gridDim.x * blockDim.x) {
        const float4 f = fac[perm[q]];
        sq[q] = (uint32_t)fixed_rint(f.x, e);
        bq[q] = fixed_rint(f.y, e);
    }
}

// Rows that do not suit the streamed sums: one warp per run of 128 sorted
// positions, lane = nibble word (32 words per pass), 8 int64 accumulators per
// lane, flushed with atomics when the cluster changes.  T[c][d] += Bq.
__global__ void chunk_sum_lvq4_kernel(const uint32_t *__restrict__ codes, const uint32_t *__restrict__ sq,
                                      const int64_t *__restrict__ bq, int d, const int32_t *__restrict__ perm,
                                      const int32_t *__restrict__ scl, const int64_t *__restrict__ offsets, int k,
                                      unsigned long long *__restrict__ T) {
    const int lane = threadIdx.x & 31;
    const int64_t gw = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    const int64_t nval = offsets[k];
    const int64_t q0 = gw * 128;
    if (q0 >= nval) return;
    const int cnt = (int)((nval - q0) < 128 ? (nval - q0) : 128);
    const int W = lvq4_words(d);
    for (int w0 = 0; w0 < W; w0 += 32) {
        const int w = w0 + lane;
        unsigned long long acc[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[j] = 0ull;
        int64_t us = 0;
        int cur = scl[q0];
        auto flush = [&](int c) {
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int col = 8 * w + j;
                if (w < W && col < d && acc[j]) atomicAdd(T + (int64_t)c * (d + 1) + col, acc[j]);
                acc[j] = 0ull;
            }
            if (w0 == 0 && lane == 0 && us) atomicAdd(T + (int64_t)c * (d + 1) + d, (unsigned long long)us);
            us = 0;
        };
        for (int i = 0; i < cnt; ++i) {
            const int64_t q = q0 + i;
            const int c = scl[q];
            if (c != cur) {
                flush(cur);
                cur = c;
            }
            const uint32_t s = sq[q];
            if (w0 == 0) us += bq[q];
            if (w < W) {
                const uint32_t v = codes[(int64_t)perm[q] * W + w];
#pragma unroll
                for (int j = 0; j < 8; ++j) acc[j] += (unsigned long long)s * ((v >> (4 * j)) & 15u);
            }
        }
        flush(cur);
    }
}

// c_i = (T_i + U) f, f = 2^-e / count formed once per cluster (one block each).
__global__ void finalize_lvq4_kernel(const int64_t *__restrict__ partial, const int64_t *__restrict__ counts, int k,
                                     int d, int e, float *__restrict__ C) {
    __shared__ double fs;
    const int j = blockIdx.x;
    const int64_t c = counts[j];
    if (c <= 0) return;  // block-uniform
    if (threadIdx.x == 0) fs = __ddiv_rn(ldexp(1.0, -e), (double)c);
    __syncthreads();
    const double f = fs;
    const int64_t *T = partial + (int64_t)j * (d + 1);
    const int64_t U = T[d];
    for (int i = threadIdx.x; i < d; i += blockDim.x)
        C[(int64_t)j * d + i] = __double2float_rn(__dmul_rn(__ll2double_rn(T[i] + U), f));
}

// Forgy initial centroids: the decode-average of one member each.
__global__ void lvq4_decode_rows_kernel(const uint32_t *__restrict__ codes, const float4 *__restrict__ fac, int64_t n,
                                        int d, int e, const int64_t *__restrict__ idx, int k, float *__restrict__ out,
                                        int *__restrict__ status) {
    const int j = blockIdx.x;
    if (j >= k) return;
    const int64_t p = idx[j];
    if (p < 0 || p >= n) {
        if (threadIdx.x == 0) atomicExch(status, 1);
        return;
    }
    const int W = lvq4_words(d);
    const double pow2 = ldexp(1.0, e);
    const float4 f = fac[p];
    const int64_t sq = __double2ll_rn(__dmul_rn((double)f.x, pow2));
    const int64_t bq = __double2ll_rn(__dmul_rn((double)f.y, pow2));
    const double g = ldexp(1.0, -e);  // the update's factor for a cluster of one member
    for (int i = threadIdx.x; i < d; i += blockDim.x) {
        const int64_t x = (codes[p * W + (i >> 3)] >> (4 * (i & 7))) & 15u;
        out[(int64_t)j * d + i] = __double2float_rn(__dmul_rn(__ll2double_rn(sq * x + bq), g));
    }
}

}  // namespace

cudaError_t launch_lvq4_encode(const float *X, int64_t n, int d, uint32_t *codes, float4 *fac, cudaStream_t st) {
    const float4 *X4 = reinterpret_cast<const float4 *>(X);
    const int g = grid_warps_rows(n);
    if (d % 4 == 0 && d <= 1024 && ((uintptr_t)X & 15) == 0) {
        switch ((d + 127) / 128) {
        case 1: lvq4_encode_v4_kernel<1><<<g, 256, 0, st>>>(X4, n, d, codes, fac); break;
        case 2: lvq4_encode_v4_kernel<2><<<g, 256, 0, st>>>(X4, n, d, codes, fac); break;
        case 3: lvq4_encode_v4_kernel<3><<<g, 256, 0, st>>>(X4, n, d, codes, fac); break;
        case 4: lvq4_encode_v4_kernel<4><<<g, 256, 0, st>>>(X4, n, d, codes, fac); break;
        case 5: lvq4_encode_v4_kernel<5><<<g, 256, 0, st>>>(X4, n, d, codes, fac); break;
        case 6: lvq4_encode_v4_kernel<6><<<g, 256, 0, st>>>(X4, n, d, codes, fac); break;
        case 7: lvq4_encode_v4_kernel<7><<<g, 256, 0, st>>>(X4, n, d, codes, fac); break;
        default: lvq4_encode_v4_kernel<8><<<g, 256, 0, st>>>(X4, n, d, codes, fac); break;
        }
    } else {
        lvq4_encode_kernel<<<g, 256, 0, st>>>(X, n, d, codes, fac);
    }
    return launched();
}

cudaError_t launch_lvq4_exponent(const float4 *fac, int64_t n, unsigned int *maxbits, int *e_dev, cudaStream_t st) {
    cudaError_t err = cudaMemsetAsync(maxbits, 0, sizeof(unsigned int), st);
    if (err != cudaSuccess) return err;
    int64_t blocks = (n + 255) / 256;
    if (blocks > 152 * 8) blocks = 152 * 8;
    lvq4_maxbits_kernel<<<(unsigned)(blocks < 1 ? 1 : blocks), 256, 0, st>>>(fac, n, maxbits);
    lvq4_exponent_kernel<<<1, 1, 0, st>>>(maxbits, e_dev);
    return launched(2);
}

cudaError_t launch_lvq4_cprep(const float *C, int k, int d, uint8_t *yq, int dq, uint32_t *yw, float4 *info,
                              cudaStream_t st) {
    lvq4_cprep_kernel<<<(k + 7) / 8, 256, 0, st>>>(C, k, d, yq, dq, yw, info);
    return launched();
}

cudaError_t launch_lvq4_expand(const uint32_t *codes, int64_t n, int d, uint8_t *xs, int dq, cudaStream_t st) {
    int64_t blocks = (n * lvq4_words(d) + 255) / 256;
    if (blocks > 152 * 8) blocks = 152 * 8;
    lvq4_expand_kernel<<<(unsigned)(blocks < 1 ? 1 : blocks), 256, 0, st>>>(codes, n, d, xs, dq);
    return launched();
}

cudaError_t launch_lvq4_pack_pairs(const float4 *info, int k, int kp, float4 *bg, float4 *sn, cudaStream_t st) {
    lvq4_pack_pairs_kernel<<<(kp / 2 + 255) / 256, 256, 0, st>>>(info, k, kp, bg, sn);
    return launched();
}

cudaError_t launch_assign_lvq4_simt(const uint32_t *codes, const float4 *fac, int64_t n, int d, const uint32_t *yw,
                                    const float4 *info, int k, int32_t *assign, float *dist, cudaStream_t st) {
    const size_t smem = (size_t)SA_KT * 2 * lvq4_words(d) * sizeof(uint32_t);
    if (smem > 48 * 1024) {
        const cudaError_t e =
            cudaFuncSetAttribute(assign_lvq4_simt_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
    }
    assign_lvq4_simt_kernel<<<(unsigned)((n + 255) / 256), 256, smem, st>>>(codes, fac, n, d, yw, info, k, assign,
                                                                            dist);
    return launched();
}

cudaError_t launch_lvq4_q(const float4 *fac, const int32_t *perm, const int64_t *offsets, int k, int64_t n, int e,
                          uint32_t *sq, int64_t *bq, cudaStream_t st) {
    int64_t blocks = (n + 255) / 256;
    if (blocks > 152 * 8) blocks = 152 * 8;
    lvq4_q_kernel<<<(unsigned)(blocks < 1 ? 1 : blocks), 256, 0, st>>>(fac, perm, offsets, k, e, sq, bq);
    return launched();
}

cudaError_t launch_chunk_sum_lvq4(const uint32_t *codes, const uint32_t *sq, const int64_t *bq, int64_t n, int d,
                                  const int32_t *perm, const int32_t *scl, const int64_t *offsets, int k, int64_t *T,
                                  cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    (void)scl;
    const int64_t warps = (n + 127) / 128;
    chunk_sum_lvq4_kernel<<<(unsigned)((warps * 32 + 255) / 256), 256, 0, st>>>(
        codes, sq, bq, d, perm, scl, offsets, k, reinterpret_cast<unsigned long long *>(T));
    return launched();
}

cudaError_t launch_finalize_lvq4(const int64_t *partial, const int64_t *counts, int k, int d, int e, float *C_inout,
                                 cudaStream_t st) {
    finalize_lvq4_kernel<<<k, 256, 0, st>>>(partial, counts, k, d, e, C_inout);
    return launched();
}

cudaError_t launch_lvq4_decode_rows(const uint32_t *codes, const float4 *fac, int64_t n, int d, int e,
                                    const int64_t *idx, int k, float *out, int *status, cudaStream_t st) {
    lvq4_decode_rows_kernel<<<k, 256, 0, st>>>(codes, fac, n, d, e, idx, k, out, status);
    return launched();
}

}  // namespace skm
