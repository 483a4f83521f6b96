// Internal declarations shared by the libskm translation units (not part of
// the ABI).  Kernels are launched through the `launch_*` functions declared
// here; every launcher returns cudaGetLastError() of its launch.
#pragma once

#include <math.h>
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>
#include <stddef.h>

#include "../../include/skm.h"

namespace skm {

// ---- error reporting (thread-local message, see skm_abi.cu) --------------
int set_error(int code, const char *fmt, ...);

#define SKM_CUDA_TRY(expr)                                                         \
    do {                                                                           \
        cudaError_t e_ = (expr);                                                   \
        if (e_ != cudaSuccess)                                                     \
            return ::skm::set_error(SKM_ERR_CUDA, "%s failed: %s (%s:%d)", #expr,  \
                                    cudaGetErrorString(e_), __FILE__, __LINE__);   \
    } while (0)

#define SKM_TRY(expr)                    \
    do {                                 \
        int s_ = (expr);                 \
        if (s_ != SKM_OK) return s_;     \
    } while (0)

// Counts `count` kernel launches (host-side, process-wide) and returns
// cudaGetLastError(); every launcher returns through it.
cudaError_t launched(int count = 1);
// True (and one armed occurrence used up) when an SKM_FAULT_* of this kind
// is armed (skm_inject_fault or the SKM_FAULT environment variable).
bool fault_take(int kind);
// the kernel timer's events around a tensor-core kernel launch (which = 0
// before, 1 after; nothing unless skm_kernel_timer enabled it)
void tc_timer_mark(cudaStream_t st, int which);

// ---- workspace carving ------------------------------------------------------
// Sub-buffers are carved from the caller's workspace at 256-byte boundaries.
// With base == nullptr the carver only measures (used by skm_workspace_size).
struct Carver {
    char *base;
    size_t off = 0;
    size_t cap;
    Carver(void *b, size_t c) : base(static_cast<char *>(b)), cap(c) {}
    template <typename T>
    T *take(size_t count) {
        off = (off + 255) & ~size_t(255);
        T *p = base ? reinterpret_cast<T *>(base + off) : nullptr;
        off += count * sizeof(T);
        return p;
    }
    bool fits() const { return off <= cap; }
};

inline int words_of(int d) { return (d + 31) / 32; }
inline int64_t cdiv(int64_t a, int64_t b) { return (a + b - 1) / b; }

// rint(v 2^e) as an integer, rounding half to even, for a finite v and
// |v 2^e| < 2^62: v's 24-bit significand is shifted by its exponent plus e and
// the dropped bits are rounded in integer arithmetic, so the result equals the
// exact fp64 product rounded to an integer, without fp64 instructions (which
// GB300 issues at a small fraction of the integer rate).
__device__ __forceinline__ int64_t fixed_rint(float v, int e) {
    const uint32_t b = __float_as_uint(v);
    const int E = (int)((b >> 23) & 0xffu);
    uint64_t m = b & 0x7fffffu;
    int sh;
    if (E) {
        m |= 0x800000u;
        sh = E - 150 + e;
    } else {
        sh = -149 + e;
    }
    uint64_t q;
    if (sh >= 0) {
        q = m << sh;
    } else if (-sh > 25) {  // m < 2^24: below one half
        q = 0;
    } else {
        const int s = -sh;
        q = m >> s;
        const uint64_t r = m & ((1ull << s) - 1ull), half = 1ull << (s - 1);
        if (r > half || (r == half && (q & 1ull))) ++q;
    }
    return (b >> 31) ? -(int64_t)q : (int64_t)q;
}

// acc += f when (word & mask) != 0: one bit test and one predicated 32-bit add
// (the 1-bit decode-average sums of a run of rows).
__device__ __forceinline__ void add_if_bit(uint32_t &acc, uint32_t word, uint32_t mask, uint32_t f) {
    asm("{\n\t.reg .pred p;\n\t"
        "and.b32 %1, %1, %2;\n\t"
        "setp.ne.u32 p, %1, 0;\n\t"
        "@p add.u32 %0, %0, %3;\n\t}"
        : "+r"(acc), "+r"(word)
        : "r"(mask), "r"(f));
}

// (lo, hi) += (flo, fhi) when (word & mask) != 0, as two predicated 32-bit
// adds (no branch, no carry); used by the 1-bit decode-average sums, which
// split each fixed-point weight as hi 2^20 + lo.
__device__ __forceinline__ void add_if_bit2(uint32_t &lo, uint32_t &hi, uint32_t word, uint32_t mask,
                                            uint32_t flo, uint32_t fhi) {
    asm("{\n\t.reg .pred p;\n\t"
        "and.b32 %2, %2, %3;\n\t"
        "setp.ne.u32 p, %2, 0;\n\t"
        "@p add.u32 %0, %0, %4;\n\t"
        "@p add.u32 %1, %1, %5;\n\t}"
        : "+r"(lo), "+r"(hi), "+r"(word)
        : "r"(mask), "r"(flo), "r"(fhi));
}

// e4m3 encodings of the integers 0..15 (sign 0, exponent bias 7, 3 mantissa
// bits): 0 -> 0x00, 1 -> 0x38, 2 -> 0x40, 3 -> 0x44, 4 -> 0x48, ... 15 -> 0x57.
__device__ __forceinline__ uint8_t e4m3_of_code(uint32_t y) {
    if (y == 0) return 0;
    const int e = 31 - __clz(y);                // floor(log2 y), 0..3
    const uint32_t mant = (y << (3 - e)) & 7u;  // 3 bits below the leading one
    return (uint8_t)(((uint32_t)(e + 7) << 3) | mant);
}

// Per-centroid terms of the RBQ1 estimator (Eq. final:rabitq), one record
// per centroid: SQ4 bias and scale multiplied by fl(1/sqrt(d)) (bd = b isd,
// sd = s isd), the sum of codes, ||c - m||^2.
struct Rbq1CInfo {
    float bd;
    float sd;
    int32_t sumy;
    float ny2;
};

// SuperKMeans with RabitQ codes: per-centroid terms of the three dimension
// segments (SQ4 bias and scale times fl(1/sqrt(d_t)), ||rho_t||^2, code sums)
struct Rbq1SegInfo {
    float bd[3];
    float sd[3];
    float ny2[3];
    int32_t sumy[3];
};
constexpr double SEG_EPS0 = 2.1;  // ADSampling's significance parameter
// segments [0, d1), [d1, d2), [d2, d): d1 = d/8 in whole 32-dimension words, d2 = 2 d1
void rbq1_seg_bounds(int d, int *d1, int *d2);
// checkpoint factors g_t = fl32((e_t / d) (1 + eps0 / sqrt(e_t))^2)
void rbq1_seg_factors(int d, int d1, int d2, float *g);
cudaError_t launch_rbq1_seg_encode(const float *X, int64_t n, int d, const float *m, float *nx2s, float *Fs,
                                   int32_t *popxs, cudaStream_t st);
cudaError_t launch_rbq1_seg_cprep(const float *C, int k, int d, const float *m, uint4 *planes, Rbq1SegInfo *info,
                                  cudaStream_t st);
cudaError_t launch_assign_rbq1_seg(const uint32_t *codes, const float *nx2s, const float *Fs, const int32_t *popxs,
                                   int64_t n, int d, const uint4 *planes, const Rbq1SegInfo *info, int k,
                                   const int32_t *prev, int32_t *assign, float *dist, unsigned long long *counters,
                                   cudaStream_t st);

// ---- kernels (launchers) ------------------------------------------------
// quantize / encode
cudaError_t launch_colminmax_partial(const float *X, int64_t n, int d, float *pmin, float *pmax,
                                     int nblk, cudaStream_t st);
// levels L = 2^bits - 1 (255 for SQ8, 15 for SQ4)
cudaError_t launch_sq8_params(const float *pmin, const float *pmax, int nblk, int d, int levels,
                              float *b, float *s, cudaStream_t st);
cudaError_t launch_sq8_encode(const float *X, int64_t n, int d, const float *b, const float *s,
                              int levels, uint8_t *codes, cudaStream_t st);
cudaError_t launch_sq8_decode(const uint8_t *codes, int64_t n, int d, const float *b,
                              const float *s, float *Y, cudaStream_t st);
cudaError_t launch_colsum_partial(const float *X, int64_t n, int d, double *psum, int nblk,
                                  cudaStream_t st);
// the RabitQ mean in exact fixed point (see k_quant.cu): the scale s of a
// maximum |x| and a point count, the max |x| bits, the column sums at scale s
// (added into S; s from s_dev when non-NULL, else s_host), and m = S / (n 2^s)
int host_mean_scale(float amax, int64_t n);
cudaError_t launch_absmax_bits(const float *X, int64_t count, unsigned *bits, cudaStream_t st);
cudaError_t launch_colsum_fixed(const float *X, int64_t n, int d, const int *s_dev, int s_host,
                                unsigned long long *S, bool zero_first, cudaStream_t st);
cudaError_t launch_mean_fixed_finish(const unsigned long long *S, int d, int64_t n, const int *s_dev, int s_host,
                                     float *m, cudaStream_t st);
cudaError_t launch_mean_fixed(const float *X, int64_t n, int d, unsigned *bits, int *s_dev, unsigned long long *S,
                              float *m, cudaStream_t st);
cudaError_t launch_colmean_finish(const double *psum, int nblk, int d, int64_t n, float *m,
                                  double *mean_d, cudaStream_t st);
cudaError_t launch_rbq1_encode(const float *X, int64_t n, int d, const float *m, uint32_t *codes,
                               float *nx2, float *F, int32_t *popx, cudaStream_t st);
cudaError_t launch_rbq1_exponent(const float *F, int64_t n, unsigned int *maxbits, int *e_dev,
                                 cudaStream_t st);
// centroid preparation
cudaError_t launch_rbq1_cprep(const float *C, int k, int d, const float *m, uint4 *planes,
                              Rbq1CInfo *info, cudaStream_t st);
// fl(1 / sqrt(d)) as both sides of the estimator use it
inline float rbq1_isd(int d) { return (float)(1.0 / sqrt((double)d)); }
cudaError_t launch_rbq1_cprep_tc(const float *C, int k, int d, const float *m, uint8_t *yq, int dq,
                                 Rbq1CInfo *info, cudaStream_t st);
// symmetric 1-bit variant: binarized centroids (e4m3 +-1 codes and/or sign words)
cudaError_t launch_rbq1_cprep_sym(const float *C, int k, int d, const float *m, uint8_t *yq, int dq, uint32_t *yw,
                                  Rbq1CInfo *info, cudaStream_t st);
cudaError_t launch_assign_rbq1_sym(const uint32_t *codes, const float *nx2, const float *F, int64_t n, int d,
                                   const uint32_t *yw, const Rbq1CInfo *info, int k, int32_t *assign, float *dist,
                                   cudaStream_t st);
cudaError_t launch_row_sqnorm_u8(const uint8_t *codes, int64_t n, int d, int32_t *out,
                                 cudaStream_t st);
// assignment
cudaError_t launch_assign_exact_f32(const float *X, int64_t n, int d, const float *C, int k,
                                    int32_t *assign, float *dist, cudaStream_t st);
cudaError_t launch_assign_exact_bf16(const uint16_t *X, int64_t n, int d, const float *C, int k,
                                     int32_t *assign, float *dist, cudaStream_t st);
// keys (optional, max_rows entries): split the centroids across the grid
cudaError_t launch_assign_exact_rows(const void *X, int x_is_bf16, const int32_t *rows,
                                     const int32_t *count_dev, int64_t max_rows, int d,
                                     const float *C, int k, int32_t *assign, float *dist,
                                     unsigned long long *keys, cudaStream_t st);
cudaError_t launch_prune_assign(const void *X, int x_is_bf16, int64_t n, int d, const float *C,
                                int k, const int32_t *prev, int32_t *assign, float *dist,
                                unsigned long long *counters, cudaStream_t st);
cudaError_t launch_prune_assign_sq8(const uint8_t *X, int64_t n, int d, const uint8_t *C, int k, const int32_t *prev,
                                    int32_t *assign, float *dist, unsigned long long *counters, cudaStream_t st);
// Per-row state of the tensor-core pruning front (bf16 points): (threshold
// on s~ over the front, the seed's pruned distance or an upper bound of it),
// the seed centroid; with bounds kept across calls (all NULL otherwise):
// (||x_F|| rounded up, ||x_F||^2 rounded down), (bound bits, centroid) for
// the next call, per centroid (., ||c' - c||) since the bounds were written,
// and the device flag saying whether the kept bounds apply.
struct PfRows {
    float2 *thr = nullptr;
    int32_t *seed = nullptr;
    float2 *xn = nullptr;
    int2 *wrow = nullptr;
    const float2 *shift = nullptr;
    const int32_t *warm_ok = nullptr;
};
// the same pruning of bf16 points over the rows rows[0 .. *nrows) only
// (device count), one CTA per row, from the seeds and distances (or bounds)
// of r; writes r.wrow when kept
cudaError_t launch_prune_rows_cta(const uint16_t *X, int d, const float *C, int k, const PfRows &r,
                                  const int32_t *rows, const int32_t *nrows, int32_t *assign,
                                  float *dist, unsigned long long *counters, cudaStream_t st);
// Tensor-core pruning front (bf16 points, d <= 1024): per row the seed, the
// pruned distance to it and the threshold on s~ over the first F dimensions
// (hz = (max h', max z) of the front's centroid records); with kept bounds
// that apply and force_cold == 0, the seed and a bound from the kept state
// instead, without reading the points.
// skm_lloyd_step_host's pruned ranges after the first (skm_abi.cu): the
// tensor-core front on centroids prepared by the first range's call this step
// (its workspace ws0, planned for x0); otherwise a plain skm_assign.
int assign_range_shared(const skm_data *x, const void *C, int k, const int32_t *prev, int32_t *assign,
                        float *dist, void *ws, size_t ws_bytes, const skm_data *x0, void *ws0, size_t ws0_bytes,
                        cudaStream_t st);
cudaError_t launch_prune_front_prep(const uint16_t *X, int64_t n, int d, int F, const float *C, int k,
                                    const int32_t *prev, const float *hz, const PfRows &r, int force_cold,
                                    unsigned long long *ctr, cudaStream_t st);
// Rows rows[0 .. *nrows) with front survivors cand[row][cap] (nsub sub-lists
// of cap / nsub, 8-bit counts in cnt[row]; entries are positions, perm[pos]
// the centroid): the pruned distances of the survivors and the smallest
// (lowest index on ties).
cudaError_t launch_prune_finish(const uint16_t *X, int d, const float *C, const float2 *thr, const uint16_t *cand,
                                const int32_t *cnt, int cap, int nsub, const int32_t *perm, const int32_t *rows,
                                const int32_t *nrows, int32_t *assign, float *dist, int2 *wrow,
                                unsigned long long *ctr, cudaStream_t st);
cudaError_t launch_assign_sq8_simt(const uint8_t *X, int64_t n, int d, const uint8_t *C, int k,
                                   const int32_t *nx, const int32_t *nc, int32_t *assign,
                                   float *dist, cudaStream_t st);
cudaError_t launch_assign_rbq1(const uint32_t *codes, const float *nx2, const float *F,
                               const int32_t *popx, int64_t n, int d, const uint4 *planes,
                               const Rbq1CInfo *info, int k, int32_t *assign, float *dist,
                               cudaStream_t st);
// update
cudaError_t launch_histogram(const int32_t *assign, int64_t n, int k, int32_t *counts32,
                             cudaStream_t st);
// *out = number of j < k with counts[j] == 0
cudaError_t launch_count_zeros(const int64_t *counts, int k, int64_t *out, cudaStream_t st);
cudaError_t launch_scan_offsets(const int32_t *counts32, int k, int64_t *offsets,
                                int64_t *counts64_out, int accumulate_counts, cudaStream_t st);
cudaError_t launch_scatter(const int32_t *assign, int64_t n, int k, const int64_t *offsets,
                           int32_t *cursor, int32_t *perm, int32_t *scl, cudaStream_t st);
// load-balanced segmented sums over the cluster-sorted order (global atomics)
cudaError_t launch_chunk_sum_float(const void *X, int x_is_bf16, int64_t n, int d,
                                   const int32_t *perm, const int32_t *scl,
                                   const int64_t *offsets, int k, float *S_f, double *S_d,
                                   cudaStream_t st);
cudaError_t launch_chunk_sum_rbq1(const uint32_t *codes, const int64_t *fq_sorted, int64_t n, int d,
                                  const int32_t *perm, const int32_t *scl, const int64_t *offsets,
                                  int k, int64_t *T, cudaStream_t st);
cudaError_t launch_finalize_float32(const float *S, const int64_t *counts, int k, int d,
                                    float *C_inout, cudaStream_t st);
cudaError_t launch_segsum_sq8(const uint8_t *X, int d, const int32_t *perm,
                              const int64_t *offsets, int k, uint8_t *C_inout, int64_t *partial,
                              cudaStream_t st);
// Fq = round(F[perm[q]] 2^e) for the sorted positions q < offsets[k]
cudaError_t launch_rbq1_fq(const float *F, const int32_t *perm, const int64_t *offsets, int k,
                           int64_t n, int e, int64_t *fq_sorted, cudaStream_t st);
// streamed segmented sums (cp.async.bulk row gathers into shared-memory rings);
// *_ok says whether the row size and alignment suit them
bool ring_sum_float_ok(const void *X, int x_is_bf16, int d);
bool ring_sum_rbq1_ok(const void *codes, int d);
bool ring_sum_sq8_ok(const void *codes, int d);
// y = H_D diag(sigma) [x - mean; 0] / sqrt(D), D a power of two in [32, 4096]
cudaError_t launch_hadamard(const float *X, int64_t n, int d, const float *mean, const float *sigma, int D,
                            int out_bf16, void *Y, cudaStream_t st);
// stable sort of rows by key in [0, m) (m <= 12288): hist int32[ceil(n/4096)][m],
// sizes int32[m]; perm[q] = row at sorted position q, skey[q] its key
cudaError_t launch_stable_sort(const int32_t *key, int64_t n, int m, int32_t *hist, int32_t *sizes,
                               int32_t *perm, int32_t *skey, cudaStream_t st);
cudaError_t launch_gather_rows_bytes(const void *src, int64_t rowbytes, const int32_t *perm, int64_t n,
                                     void *dst, cudaStream_t st);
// out[perm[q]] = in[q] for 4-byte values
cudaError_t launch_unpermute(const void *in, const int32_t *perm, int64_t n, void *out, cudaStream_t st);
// x = y P^T + mu (n <= 65535 * 16 rows)
cudaError_t launch_unproject(const float *Y, int64_t n, int dout, const float *P, const float *mu, int d,
                             float *X, cudaStream_t st);
// empty clusters take half of the largest one (w: k int64 of workspace)
cudaError_t launch_split_empty(void *C, int code_bytes, const int64_t *counts, int k, int d,
                               int64_t *w, cudaStream_t st);
cudaError_t launch_ring_sum_sq8(const uint8_t *codes, int64_t n, int d, const int32_t *perm,
                                const int32_t *scl, const int64_t *offsets, int k, int64_t *S,
                                int32_t *flag, cudaStream_t st);
cudaError_t launch_ring_sum_float(const void *X, int x_is_bf16, int64_t n, int d, const int32_t *perm,
                                  const int32_t *scl, const int64_t *offsets, int k, float *S_f,
                                  double *S_d, int32_t *flag, cudaStream_t st);
cudaError_t launch_ring_sum_rbq1(const uint32_t *codes, const int64_t *fq_sorted, int64_t n, int d,
                                 const int32_t *perm, const int32_t *scl, const int64_t *offsets,
                                 int k, int64_t *T, int32_t *flag, cudaStream_t st);
cudaError_t launch_finalize_float(const double *partial, const int64_t *counts, int k, int d,
                                  float *C_inout, cudaStream_t st);
cudaError_t launch_finalize_sq8(const int64_t *partial, const int64_t *counts, int k, int d,
                                uint8_t *C_inout, cudaStream_t st);
cudaError_t launch_finalize_rbq1(const int64_t *partial, const int64_t *counts, int k, int d,
                                 const float *m, int e, float *C_inout, cudaStream_t st);
cudaError_t launch_merge(void *dst, const void *src, int64_t count, int elem_type,
                         cudaStream_t st);
// init / objective / projection / pca
cudaError_t launch_gather_rows(const void *X, int64_t n, int elem_bytes, int64_t row_elems,
                               const int64_t *idx, int k, void *out, int *status,
                               cudaStream_t st);
cudaError_t launch_rbq1_decode_rows(const uint32_t *codes, const float *F, int64_t n, int d,
                                    const float *m, int e, const int64_t *idx, int k,
                                    float *out, int *status, cudaStream_t st);
cudaError_t launch_objective(const void *X, int x_is_bf16, int64_t n, int d, const float *C,
                             const int32_t *assign, double *partials, int nblk,
                             cudaStream_t st);
cudaError_t launch_sum_double(const double *in, int64_t count, double *out, cudaStream_t st);
cudaError_t launch_sum_float_to_double(const float *in, int64_t count, double *partials,
                                       int nblk, cudaStream_t st);
cudaError_t launch_project(const float *X, int64_t n, int d, const float *mean, const float *P,
                           int d_out, int out_bf16, void *Y, cudaStream_t st);
cudaError_t launch_cov_partial(const float *X, int64_t n, int d, const float *mean,
                               double *partial, int splits, cudaStream_t st);
cudaError_t launch_cov_reduce(const double *partial, int splits, int d, double *cov,
                              cudaStream_t st);

// LVQ4 (Section 3.1 "LVQ4"; k_lvq4.cu).  Codes: uint32 [n][ceil(d/8)] nibbles;
// per-vector terms float4 (s, b, N, A) for points, (s, b, N, G) for centroids.
// dst (device) <- src (device address of mapped page-locked host memory)
cudaError_t launch_copy_from_host(const void *src, void *dst, size_t bytes, cudaStream_t st);
__host__ __device__ inline int lvq4_words(int d) { return (d + 7) / 8; }
cudaError_t launch_lvq4_encode(const float *X, int64_t n, int d, uint32_t *codes, float4 *fac,
                               cudaStream_t st);
cudaError_t launch_lvq4_exponent(const float4 *fac, int64_t n, unsigned int *maxbits, int *e_dev,
                                 cudaStream_t st);
// centroid re-encoding: yq != nullptr -> e4m3 bytes (row stride dq); yw != nullptr
// -> nibble words; info (s, b, N, G) per centroid
cudaError_t launch_lvq4_cprep(const float *C, int k, int d, uint8_t *yq, int dq, uint32_t *yw,
                              float4 *info, cudaStream_t st);
// nibble codes -> e4m3 bytes, row stride dq
cudaError_t launch_lvq4_expand(const uint32_t *codes, int64_t n, int d, uint8_t *xs, int dq,
                               cudaStream_t st);
// column-pair records for the tensor epilogue: bg = (b x2, G x2), sn = (s x2, N x2)
cudaError_t launch_lvq4_pack_pairs(const float4 *info, int k, int kp, float4 *bg, float4 *sn,
                                   cudaStream_t st);
cudaError_t launch_assign_lvq4_simt(const uint32_t *codes, const float4 *fac, int64_t n, int d,
                                    const uint32_t *yw, const float4 *info, int k, int32_t *assign,
                                    float *dist, cudaStream_t st);
// Sq = round(s 2^e) (uint32) and Bq = round(b 2^e) (int64) in cluster-sorted order
cudaError_t launch_lvq4_q(const float4 *fac, const int32_t *perm, const int64_t *offsets, int k, int64_t n,
                          int e, uint32_t *sq, int64_t *bq, cudaStream_t st);
bool ring_sum_lvq4_ok(const void *codes, int d);
cudaError_t launch_ring_sum_lvq4(const uint32_t *codes, const uint32_t *sq, const int64_t *bq, int64_t n,
                                 int d, const int32_t *perm, const int32_t *scl, const int64_t *offsets,
                                 int k, int64_t *T, int32_t *flag, cudaStream_t st);
cudaError_t launch_chunk_sum_lvq4(const uint32_t *codes, const uint32_t *sq, const int64_t *bq, int64_t n,
                                  int d, const int32_t *perm, const int32_t *scl, const int64_t *offsets,
                                  int k, int64_t *T, cudaStream_t st);
cudaError_t launch_finalize_lvq4(const int64_t *partial, const int64_t *counts, int k, int d, int e,
                                 float *C_inout, cudaStream_t st);
cudaError_t launch_lvq4_decode_rows(const uint32_t *codes, const float4 *fac, int64_t n, int d, int e,
                                    const int64_t *idx, int k, float *out, int *status, cudaStream_t st);

// host helpers (skm_linalg.cpp)
void philox_gaussians(uint64_t seed, int64_t count, double *out);
void forgy_indices(uint64_t seed, int64_t n, int k, int64_t *out);
void householder_qr_q(int d, double *A /* d*d in, Q out, row-major */);
int symmetric_eigen(int n, double *A /* in: symmetric; out: eigenvectors as columns */,
                    double *w /* eigenvalues */);

}  // namespace skm
