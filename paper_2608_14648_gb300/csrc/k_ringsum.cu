// Streamed segmented sums for the centroid update (Section 2.3 STEP 3; SQ8
// codes summed exactly in the code domain and, for 1-bit codes, the fused
// decode-average of Section 3.1 "RabitQ").
//
// The cluster-sorted member order is cut into runs of RS_ROWS positions and
// each of the RS_CW warps of a CTA owns one run.  A warp gathers the member
// rows of its run with cp.async.bulk (global -> shared, completion counted in
// bytes on one mbarrier per slot) into its own ring of slots, R rows per slot,
// one copy per lane, so that a whole slot is requested by one instruction and
// tens of rows per SM are in flight without holding them in registers.  It
// adds each row into register accumulators, refills the slot it has just read
// with the rows ns slots ahead, and flushes the accumulators into the
// cluster's global accumulator with atomics whenever the cluster id changes
// and at the end of the run; every warp has the same number of rows whatever
// the cluster sizes.
//
// Every barrier wait is bounded (2 s of %globaltimer).  A wait that gives up
// raises *flag (which skm_fit reports as SKM_ERR_TIMEOUT), the warp stops, and
// waits (bounded again) for the copies it issued before the CTA returns, so no
// copy lands in the shared memory of a finished CTA.
//
// 1-bit codes take a separate kernel (rows read straight into registers, bit
// transposes and subset-sum tables; see "1-bit rows" below).
#include <algorithm>

#include "skm_internal.cuh"

namespace skm {
namespace {

constexpr int RS_CW = 8;                      // warps per CTA, one run each
constexpr int RS_THREADS = 32 * RS_CW;
constexpr int RS_ROWS = 128;                  // sorted positions per consumer warp
constexpr int RS_MAX_SLOTS = 16;              // ring slots per consumer warp
constexpr int RS_RING_BYTES = 96 * 1024;      // all rings of a CTA
constexpr unsigned long long RS_WAIT_NS = 2000000000ull;

__device__ __forceinline__ uint32_t su32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ unsigned long long gtimer() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}
__device__ __forceinline__ void bar_init(uint32_t b, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(b), "r"(count) : "memory");
}
__device__ __forceinline__ void bar_arrive_tx(uint32_t b, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(b), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ bool bar_try(uint32_t b, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}\n"
        : "=r"(ok)
        : "r"(b), "r"(parity)
        : "memory");
    return ok != 0;
}
// false once the flag is up or the limit has elapsed (the flag is then raised)
__device__ __forceinline__ bool bar_wait(uint32_t b, uint32_t parity, volatile int32_t *flag) {
    if (bar_try(b, parity)) return true;
    const unsigned long long t0 = gtimer();
    for (uint32_t i = 1;; ++i) {
        if (bar_try(b, parity)) return true;
        if ((i & 63) == 0) {
            if (*flag) return false;
            if (gtimer() - t0 > RS_WAIT_NS) {
                *flag = 1;
                return false;
            }
        }
    }
}
// wait with a limit only (used to drain copies already issued)
__device__ __forceinline__ bool bar_wait_drain(uint32_t b, uint32_t parity) {
    const unsigned long long t0 = gtimer();
    while (!bar_try(b, parity))
        if (gtimer() - t0 > RS_WAIT_NS) return false;
    return true;
}
__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void *src, uint32_t bytes, uint32_t b) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
        "l"(src), "r"(bytes), "r"(b)
        : "memory");
}

__device__ __forceinline__ int run_len(int64_t nval, int64_t q0) {
    const int64_t r = nval - q0;
    return r <= 0 ? 0 : (r >= RS_ROWS ? RS_ROWS : (int)r);
}

// Shared-memory layout of one CTA: ns slots per warp, each holding up to R
// rows of rb bytes (R <= 32: one row per lane).
struct RingLayout {
    int ns, R, rb;
    int lsu;  // 1: rows gathered by 16-byte cp.async per lane (ns == LSU_STAGES)
    __host__ __device__ size_t slot_bytes() const { return (size_t)R * rb; }
    __host__ __device__ size_t ring_bytes() const { return (size_t)RS_CW * ns * slot_bytes(); }
    __host__ __device__ size_t bytes() const {
        return ring_bytes() + (size_t)RS_CW * ns * 8 + (size_t)RS_CW * RS_ROWS * 4;
    }
};

// Gather loop shared by every row type.  A warp calls cons.start(q0, cnt,
// lane) before the first row of its run (positions q0 .. q0 + cnt - 1),
// cons.row(i, row, lane) for its i-th row (in shared memory), and
// cons.finish(lane) after the last.
template <typename Consumer>
__device__ __forceinline__ void ring_run(const uint8_t *__restrict__ rows,
                                         const int32_t *__restrict__ perm, int64_t nval,
                                         RingLayout L, volatile int32_t *flag, Consumer &cons) {
    extern __shared__ __align__(128) uint8_t rs_smem[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const size_t sb = L.slot_bytes();
    uint8_t *ring = rs_smem + (size_t)warp * L.ns * sb;
    uint64_t *full = reinterpret_cast<uint64_t *>(rs_smem + L.ring_bytes()) + warp * L.ns;
    int32_t *sperm = reinterpret_cast<int32_t *>(rs_smem + L.ring_bytes() + (size_t)RS_CW * L.ns * 8) +
                     warp * RS_ROWS;
    const int64_t q0 = ((int64_t)blockIdx.x * RS_CW + warp) * RS_ROWS;
    const int cnt = run_len(nval, q0);
    if (cnt == 0) return;  // warp-uniform; no other warp waits on this one
    const uint32_t rb = (uint32_t)L.rb;
    if (lane == 0)
        for (int s = 0; s < L.ns; ++s) bar_init(su32(full + s), 1);
    for (int i = lane; i < cnt; i += 32) sperm[i] = perm[q0 + i];
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    __syncwarp();
    const int nch = (cnt + L.R - 1) / L.R;  // slots' worth of rows in this run
    // chunk j -> slot j % ns: lane 0 announces the bytes, lane r copies row r
    auto fill = [&](int j) {
        const int s = j % L.ns;
        const int nr = min(L.R, cnt - j * L.R);
        const uint32_t fb = su32(full + s);
        if (lane == 0) bar_arrive_tx(fb, (uint32_t)nr * rb);
        __syncwarp();
        if (lane < nr)
            bulk_g2s(su32(ring + (size_t)s * sb + (size_t)lane * rb),
                     rows + (size_t)sperm[j * L.R + lane] * rb, rb, fb);
    };
    const int pre = nch < L.ns ? nch : L.ns;
    for (int j = 0; j < pre; ++j) fill(j);
    int issued = pre, j = 0;
    cons.start(q0, cnt, lane);
    for (; j < nch; ++j) {
        const int s = j % L.ns;
        const bool ok = bar_wait(su32(full + s), (uint32_t)(j / L.ns) & 1u, flag);
        if (!__all_sync(0xffffffffu, ok)) break;
        const uint8_t *src = ring + (size_t)s * sb;
        const int nr = min(L.R, cnt - j * L.R);
        for (int r = 0; r < nr; ++r) cons.row(j * L.R + r, src + (size_t)r * rb, lane);
        if (j + L.ns < nch) {
            // the slot's generic-proxy reads are ordered before the async copies
            // that overwrite it
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            __syncwarp();
            fill(j + L.ns);
            ++issued;
        }
    }
    cons.finish(lane);
    // slots filled but never read (only after a wait gave up): let their
    // copies land before the CTA's shared memory goes away
    for (int jj = j; jj < issued; ++jj)
        if (!bar_wait_drain(su32(full + jj % L.ns), (uint32_t)(jj / L.ns) & 1u)) break;
    __syncwarp();
}

// Mid-size rows (about 1 KB, where the consumer does little work per byte):
// the warp's lanes gather the rows themselves with 16-byte cp.async (LSU
// path) into LSU_STAGES slots of R rows, one commit group per slot; a
// slot is read once cp.async.wait_group leaves only the younger groups
// pending (empty groups keep the count uniform at the tail).  These loads
// always complete, so there is no wait that could hang.
constexpr int LSU_STAGES = 4;
template <typename Consumer>
__device__ __forceinline__ void ring_run_lsu(const uint8_t *__restrict__ rows,
                                             const int32_t *__restrict__ perm, int64_t nval,
                                             RingLayout L, Consumer &cons) {
    extern __shared__ __align__(128) uint8_t rs_smem[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const size_t sb = L.slot_bytes();
    uint8_t *ring = rs_smem + (size_t)warp * LSU_STAGES * sb;
    int32_t *sperm = reinterpret_cast<int32_t *>(rs_smem + L.ring_bytes() + (size_t)RS_CW * L.ns * 8) +
                     warp * RS_ROWS;
    const int64_t q0 = ((int64_t)blockIdx.x * RS_CW + warp) * RS_ROWS;
    const int cnt = run_len(nval, q0);
    if (cnt == 0) return;
    for (int i = lane; i < cnt; i += 32) sperm[i] = perm[q0 + i];
    __syncwarp();
    const int rb = L.rb, per_row = rb >> 4;  // 16-byte pieces per row
    const int nch = (cnt + L.R - 1) / L.R;
    auto fill = [&](int j) {  // always commits one group (empty past the last chunk)
        if (j < nch) {
            uint8_t *dst = ring + (size_t)(j % LSU_STAGES) * sb;
            const int nr = min(L.R, cnt - j * L.R);
            for (int r = 0; r < nr; ++r) {
                const uint8_t *src = rows + (size_t)sperm[j * L.R + r] * rb;
                for (int c = lane; c < per_row; c += 32)
                    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(su32(dst + (size_t)r * rb + 16 * c)),
                                 "l"(src + 16 * c)
                                 : "memory");
            }
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
    };
#pragma unroll
    for (int j = 0; j < LSU_STAGES; ++j) fill(j);
    cons.start(q0, cnt, lane);
    for (int j = 0; j < nch; ++j) {
        asm volatile("cp.async.wait_group %0;" ::"n"(LSU_STAGES - 1) : "memory");
        __syncwarp();
        const uint8_t *src = ring + (size_t)(j % LSU_STAGES) * sb;
        const int nr = min(L.R, cnt - j * L.R);
        for (int r = 0; r < nr; ++r) cons.row(j * L.R + r, src + (size_t)r * rb, lane);
        __syncwarp();  // every lane has read the slot before it is refilled
        fill(j + LSU_STAGES);
    }
    cons.finish(lane);
    asm volatile("cp.async.wait_group 0;" ::: "memory");
}

template <typename Consumer>
__device__ __forceinline__ void ring_gather(const uint8_t *__restrict__ rows, const int32_t *__restrict__ perm,
                                            int64_t nval, RingLayout L, volatile int32_t *flag, Consumer &cons) {
    if (L.lsu)
        ring_run_lsu(rows, perm, nval, L, cons);
    else
        ring_run(rows, perm, nval, L, flag, cons);
}

// ---------------------------------------------------------- fp32 / bf16 rows
// Lane l holds columns 4 (l + 32 t) .. +3, t < NF.
template <bool BF16, typename ACC, int NF>
struct FloatCons {
    const int32_t *scl;
    ACC *S;
    int64_t stride;
    int d;
    float acc[4 * NF];
    int cur;
    int64_t q0;
    int clw, cln;  // cluster ids of this and the next 32 positions (lane-held)
    int cnt;
    __device__ __forceinline__ void flush(int c, int lane) {
#pragma unroll
        for (int t = 0; t < NF; ++t)
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int col = 4 * (lane + 32 * t) + u;
                if (col < d) atomicAdd(S + (int64_t)c * stride + col, (ACC)acc[4 * t + u]);
                acc[4 * t + u] = 0.0f;
            }
    }
    __device__ __forceinline__ void start(int64_t q0_, int cnt_, int lane) {
        q0 = q0_;
        cnt = cnt_;
#pragma unroll
        for (int t = 0; t < 4 * NF; ++t) acc[t] = 0.0f;
        clw = lane < cnt ? __ldg(scl + q0 + lane) : -1;
        cln = 32 + lane < cnt ? __ldg(scl + q0 + 32 + lane) : -1;
        cur = __shfl_sync(0xffffffffu, clw, 0);
    }
    __device__ __forceinline__ void row(int i, const uint8_t *slot, int lane) {
        if ((i & 31) == 0 && i > 0) {
            clw = cln;
            const int nx = i + 32 + lane;
            cln = nx < cnt ? __ldg(scl + q0 + nx) : -1;
        }
        const int c = __shfl_sync(0xffffffffu, clw, i & 31);
        if (c != cur) {
            flush(cur, lane);
            cur = c;
        }
        const int nq = d >> 2;  // float4 groups (d % 4 == 0 on this path)
#pragma unroll
        for (int t = 0; t < NF; ++t) {
            const int f = lane + 32 * t;
            if (f < nq) {
                if (BF16) {
                    const uint2 wv = reinterpret_cast<const uint2 *>(slot)[f];
                    acc[4 * t + 0] += __uint_as_float(wv.x << 16);
                    acc[4 * t + 1] += __uint_as_float(wv.x & 0xffff0000u);
                    acc[4 * t + 2] += __uint_as_float(wv.y << 16);
                    acc[4 * t + 3] += __uint_as_float(wv.y & 0xffff0000u);
                } else {
                    const float4 v = reinterpret_cast<const float4 *>(slot)[f];
                    acc[4 * t + 0] += v.x;
                    acc[4 * t + 1] += v.y;
                    acc[4 * t + 2] += v.z;
                    acc[4 * t + 3] += v.w;
                }
            }
        }
    }
    __device__ __forceinline__ void finish(int lane) { flush(cur, lane); }
};

template <bool BF16, typename ACC, int NF>
__global__ void __launch_bounds__(RS_THREADS) ring_sum_float_kernel(
    const void *__restrict__ X, int d, const int32_t *__restrict__ perm,
    const int32_t *__restrict__ scl, const int64_t *__restrict__ offsets, int k, ACC *__restrict__ S,
    int64_t stride, RingLayout L, int32_t *flag) {
    const int64_t nval = offsets[k];
    if ((int64_t)blockIdx.x * RS_CW * RS_ROWS >= nval) return;
    FloatCons<BF16, ACC, NF> cons;
    cons.scl = scl;
    cons.S = S;
    cons.stride = stride;
    cons.d = d;
    ring_gather(static_cast<const uint8_t *>(X), perm, nval, L, flag, cons);
}

// ------------------------------------------------------------- 1-bit rows
// T[c][i] += Fq for every member with bit i set; T[c][d] += Fq (= U) (the
// fused decode-average of Section 3.1 "RabitQ"), without a bit test and a
// predicated add per row and dimension.  A warp takes TR_ROWS sorted positions in
// chunks of 32 rows, lane r holding row r's W code words in registers (the
// next chunk's words load while this one is summed).  Per word, a 32 x 32
// bit transpose (five shuffle stages) leaves lane l with the bits of
// dimension 32 w + l over the chunk's rows, and the weighted sum over those
// bits is read from seven tables of subset sums of the rows' weights: rows
// 5g .. 5g + 4 (g < 6) and rows 30, 31 (g = 6), 32 entries each, so that a
// warp-wide lookup in one table touches every shared-memory bank once.  A
// chunk with two clusters runs once per cluster with the other rows' weights
// zero; a chunk with more takes its rows one at a time.  The sums stay in 32
// bits over a run (at most TR_ROWS = 128 weights of at most 2^24) and flush
// into the int64 accumulators when the cluster changes and at the run's end.
constexpr int TR_WARPS = 8;
constexpr int TR_ROWS = 128;

// Lane r holds row r of a 32 x 32 bit matrix (bit i = column i); afterwards
// lane i holds column i (bit r = row r).  Stage j exchanges j-bit groups with
// lane r ^ j: one shuffle, one rotate and one three-input select.
__device__ __forceinline__ uint32_t bit_transpose32(uint32_t x, int lane) {
    const uint32_t M[5] = {0x0000ffffu, 0x00ff00ffu, 0x0f0f0f0fu, 0x33333333u, 0x55555555u};
#pragma unroll
    for (int s = 0; s < 5; ++s) {
        const int j = 16 >> s;
        const bool up = (lane & j) != 0;
        const uint32_t keep = up ? ~M[s] : M[s];
        const uint32_t y = __shfl_xor_sync(0xffffffffu, x, j);
        const uint32_t yr = __funnelshift_l(y, y, up ? 32 - j : j);
        x = (x & keep) | (yr & ~keep);
    }
    return x;
}

// sum over the set bits r of t of the weight of row r, from the seven tables
// at shared address tbase (1 KiB aligned, so the offsets are OR-ed in)
__device__ __forceinline__ uint32_t lds_u32(uint32_t addr) {
    uint32_t v;
    asm("ld.shared.u32 %0, [%1];" : "=r"(v) : "r"(addr) : "memory");
    return v;
}
__device__ __forceinline__ uint32_t table_sum(uint32_t tbase, uint32_t t) {
    uint32_t s = lds_u32(tbase | ((t << 2) & 124u));
    s += lds_u32((tbase | 128u) | ((t >> 3) & 124u));
    s += lds_u32((tbase | 256u) | ((t >> 8) & 124u));
    s += lds_u32((tbase | 384u) | ((t >> 13) & 124u));
    s += lds_u32((tbase | 512u) | ((t >> 18) & 124u));
    s += lds_u32((tbase | 640u) | ((t >> 23) & 124u));
    s += lds_u32((tbase | 768u) | ((t >> 28) & 12u));
    return s;
}

template <int W4>
__device__ __forceinline__ uint32_t word_of(const uint4 (&x)[W4], int w) {
    const uint4 v = x[w >> 2];
    return (w & 3) == 0 ? v.x : (w & 3) == 1 ? v.y : (w & 3) == 2 ? v.z : v.w;
}

// PF: the next chunk's words load into registers while this one is summed
// (two CTAs per SM); without it three CTAs per SM hide the loads instead.
// Measured on GB300 (kernel time per 1M points): d = 768 81 us with PF
// against 95 without, d = 1024 120 us with PF against 113 without.
template <int W4>
constexpr bool tr_prefetch() { return W4 <= 6; }

template <int W4, bool PF>
__global__ void __launch_bounds__(TR_WARPS * 32, PF ? 2 : 3) rbq1_sum_table_kernel(
    const uint32_t *__restrict__ codes, const int64_t *__restrict__ fqs, int d,
    const int32_t *__restrict__ perm, const int32_t *__restrict__ scl,
    const int64_t *__restrict__ offsets, int k, unsigned long long *__restrict__ T) {
    constexpr int W = 4 * W4;
    __shared__ __align__(1024) uint32_t tabs[TR_WARPS][256];  // 7 x 32 entries used per warp
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t nval = offsets[k];
    const int64_t q0 = ((int64_t)blockIdx.x * TR_WARPS + warp) * TR_ROWS;
    if (q0 >= nval) return;  // warp-uniform; no other warp waits on this one
    const int cnt = (int)min((int64_t)TR_ROWS, nval - q0);
    uint32_t *tab = tabs[warp];
    const uint32_t tbase = (uint32_t)__cvta_generic_to_shared(tab);
    uint32_t acc[W];
#pragma unroll
    for (int w = 0; w < W; ++w) acc[w] = 0;
    unsigned long long usum = 0;  // this lane's share of U = sum Fq
    int cur = -1;
    auto flush = [&](int c) {
        unsigned long long *Tc = T + (int64_t)c * (d + 1);
#pragma unroll
        for (int w = 0; w < W; ++w) {
            const int col = 32 * w + lane;
            if (col < d && acc[w]) atomicAdd(Tc + col, (unsigned long long)acc[w]);
            acc[w] = 0;
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) usum += __shfl_xor_sync(0xffffffffu, usum, o);
        if (lane == 0 && usum) atomicAdd(Tc + d, usum);
        usum = 0;
    };
    // chunk ch: this lane's row words, cluster id (-1 past the run) and weight
    auto load = [&](int ch, uint4 (&x)[W4], int &cl, uint32_t &f) {
        const int i = ch * 32 + lane;
        if (i < cnt) {
            const int64_t q = q0 + i;
            const int64_t row = __ldg(perm + q);
            cl = __ldg(scl + q);
            f = (uint32_t)__ldg(fqs + q);  // Fq <= 2^24
            const uint4 *src = reinterpret_cast<const uint4 *>(codes + row * W);
#pragma unroll
            for (int g = 0; g < W4; ++g) x[g] = __ldg(src + g);
        } else {
            cl = -1;
            f = 0;
#pragma unroll
            for (int g = 0; g < W4; ++g) x[g] = make_uint4(0u, 0u, 0u, 0u);
        }
    };
    const int nch = (cnt + 31) >> 5;
    uint4 x[W4];
    int cl;
    uint32_t f;
    if (PF) load(0, x, cl, f);
    for (int ch = 0; ch < nch; ++ch) {
        uint4 xn[W4];
        int cln = -1;
        uint32_t fn = 0;
        if (PF) {
            if (ch + 1 < nch) load(ch + 1, xn, cln, fn);  // warp-uniform
        } else {
            load(ch, x, cl, f);
        }
        const bool valid = cl >= 0;
        // positions are sorted by cluster: each cluster's rows are contiguous
        const int clp = __shfl_up_sync(0xffffffffu, cl, 1);
        const int nseg = __popc(__ballot_sync(0xffffffffu, valid && (lane == 0 || cl != clp)));
        if (nseg <= 2) {
            int c = __shfl_sync(0xffffffffu, cl, 0);  // row 0 of a chunk is always valid
            for (;;) {
                if (c != cur) {
                    if (cur >= 0) flush(cur);
                    cur = c;
                }
                const bool in = valid && cl == c;
                const uint32_t fm = in ? f : 0u;
                usum += fm;
                __syncwarp();  // the previous lookups are done before the tables change
#pragma unroll
                for (int g = 0; g < 7; ++g) {
                    uint32_t e = 0;
#pragma unroll
                    for (int j = 0; j < (g < 6 ? 5 : 2); ++j) {
                        const uint32_t fj = __shfl_sync(0xffffffffu, fm, 5 * g + j);
                        e += ((lane >> j) & 1) ? fj : 0u;
                    }
                    tab[32 * g + lane] = e;
                }
                __syncwarp();
#pragma unroll
                for (int w = 0; w < W; ++w) acc[w] += table_sum(tbase, bit_transpose32(word_of(x, w), lane));
                const unsigned rest = __ballot_sync(0xffffffffu, valid && cl > c);
                if (!rest) break;
                c = __shfl_sync(0xffffffffu, cl, __ffs(rest) - 1);
            }
        } else {
            // many small clusters: one row at a time, its words broadcast
            const int nr = min(32, cnt - ch * 32);
            for (int r = 0; r < nr; ++r) {
                const int c = __shfl_sync(0xffffffffu, cl, r);
                const uint32_t fr = __shfl_sync(0xffffffffu, f, r);
                if (c != cur) {
                    if (cur >= 0) flush(cur);
                    cur = c;
                }
                if (lane == r) usum += fr;
                const uint32_t lm = 1u << lane;
#pragma unroll
                for (int w = 0; w < W; ++w) add_if_bit(acc[w], __shfl_sync(0xffffffffu, word_of(x, w), r), lm, fr);
            }
        }
        if (PF) {
#pragma unroll
            for (int g = 0; g < W4; ++g) x[g] = xn[g];
            cl = cln;
            f = fn;
        }
    }
    if (cur >= 0) flush(cur);
}

// --------------------------------------------------------------- SQ8 rows
// S[c][i] += code_i (int64).  Lane l holds the 16-byte column groups
// l + 32 t (t < NG).  Inside a run (at most RS_ROWS rows between flushes)
// each 32-bit word's four codes are summed as two words of two 16-bit lanes
// (bytes 0, 2 and bytes 1, 3), which cannot overflow (128 x 255 < 2^16).
template <int NG>
struct Sq8Cons {
    const int32_t *scl;
    unsigned long long *S;
    int d;
    uint32_t ev[4 * NG], od[4 * NG];  // per word: bytes 0,2 and bytes 1,3
    int cur;
    int64_t q0;
    int clw, cln;
    int cnt;
    __device__ __forceinline__ void flush(int c, int lane) {
#pragma unroll
        for (int t = 0; t < NG; ++t)
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int col = 16 * (lane + 32 * t) + 4 * u;
                if (col < d) {
                    unsigned long long *dst = S + (int64_t)c * d + col;
                    const uint32_t e = ev[4 * t + u], o = od[4 * t + u];
                    if (e & 0xffffu) atomicAdd(dst + 0, (unsigned long long)(e & 0xffffu));
                    if (o & 0xffffu) atomicAdd(dst + 1, (unsigned long long)(o & 0xffffu));
                    if (e >> 16) atomicAdd(dst + 2, (unsigned long long)(e >> 16));
                    if (o >> 16) atomicAdd(dst + 3, (unsigned long long)(o >> 16));
                }
                ev[4 * t + u] = 0u;
                od[4 * t + u] = 0u;
            }
    }
    __device__ __forceinline__ void start(int64_t q0_, int cnt_, int lane) {
        q0 = q0_;
        cnt = cnt_;
#pragma unroll
        for (int t = 0; t < 4 * NG; ++t) ev[t] = od[t] = 0u;
        clw = lane < cnt ? __ldg(scl + q0 + lane) : -1;
        cln = 32 + lane < cnt ? __ldg(scl + q0 + 32 + lane) : -1;
        cur = __shfl_sync(0xffffffffu, clw, 0);
    }
    __device__ __forceinline__ void row(int i, const uint8_t *slot, int lane) {
        uint4 w[NG];
        const int ng16 = d >> 4;  // 16-byte groups (d % 16 == 0 on this path)
#pragma unroll
        for (int t = 0; t < NG; ++t)
            if (lane + 32 * t < ng16) w[t] = reinterpret_cast<const uint4 *>(slot)[lane + 32 * t];
        row_regs(i, w, lane);
    }
    // the same with the lane's 16-byte groups of the row already in registers
    __device__ __forceinline__ void row_regs(int i, const uint4 (&wr)[NG], int lane) {
        if ((i & 31) == 0 && i > 0) {
            clw = cln;
            const int nx = i + 32 + lane;
            cln = nx < cnt ? __ldg(scl + q0 + nx) : -1;
        }
        const int c = __shfl_sync(0xffffffffu, clw, i & 31);
        if (c != cur) {
            flush(cur, lane);
            cur = c;
        }
        const int ng16 = d >> 4;
#pragma unroll
        for (int t = 0; t < NG; ++t) {
            const int gidx = lane + 32 * t;
            if (gidx < ng16) {
                const uint4 w = wr[t];
                ev[4 * t + 0] += w.x & 0x00ff00ffu;
                od[4 * t + 0] += (w.x >> 8) & 0x00ff00ffu;
                ev[4 * t + 1] += w.y & 0x00ff00ffu;
                od[4 * t + 1] += (w.y >> 8) & 0x00ff00ffu;
                ev[4 * t + 2] += w.z & 0x00ff00ffu;
                od[4 * t + 2] += (w.z >> 8) & 0x00ff00ffu;
                ev[4 * t + 3] += w.w & 0x00ff00ffu;
                od[4 * t + 3] += (w.w >> 8) & 0x00ff00ffu;
            }
        }
    }
    __device__ __forceinline__ void finish(int lane) { flush(cur, lane); }
};

template <int NG>
__global__ void __launch_bounds__(RS_THREADS) ring_sum_sq8_kernel(
    const uint8_t *__restrict__ codes, int d, const int32_t *__restrict__ perm,
    const int32_t *__restrict__ scl, const int64_t *__restrict__ offsets, int k,
    unsigned long long *__restrict__ S, RingLayout L, int32_t *flag) {
    const int64_t nval = offsets[k];
    if ((int64_t)blockIdx.x * RS_CW * RS_ROWS >= nval) return;
    Sq8Cons<NG> cons;
    cons.scl = scl;
    cons.S = S;
    cons.d = d;
    ring_gather(codes, perm, nval, L, flag, cons);
}

// SQ8 rows of at most 1 KB, read straight into registers: no ring.  Lane l
// loads the 16-byte groups l + 32 t of a row with 128-bit loads; the loads of
// the next SQ8_PF rows of the warp's run are in flight while a row is summed
// (a row's slot in the register buffer is refilled right after it is read),
// and with little shared memory many warps fit per SM.
constexpr int SQ8_PF = 4;
template <int NG>
__global__ void __launch_bounds__(RS_THREADS) direct_sum_sq8_kernel(
    const uint8_t *__restrict__ codes, int d, const int32_t *__restrict__ perm,
    const int32_t *__restrict__ scl, const int64_t *__restrict__ offsets, int k,
    unsigned long long *__restrict__ S) {
    __shared__ int32_t sperm_all[RS_CW][RS_ROWS];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t nval = offsets[k];
    const int64_t q0 = ((int64_t)blockIdx.x * RS_CW + warp) * RS_ROWS;
    const int cnt = run_len(nval, q0);
    if (cnt == 0) return;
    int32_t *sperm = sperm_all[warp];
    for (int i = lane; i < cnt; i += 32) sperm[i] = perm[q0 + i];
    __syncwarp();
    const int ng16 = d >> 4;
    auto load = [&](int r, uint4(&w)[NG]) {
        const uint4 *src = reinterpret_cast<const uint4 *>(codes + (size_t)sperm[r] * d);
#pragma unroll
        for (int t = 0; t < NG; ++t)
            if (lane + 32 * t < ng16) w[t] = __ldg(src + lane + 32 * t);
    };
    Sq8Cons<NG> cons;
    cons.scl = scl;
    cons.S = S;
    cons.d = d;
    uint4 buf[SQ8_PF][NG];
#pragma unroll
    for (int p = 0; p < SQ8_PF; ++p)
        if (p < cnt) load(p, buf[p]);
    cons.start(q0, cnt, lane);
    for (int r0 = 0; r0 < cnt; r0 += SQ8_PF) {
#pragma unroll
        for (int p = 0; p < SQ8_PF; ++p) {
            const int r = r0 + p;
            if (r < cnt) {  // warp-uniform
                cons.row_regs(r, buf[p], lane);
                if (r + SQ8_PF < cnt) load(r + SQ8_PF, buf[p]);
            }
        }
    }
    cons.finish(lane);
}

// bf16 rows of at most 1 KB (d <= 512, d % 8 == 0) straight into registers
// like the SQ8 rows: lane l loads the 16-byte groups l + 32 t (columns
// 8 (l + 32 t) .. + 7) of a row, a whole row per load instruction of the warp,
// with the next SQ8_PF rows' loads in flight while one is summed (one bulk
// copy per 512-byte row left the copy engine, not HBM, as the limit).
template <typename ACC, int NG>
__global__ void __launch_bounds__(RS_THREADS) direct_sum_bf16_kernel(
    const uint16_t *__restrict__ X, int d, const int32_t *__restrict__ perm,
    const int32_t *__restrict__ scl, const int64_t *__restrict__ offsets, int k, ACC *__restrict__ S,
    int64_t stride) {
    __shared__ int32_t sperm_all[RS_CW][RS_ROWS];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t nval = offsets[k];
    const int64_t q0 = ((int64_t)blockIdx.x * RS_CW + warp) * RS_ROWS;
    const int cnt = run_len(nval, q0);
    if (cnt == 0) return;
    int32_t *sperm = sperm_all[warp];
    for (int i = lane; i < cnt; i += 32) sperm[i] = perm[q0 + i];
    __syncwarp();
    const int ng = d >> 3;
    auto load = [&](int r, uint4(&w)[NG]) {
        const uint4 *src = reinterpret_cast<const uint4 *>(X + (size_t)sperm[r] * d);
#pragma unroll
        for (int t = 0; t < NG; ++t)
            if (lane + 32 * t < ng) w[t] = __ldg(src + lane + 32 * t);
    };
    float acc[8 * NG];
#pragma unroll
    for (int t = 0; t < 8 * NG; ++t) acc[t] = 0.0f;
    auto flush = [&](int c) {
#pragma unroll
        for (int t = 0; t < NG; ++t)
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int col = 8 * (lane + 32 * t) + u;
                if (col < d) atomicAdd(S + (int64_t)c * stride + col, (ACC)acc[8 * t + u]);
                acc[8 * t + u] = 0.0f;
            }
    };
    // cluster ids of positions 32 b .. 32 b + 31 (lane-held), this and the next window
    int clw = lane < cnt ? __ldg(scl + q0 + lane) : -1;
    int cln = 32 + lane < cnt ? __ldg(scl + q0 + 32 + lane) : -1;
    int cur = __shfl_sync(0xffffffffu, clw, 0);
    uint4 buf[SQ8_PF][NG];
#pragma unroll
    for (int p = 0; p < SQ8_PF; ++p)
        if (p < cnt) load(p, buf[p]);
    for (int r0 = 0; r0 < cnt; r0 += SQ8_PF) {
#pragma unroll
        for (int p = 0; p < SQ8_PF; ++p) {
            const int r = r0 + p;
            if (r < cnt) {  // warp-uniform
                if ((r & 31) == 0 && r > 0) {
                    clw = cln;
                    const int nx = r + 32 + lane;
                    cln = nx < cnt ? __ldg(scl + q0 + nx) : -1;
                }
                const int c = __shfl_sync(0xffffffffu, clw, r & 31);
                if (c != cur) {
                    flush(cur);
                    cur = c;
                }
#pragma unroll
                for (int t = 0; t < NG; ++t) {
                    if (lane + 32 * t < ng) {
                        const uint4 w = buf[p][t];
                        const uint32_t ww[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
                        for (int u = 0; u < 4; ++u) {
                            acc[8 * t + 2 * u] += __uint_as_float(ww[u] << 16);
                            acc[8 * t + 2 * u + 1] += __uint_as_float(ww[u] & 0xffff0000u);
                        }
                    }
                }
                if (r + SQ8_PF < cnt) load(r + SQ8_PF, buf[p]);
            }
        }
    }
    flush(cur);
}

// ------------------------------------------------------------- LVQ4 rows
// T[c][i] += Sq code_i (the fused decode-average of Section 3.1 "LVQ4"),
// T[c][d] += Bq.  Lane l holds nibble words l + 32 t (t < NW), 8 dimensions
// each.  Rows are taken in pairs of the same cluster: the two weights are
// split into 16-bit halves (lo = Sq & 0xffff, hi = Sq >> 16), the two rows'
// nibbles of two dimensions are interleaved into one word of bytes by a byte
// permute, and __dp2a adds lo_a x_a + lo_b x_b (and the same with hi) into
// 32-bit sums per dimension: about 1.6 instructions per row and dimension.  A
// row without a partner of its cluster pairs with a zero weight.  Inside a run
// of at most RS_ROWS rows the sums stay below 128 x 65535 x 15 < 2^32; the
// flush adds lo + hi 2^16 to the int64 accumulator.
template <int NW>
struct Lvq4Cons {
    const int32_t *scl;
    const uint32_t *sqs;  // Sq in sorted order
    const int64_t *bqs;   // Bq in sorted order
    unsigned long long *T;
    int d, W;
    uint32_t alo[8 * NW], ahi[8 * NW];
    uint32_t pw[NW];  // the row waiting for a partner
    uint32_t psq;
    bool pend;
    int64_t usum;
    int cur;
    int64_t q0;
    int clw, cln;
    uint32_t sqw, sqn;
    int64_t bqw, bqn;
    int cnt;
    __device__ __forceinline__ void flush(int c, int lane) {
#pragma unroll
        for (int t = 0; t < NW; ++t)
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int col = 8 * (lane + 32 * t) + j;
                const unsigned long long v =
                    (unsigned long long)alo[8 * t + j] + ((unsigned long long)ahi[8 * t + j] << 16);
                if (col < d && v) atomicAdd(T + (int64_t)c * (d + 1) + col, v);
                alo[8 * t + j] = 0u;
                ahi[8 * t + j] = 0u;
            }
        if (lane == 0 && usum) atomicAdd(T + (int64_t)c * (d + 1) + d, (unsigned long long)usum);
        usum = 0;
    }
    // rows a (words xa, weight sa) and b (xb, sb) of the current cluster
    __device__ __forceinline__ void pair(const uint32_t (&xa)[NW], uint32_t sa, const uint32_t (&xb)[NW], uint32_t sb) {
        const uint32_t wlo = (sa & 0xffffu) | (sb << 16);
        const uint32_t whi = (sa >> 16) | (sb & 0xffff0000u);
#pragma unroll
        for (int t = 0; t < NW; ++t) {
            const uint32_t ea = xa[t] & 0x0f0f0f0fu, oa = (xa[t] >> 4) & 0x0f0f0f0fu;
            const uint32_t eb = xb[t] & 0x0f0f0f0fu, ob = (xb[t] >> 4) & 0x0f0f0f0fu;
            const uint32_t m02 = __byte_perm(ea, eb, 0x5140), m46 = __byte_perm(ea, eb, 0x7362);
            const uint32_t m13 = __byte_perm(oa, ob, 0x5140), m57 = __byte_perm(oa, ob, 0x7362);
            uint32_t *lo = alo + 8 * t, *hi = ahi + 8 * t;
            lo[0] = __dp2a_lo(wlo, m02, lo[0]);
            lo[2] = __dp2a_hi(wlo, m02, lo[2]);
            lo[4] = __dp2a_lo(wlo, m46, lo[4]);
            lo[6] = __dp2a_hi(wlo, m46, lo[6]);
            lo[1] = __dp2a_lo(wlo, m13, lo[1]);
            lo[3] = __dp2a_hi(wlo, m13, lo[3]);
            lo[5] = __dp2a_lo(wlo, m57, lo[5]);
            lo[7] = __dp2a_hi(wlo, m57, lo[7]);
            hi[0] = __dp2a_lo(whi, m02, hi[0]);
            hi[2] = __dp2a_hi(whi, m02, hi[2]);
            hi[4] = __dp2a_lo(whi, m46, hi[4]);
            hi[6] = __dp2a_hi(whi, m46, hi[6]);
            hi[1] = __dp2a_lo(whi, m13, hi[1]);
            hi[3] = __dp2a_hi(whi, m13, hi[3]);
            hi[5] = __dp2a_lo(whi, m57, hi[5]);
            hi[7] = __dp2a_hi(whi, m57, hi[7]);
        }
    }
    __device__ __forceinline__ void single() {  // the waiting row with a zero-weight partner
        const uint32_t zero[NW] = {};
        pair(pw, psq, zero, 0u);
        pend = false;
    }
    __device__ __forceinline__ void start(int64_t q0_, int cnt_, int lane) {
        q0 = q0_;
        cnt = cnt_;
#pragma unroll
        for (int t = 0; t < 8 * NW; ++t) alo[t] = ahi[t] = 0u;
        pend = false;
        psq = 0u;
        usum = 0;
        clw = lane < cnt ? __ldg(scl + q0 + lane) : -1;
        cln = 32 + lane < cnt ? __ldg(scl + q0 + 32 + lane) : -1;
        sqw = lane < cnt ? __ldg(sqs + q0 + lane) : 0u;
        sqn = 32 + lane < cnt ? __ldg(sqs + q0 + 32 + lane) : 0u;
        bqw = lane < cnt ? __ldg(bqs + q0 + lane) : 0;
        bqn = 32 + lane < cnt ? __ldg(bqs + q0 + 32 + lane) : 0;
        cur = __shfl_sync(0xffffffffu, clw, 0);
    }
    __device__ __forceinline__ void row(int i, const uint8_t *slot, int lane) {
        if ((i & 31) == 0 && i > 0) {
            clw = cln;
            sqw = sqn;
            bqw = bqn;
            const int nx = i + 32 + lane;
            cln = nx < cnt ? __ldg(scl + q0 + nx) : -1;
            sqn = nx < cnt ? __ldg(sqs + q0 + nx) : 0u;
            bqn = nx < cnt ? __ldg(bqs + q0 + nx) : 0;
        }
        const int c = __shfl_sync(0xffffffffu, clw, i & 31);
        const uint32_t sq = __shfl_sync(0xffffffffu, sqw, i & 31);
        const int64_t bq = __shfl_sync(0xffffffffu, bqw, i & 31);
        if (c != cur) {  // warp-uniform
            if (pend) single();
            flush(cur, lane);
            cur = c;
        }
        usum += bq;
        const uint32_t *words = reinterpret_cast<const uint32_t *>(slot);
        uint32_t x[NW];
#pragma unroll
        for (int t = 0; t < NW; ++t) {
            const int w = lane + 32 * t;
            x[t] = w < W ? words[w] : 0u;
        }
        if (pend) {
            pair(pw, psq, x, sq);
            pend = false;
        } else {
#pragma unroll
            for (int t = 0; t < NW; ++t) pw[t] = x[t];
            psq = sq;
            pend = true;
        }
    }
    __device__ __forceinline__ void finish(int lane) {
        if (pend) single();
        flush(cur, lane);
    }
};

template <int NW>
__global__ void __launch_bounds__(RS_THREADS) ring_sum_lvq4_kernel(
    const uint32_t *__restrict__ codes, const uint32_t *__restrict__ sqs, const int64_t *__restrict__ bqs, int d,
    const int32_t *__restrict__ perm, const int32_t *__restrict__ scl, const int64_t *__restrict__ offsets, int k,
    unsigned long long *__restrict__ T, RingLayout L, int32_t *flag) {
    const int64_t nval = offsets[k];
    if ((int64_t)blockIdx.x * RS_CW * RS_ROWS >= nval) return;
    Lvq4Cons<NW> cons;
    cons.scl = scl;
    cons.sqs = sqs;
    cons.bqs = bqs;
    cons.T = T;
    cons.d = d;
    cons.W = lvq4_words(d);
    ring_gather(reinterpret_cast<const uint8_t *>(codes), perm, nval, L, flag, cons);
}

// Rows of [RS_LSU_MIN_ROW, RS_LSU_MAX_ROW) bytes take the LSU path (per-lane
// cp.async), all others one bulk copy each (measured on GB300 at 1M points:
// 1 KB SQ8 rows 0.294 vs 0.331 ms per update with the LSU path; 96-512 B code
// rows and 3 KB fp32 rows equal or faster with bulk copies).
constexpr uint32_t RS_LSU_MIN_ROW = 1024;
constexpr uint32_t RS_LSU_MAX_ROW = 2048;

bool ring_layout(uint32_t rb, RingLayout &L) {
    if (rb == 0 || rb % 16 != 0) return false;
    L.rb = (int)rb;
    if (rb >= RS_LSU_MIN_ROW && rb < RS_LSU_MAX_ROW) {
        L.lsu = 1;
        L.ns = LSU_STAGES;
        L.R = (int)std::max<size_t>(1, std::min<size_t>(32, RS_RING_BYTES / ((size_t)RS_CW * LSU_STAGES * rb)));
        return true;
    }
    L.lsu = 0;
    L.R = (int)std::max<uint32_t>(1u, std::min<uint32_t>(32u, 2048u / rb));
    L.ns = (int)std::min<size_t>(RS_MAX_SLOTS, RS_RING_BYTES / ((size_t)RS_CW * L.slot_bytes()));
    return L.ns >= 2;
}

unsigned ring_blocks(int64_t n) {
    const int64_t per = (int64_t)RS_CW * RS_ROWS;
    const int64_t b = (n + per - 1) / per;
    return (unsigned)(b < 1 ? 1 : b);
}

template <bool BF16, typename ACC>
cudaError_t launch_float_nf(int nf, const void *X, int64_t n, int d, const int32_t *perm,
                            const int32_t *scl, const int64_t *offsets, int k, ACC *S, RingLayout L,
                            int32_t *flag, cudaStream_t st) {
    const size_t smem = L.bytes();
    const unsigned g = ring_blocks(n);
#define RS_CASE(NFV)                                                                                \
    case NFV: {                                                                                     \
        auto kern = ring_sum_float_kernel<BF16, ACC, NFV>;                                          \
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem); \
        if (e != cudaSuccess) return e;                                                             \
        kern<<<g, RS_THREADS, smem, st>>>(X, d, perm, scl, offsets, k, S, d, L, flag);               \
        return launched();                                                                          \
    }
    switch (nf) {
        RS_CASE(2)
        RS_CASE(4)
        RS_CASE(6)
        RS_CASE(8)
        RS_CASE(12)
    default:
        return cudaErrorInvalidValue;
    }
#undef RS_CASE
}

}  // namespace

bool ring_sum_float_ok(const void *X, int x_is_bf16, int d) {
    RingLayout L;
    const uint32_t rb = (uint32_t)d * (x_is_bf16 ? 2u : 4u);
    return d % 4 == 0 && (reinterpret_cast<uintptr_t>(X) & 15u) == 0 && d <= 12 * 128 &&
           ring_layout(rb, L);
}

bool ring_sum_rbq1_ok(const void *codes, int d) {
    const int W = (d + 31) >> 5;
    return W % 4 == 0 && W <= 32 && (reinterpret_cast<uintptr_t>(codes) & 15u) == 0;
}

cudaError_t launch_ring_sum_float(const void *X, int x_is_bf16, int64_t n, int d, const int32_t *perm,
                                  const int32_t *scl, const int64_t *offsets, int k, float *S_f,
                                  double *S_d, int32_t *flag, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    if (x_is_bf16 && d % 8 == 0 && d <= 512 && (reinterpret_cast<uintptr_t>(X) & 15u) == 0) {
        // rows of at most 1 KB: straight into registers
        const unsigned g = ring_blocks(n);
        const uint16_t *Xb = static_cast<const uint16_t *>(X);
        if (d <= 256) {
            if (S_d) direct_sum_bf16_kernel<double, 1><<<g, RS_THREADS, 0, st>>>(Xb, d, perm, scl, offsets, k, S_d, d);
            else direct_sum_bf16_kernel<float, 1><<<g, RS_THREADS, 0, st>>>(Xb, d, perm, scl, offsets, k, S_f, d);
        } else {
            if (S_d) direct_sum_bf16_kernel<double, 2><<<g, RS_THREADS, 0, st>>>(Xb, d, perm, scl, offsets, k, S_d, d);
            else direct_sum_bf16_kernel<float, 2><<<g, RS_THREADS, 0, st>>>(Xb, d, perm, scl, offsets, k, S_f, d);
        }
        return launched();
    }
    RingLayout L;
    if (!ring_layout((uint32_t)d * (x_is_bf16 ? 2u : 4u), L)) return cudaErrorInvalidValue;
    const int q = (d / 4 + 31) / 32;  // float4 groups per lane
    const int nf = q <= 2 ? 2 : q <= 4 ? 4 : q <= 6 ? 6 : q <= 8 ? 8 : 12;
    if (S_d)
        return x_is_bf16 ? launch_float_nf<true, double>(nf, X, n, d, perm, scl, offsets, k, S_d, L, flag, st)
                         : launch_float_nf<false, double>(nf, X, n, d, perm, scl, offsets, k, S_d, L, flag, st);
    return x_is_bf16 ? launch_float_nf<true, float>(nf, X, n, d, perm, scl, offsets, k, S_f, L, flag, st)
                     : launch_float_nf<false, float>(nf, X, n, d, perm, scl, offsets, k, S_f, L, flag, st);
}

bool ring_sum_sq8_ok(const void *codes, int d) {
    RingLayout L;
    return d % 16 == 0 && d <= 4096 && (reinterpret_cast<uintptr_t>(codes) & 15u) == 0 &&
           ring_layout((uint32_t)d, L);
}

cudaError_t launch_ring_sum_sq8(const uint8_t *codes, int64_t n, int d, const int32_t *perm,
                                const int32_t *scl, const int64_t *offsets, int k, int64_t *S,
                                int32_t *flag, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    RingLayout L;
    if (!ring_layout((uint32_t)d, L)) return cudaErrorInvalidValue;
    const size_t smem = L.bytes();
    const unsigned g = ring_blocks(n);
    auto S64 = reinterpret_cast<unsigned long long *>(S);
    const int q = (d / 16 + 31) / 32;  // 16-byte groups per lane
    if (d <= 1024) {  // rows of at most 1 KB: straight into registers
        if (q <= 1)
            direct_sum_sq8_kernel<1><<<g, RS_THREADS, 0, st>>>(codes, d, perm, scl, offsets, k, S64);
        else
            direct_sum_sq8_kernel<2><<<g, RS_THREADS, 0, st>>>(codes, d, perm, scl, offsets, k, S64);
        return launched();
    }
#define RS_CASE(NGV)                                                                                \
    if (q <= NGV) {                                                                                 \
        auto kern = ring_sum_sq8_kernel<NGV>;                                                       \
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem); \
        if (e != cudaSuccess) return e;                                                             \
        kern<<<g, RS_THREADS, smem, st>>>(codes, d, perm, scl, offsets, k, S64, L, flag);            \
        return launched();                                                                          \
    }
    RS_CASE(1)
    RS_CASE(2)
    RS_CASE(4)
    RS_CASE(8)
#undef RS_CASE
    return cudaErrorInvalidValue;
}

cudaError_t launch_ring_sum_rbq1(const uint32_t *codes, const int64_t *fqs, int64_t n, int d,
                                 const int32_t *perm, const int32_t *scl, const int64_t *offsets,
                                 int k, int64_t *T, int32_t *flag, cudaStream_t st) {
    (void)flag;  // no waits in this kernel
    if (n == 0) return cudaSuccess;
    if (!ring_sum_rbq1_ok(codes, d)) return cudaErrorInvalidValue;
    const int W = (d + 31) >> 5;
    auto T64 = reinterpret_cast<unsigned long long *>(T);
    const int64_t per = (int64_t)TR_WARPS * TR_ROWS;
    const unsigned g = (unsigned)std::max<int64_t>(1, (n + per - 1) / per);
#define TR_CASE(W4V)                                                                                          \
    case W4V:                                                                                                 \
        rbq1_sum_table_kernel<W4V, tr_prefetch<W4V>()><<<g, TR_WARPS * 32, 0, st>>>(codes, fqs, d, perm, scl, \
                                                                                   offsets, k, T64);           \
        return launched();
    switch (W / 4) {
        TR_CASE(1)
        TR_CASE(2)
        TR_CASE(3)
        TR_CASE(4)
        TR_CASE(5)
        TR_CASE(6)
        TR_CASE(7)
        TR_CASE(8)
    default:
        break;
    }
#undef TR_CASE
    return cudaErrorInvalidValue;
}

bool ring_sum_lvq4_ok(const void *codes, int d) {
    RingLayout L;
    const int W = lvq4_words(d);
    return W % 4 == 0 && W <= 128 && (reinterpret_cast<uintptr_t>(codes) & 15u) == 0 &&
           ring_layout((uint32_t)W * 4u, L);
}

cudaError_t launch_ring_sum_lvq4(const uint32_t *codes, const uint32_t *sq, const int64_t *bq, int64_t n, int d,
                                 const int32_t *perm, const int32_t *scl, const int64_t *offsets, int k, int64_t *T,
                                 int32_t *flag, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    const int W = lvq4_words(d);
    RingLayout L;
    if (!ring_layout((uint32_t)W * 4u, L)) return cudaErrorInvalidValue;
    const size_t smem = L.bytes();
    const unsigned g = ring_blocks(n);
    auto T64 = reinterpret_cast<unsigned long long *>(T);
#define RS_CASE(NWV)                                                                                \
    case NWV: {                                                                                     \
        auto kern = ring_sum_lvq4_kernel<NWV>;                                                      \
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem); \
        if (e != cudaSuccess) return e;                                                             \
        kern<<<g, RS_THREADS, smem, st>>>(codes, sq, bq, d, perm, scl, offsets, k, T64, L, flag);    \
        return launched();                                                                          \
    }
    switch ((W + 31) / 32) {
        RS_CASE(1)
        RS_CASE(2)
        RS_CASE(3)
        RS_CASE(4)
    default:
        break;
    }
#undef RS_CASE
    return cudaErrorInvalidValue;
}

}  // namespace skm
