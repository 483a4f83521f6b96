// Tensor-core assignment (Section 2.3 STEP 2 "GEMM of the data points and
// centroids", Section 3.1 8-bit GEMM) on sm_103a with tcgen05 + TMEM + TMA.
//
// One persistent CTA per SM walks (point tile, centroid tile) jobs; its point
// tiles form two job streams whose jobs are issued alternately:
//   warp 0      TMA producer: 128 x 64 point slice and 256 x 64 centroid slice
//               (bf16, 128-byte swizzle) per stage, 4-stage mbarrier ring
//   warp 1      MMA issuer: 4 x tcgen05.mma.kind::f16 (M=128, N=256, K=16)
//               per stage into the stream's 128 x 256 fp32 TMEM accumulator
//   warps 2..   epilogue, one group of warps per stream: tcgen05.ld of the
//               accumulator (thread = point row; NH / 2 warps per TMEM lane
//               quarter, each taking a slice of the columns), fused per-row
//               reduction over centroids, so the N x K distance matrix never
//               leaves the SM; the column slices of a row merge through
//               shared memory at the end of its point tile
// Epilogues:
//  SCREEN (fp32 / bf16 points): bf16 operands, so the dot product carries a
//    rounding error.  Each pair gets a rigorous interval [L, U] for
//    s = ||c||^2 - 2 x.c (the distance minus ||x||^2) from per-row and
//    per-centroid bf16 residual norms.  Per row the epilogue keeps the
//    smallest U (Umin), the T smallest L among pairs with L <= Umin at the
//    time they are seen (a pair above the running Umin can never be the
//    nearest), and the smallest such L it could not keep (Lev).  The nearest
//    centroid has L <= Umin, so a row whose only such candidate is its first
//    is decided; rows with 2..T candidates are re-scored exactly in fp32;
//    rows with Lev <= Umin are rescanned over all k in fp32.
//  SQ8: centred codes (code - 128) are exact in bf16 and every partial sum is
//    an integer below 2^24 for d <= 1024, so the fp32 accumulator holds the
//    exact integer dot product; the epilogue forms the integer distance and
//    keeps the argmin (ties to the lowest index).
//  RBQ1: point bits as e4m3 -1 / +1 (2 xbar - 1) and centroid SQ4 codes as
//    e4m3 {0..15} (kind::f8f6f4, K = 32 per instruction), so the accumulator
//    is the exact integer 2P - sum ybar of Eq. final:rabitq (|.| <= 15 d; the
//    products are exact and every partial sum is an integer far below 2^24),
//    and the epilogue evaluates the estimator in fp32 in the library's fixed
//    order, so the result equals the AND+popcount kernel's bit for bit.
//  LVQ4: point and centroid codes 0..15 in e4m3, the accumulator is the exact
//    integer P = <xbar, ybar> (<= 225 d) of Eq. final:lvq.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <cfloat>
#include <mutex>

#include "skm_tc.cuh"

namespace skm {
namespace {

constexpr int BM = 128;  // points per tile (TMEM lanes)
constexpr int BN = 256;  // centroids per tile (fp32 accumulator columns)
constexpr int BK = 64;   // bf16 elements per 128-byte swizzle row
constexpr int STAGES = 4;
constexpr int A_STAGE = BM * BK * 2;  // 16 KiB
constexpr int B_STAGE = BN * BK * 2;  // 32 KiB
// 1-bit points kept packed in HBM: CONV_WARPS converter warps expand each of
// a CTA's point tiles once, a tile ahead of the producer, into that CTA's
// scratch in global memory (two slots per job stream, 128 rows of round16(d)
// e4m3 bytes each: at most PK_MAX_CTAS x 2 x 2 x 128 KiB, which L2 keeps),
// from where the TMA loads the A slices exactly as from an e4m3 copy of all
// the points.  The conversion is paid once per point tile instead of once
// per (point tile, centroid tile) job.
constexpr int CONV_WARPS = 4;
constexpr int PK_MAX_CTAS = 160;
// SKM_FLAG_WARM: stamp word 0 of a workspace whose last call completed
constexpr int64_t WARM_MAGIC = 0x534b4d5741524d31LL;
constexpr int TCAND = 4;
constexpr unsigned long long WAIT_LIMIT_NS = 2000000000ull;  // 2 s per barrier wait

enum { MODE_SCREEN = 0, MODE_SQ8 = 1, MODE_RBQ1 = 2, MODE_LVQ4 = 3, MODE_GEMM = 4, MODE_PFRONT = 5 };
// Epilogue warps per TMEM lane quarter, by mode.  Every CTA works alone
// (no thread-block clusters): it loads its own centroid slices.
constexpr int TC_NH[6] = {4, 4, 4, 4, 4, 4};
// Job streams per CTA, by mode.  NS = 2: the CTA's point tiles form two
// streams whose jobs the MMA warp issues alternately, each into its own TMEM
// accumulator, each drained by its own half of the epilogue warps; an
// epilogue group then has two MMA jobs' time per job.  NS = 1: one stream, the
// two accumulators alternate by job and every epilogue warp takes every job.
// (NS = 2 needs at least 256 epilogue threads per group for the e4m3 and SQ8
// records.)  Measured at 1M x 1000 x 768 against one stream: 1-bit 0.508 vs
// 0.574 ms, LVQ4 0.532 vs 0.575, fp32 screen 0.99 vs 1.02, SQ8 (with NH = 4)
// 0.847 vs 0.882.
constexpr int TC_NS[6] = {2, 2, 2, 2, 2, 2};
// GEMM mode (the projection Y = (X - mean) P in fp32 accuracy from bf16
// parts x = x1 + x2 + x3, P = p1 + p2 + p3): K segments of (A part, B part),
// the smallest products first; parts i + j > 4 (below 2^-24 relative) are left
// out.  The A parts are stacked as rows [part][n], the B parts as [part][dout].
constexpr int GEMM_NSEG = 6;
__device__ constexpr int GEMM_SEG_A[GEMM_NSEG] = {2, 1, 0, 1, 0, 0};
__device__ constexpr int GEMM_SEG_B[GEMM_NSEG] = {0, 1, 2, 0, 1, 0};
// Columns per TMEM load in the e4m3 epilogues (32: one load and wait per 32
// columns; 16: two buffers, the next load in flight).  Measured on GB300 at
// 1M x 1000 x 768 with two job streams: 16 for the 1-bit epilogue (0.511 vs
// 0.529 ms), 32 for LVQ4 (0.516 vs 0.531 ms).
template <int MODE>
constexpr int f8_cw() { return MODE == 3 /* MODE_LVQ4 */ ? 32 : 16; }
// The same choice for the fp32 / bf16 screen's epilogue, whose pass 1 is one
// packed FMA per column pair: 32 is 2-4% faster there (C1 1.014 vs 1.032 ms,
// C4 38.1 vs 39.7 ms).
constexpr int SCR_CW = 32;
// PFRONT: the tensor-core front of exact dimension pruning takes the first
// PF_DIMS dimensions; each row keeps at most PF_CAP survivors (PF_CAP / NHG
// per column slice of the epilogue, as 16-bit sorted positions, k <= 65536),
// more send it to the CUDA-core pruning over all k.  Measured on the 10M x 256 PCA workload (k = 10,000, bound from
// the previous centroid): 1.3 survivors a row after 128 dimensions (99.9% of
// rows at most 37), 80 after 64 (1% of rows above 2,000).
constexpr int PF_DIMS = 128;
constexpr int PF_CAP = 128;
// the e4m3 (kind::f8f6f4) modes: 128 elements per 128-byte K slice
template <int MODE>
constexpr bool f8_mode() { return MODE == MODE_RBQ1 || MODE == MODE_LVQ4; }

// Epilogue shape: NH warps per TMEM lane quarter (column slices of 256 / NH).
template <int NH>
constexpr int epi_threads() { return 128 * NH; }
template <int NH, bool PK = false>
constexpr int tc_threads() { return 64 + epi_threads<NH>() + (PK ? 32 * CONV_WARPS : 0); }
// one row's state for the merge: the screen list, or (best, index)
template <int MODE>
constexpr int merge_words() { return MODE == MODE_SCREEN ? 2 * TCAND + 2 : 2; }
// Per-centroid epilogue records of one centroid tile (256 columns): 4 KiB,
// double-buffered by job.
constexpr int REC_BYTES = 4096;
// 1024-byte alignment slack, the stages, barriers + TMEM slot (352 bytes), the
// merge buffer (per group, slices 1..NH/NS-1 publish) and the record buffers
// (two per group).
template <int MODE, int NH, int NS>
constexpr size_t tc_lut_offset() {  // LVQ4 read packed: byte -> two e4m3 codes, after the records
    return (size_t)STAGES * (A_STAGE + B_STAGE) + 512 + (size_t)(NH - NS) * BM * merge_words<MODE>() * 4 +
           2 * NS * REC_BYTES;
}
template <int MODE, int NH, int NS>
constexpr size_t tc_smem_bytes() {
    return 1024 + tc_lut_offset<MODE, NH, NS>() + (MODE == 3 /* MODE_LVQ4 */ ? 512 : 0);
}

struct TcParams {
    int64_t n;
    int64_t nrt;  // point tiles
    int k;
    int nct;  // centroid tiles
    int nkc;  // 64-wide k-slices
    const float4 *cinfo;  // SCREEN: per column pair (||c||^2 x2, h' x2), padded to 256
    const float *hz;      // SCREEN: (max h', max z) over the centroids
    const float2 *cinfoz; // SCREEN: per column pair (z x2)
    const float2 *xinfo;  // SCREEN: per point (||x~||, ||x~ - x||)
    int32_t *cand;        // SCREEN: [n][TCAND + 1]
    int32_t *resc_rows;
    int32_t *fall_rows;
    int32_t *counters;  // [0] rescore rows, [1] fallback rows, [2] abort flag
    int32_t *assign;
    const int32_t *nx;  // SQ8: centred ||x||^2
    const int32_t *nc;  // SQ8: centred ||c||^2, padded to 256 with a large value
    float *dist;        // SQ8 / RBQ1 (may be null)
    const float4 *rinfo;     // RBQ1: per column pair (bd x2, sd x2), padded
    const float4 *rinfoq;    // RBQ1: per column pair (-sum ybar x2, ||c - m||^2 x2)
    const float *nx2;        // RBQ1 per point
    const float *F;
    const int32_t *popx;
    const float4 *lvq;       // LVQ4 per point (s, b, N, A); rinfo / rinfoq hold
                             // the column pairs (b x2, G x2) / (s x2, N x2)
    int d;
    // RBQ1 read packed: the codes [n][pk_words] and the CTAs' expansion
    // scratch (slot ((cta NS + stream) 2 + i) of BM x pk_dp bytes)
    const uint32_t *pk_codes;
    uint8_t *pk_scratch;
    int pk_words, pk_dp;
    // SCREEN with SKM_FLAG_WARM (NULL otherwise): per row (bits of the bound
    // U on s for its centroid, that centroid) read at the start and written
    // at the end; per centroid (||c'||^2 - ||c||^2, ||c' - c||) since the
    // bounds were written; whether they apply (set by the centroid prep)
    int2 *warm_row;
    const float2 *warm_shift;
    const int32_t *warm_ok;
    // Segmented mode (all NULL otherwise): the point rows are sorted by
    // group and row r may only take centroids [seg_base[g], seg_base[g + 1])
    // of its group g = seg_group[r]; point tile rt covers the centroid tiles
    // seg_ct0[rt] .. seg_ct0[rt] + seg_nct[rt] - 1.
    const int32_t *seg_ct0;
    const int32_t *seg_nct;
    const int32_t *seg_group;
    const int32_t *seg_base;
    int nseg;
    // GEMM mode: Y [n][dout] (fp32, or bf16 bits when y_bf16), row stride ydout
    void *y;
    int y_bf16;
    int ydout;
    // PFRONT: per row (threshold on s~ over the front dimensions, the seed's
    // pruned distance), survivor lists [n][PF_CAP] (sorted positions, one
    // sub-list of PF_CAP / NHG per column slice), per listed row the
    // sub-lists' counts (8 bits each), the seed centroids (NULL: centroid 0)
    // and the pruning counters ([0] pairs alive after the front); the rows
    // listed for the CUDA-core finish and the rows whose lists overflowed
    // go to resc_rows / fall_rows (counts: counters[0] / counters[1], per call)
    const float2 *pf_thr;
    uint16_t *pf_cand;
    // PFRONT: the centroid operand and records are sorted by ||c_F||^2
    // (pf_perm: sorted position -> centroid); pf_cmin: per 32-column chunk of
    // sorted positions, the smallest ||c_F||^2
    const int32_t *pf_perm;
    const float *pf_cmin;
    int32_t *pf_cnt;
    const int32_t *pf_seed;
    unsigned long long *pf_ctr;
    int2 *pf_wrow;  // kept bounds: (bound bits, centroid) of decided rows (NULL: none)
    // Fault injection (0 = off): the producer first waits this long on a
    // barrier that nothing arrives on, so the launch gives up before it has
    // loaded anything and reports through the abort flag.
    unsigned long long inject_wait_ns;
};

// ------------------------------------------------------------- PTX helpers
__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ unsigned long long globaltimer() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}\n"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}
// Bounded wait: false when the abort flag is raised or the limit elapses
// (the flag is then raised so that every role stops).
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int32_t *abort_flag,
                                          unsigned long long limit_ns = WAIT_LIMIT_NS) {
    if (mbar_try_wait(bar, parity)) return true;
    const unsigned long long t0 = globaltimer();
    for (uint32_t i = 1;; ++i) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((i & 255) == 0) {
            if (*abort_flag) return false;
            if (globaltimer() - t0 > limit_ns) {
                *abort_flag = 1;
                return false;
            }
        }
    }
}
// Wait with the limit only (the abort flag is already up): used after a
// role gave up, to let the asynchronous copies or MMAs it had issued finish
// before the CTA releases its shared memory and TMEM.
__device__ __forceinline__ bool mbar_drain(uint32_t bar, uint32_t parity) {
    const unsigned long long t0 = globaltimer();
    for (uint32_t i = 0;; ++i) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((i & 255) == 255 && globaltimer() - t0 > WAIT_LIMIT_NS) return false;
    }
}
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *map, int x, int y,
                                            uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
        : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                     bar)
                 : "memory");
}
__device__ __forceinline__ void tc_mma(uint32_t dtmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                       uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(dtmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}
__device__ __forceinline__ void tc_mma_f8(uint32_t dtmem, uint64_t adesc, uint64_t bdesc,
                                          uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(dtmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}
// 32 lanes x 32 consecutive 32-bit columns: thread i receives lane (base + i).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&v)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
        "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),
          "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]),
          "=r"(v[14]), "=r"(v[15]), "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]),
          "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]), "=r"(v[25]),
          "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
        : "r"(taddr)
        : "memory");
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// 16 columns, no wait: the registers are valid only after tmem_wait16 on the
// same array (which names them as operands, so nothing reads them earlier).
__device__ __forceinline__ void tmem_ld16_async(uint32_t taddr, uint32_t (&v)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
          "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15])
        : "r"(taddr)
        : "memory");
}
__device__ __forceinline__ void tmem_wait16(uint32_t (&v)[16]) {
    asm volatile("tcgen05.wait::ld.sync.aligned;"
                 : "+r"(v[0]), "+r"(v[1]), "+r"(v[2]), "+r"(v[3]), "+r"(v[4]), "+r"(v[5]), "+r"(v[6]), "+r"(v[7]),
                   "+r"(v[8]), "+r"(v[9]), "+r"(v[10]), "+r"(v[11]), "+r"(v[12]), "+r"(v[13]), "+r"(v[14]),
                   "+r"(v[15])
                 :
                 : "memory");
}

// Packed fp32 pairs (two IEEE round-to-nearest operations per instruction).
__device__ __forceinline__ float2 ffma2(float2 a, float2 b, float2 c) {
    float2 r;
    asm("{\n\t.reg .b64 ra, rb, rc, rd;\n\t"
        "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\tmov.b64 rc, {%6, %7};\n\t"
        "fma.rn.f32x2 rd, ra, rb, rc;\n\tmov.b64 {%0, %1}, rd;\n\t}"
        : "=f"(r.x), "=f"(r.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
    return r;
}
__device__ __forceinline__ float2 fadd2(float2 a, float2 b) {
    float2 r;
    asm("{\n\t.reg .b64 ra, rb, rd;\n\t"
        "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
        "add.rn.f32x2 rd, ra, rb;\n\tmov.b64 {%0, %1}, rd;\n\t}"
        : "=f"(r.x), "=f"(r.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return r;
}
__device__ __forceinline__ float2 fmul2(float2 a, float2 b) {
    float2 r;
    asm("{\n\t.reg .b64 ra, rb, rd;\n\t"
        "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
        "mul.rn.f32x2 rd, ra, rb;\n\tmov.b64 {%0, %1}, rd;\n\t}"
        : "=f"(r.x), "=f"(r.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return r;
}

// Bits 0..3 of v -> four e4m3 bytes, bit j -> byte j: +1.0 (0x38) when set,
// -1.0 (0xB8) when clear.  The product puts bit j of the nibble at bit 8j + 7
// (the partial products land on distinct bits, so nothing carries).
__device__ __forceinline__ uint32_t pm1_e4m3(uint32_t v) {
    const uint32_t t = (v & 15u) * 0x10204080u;
    return (t & 0x80808080u) ^ 0xB8B8B8B8u;
}

// min(a, b, c) in one instruction (sm_100 family three-input min)
__device__ __forceinline__ float fmin3(float a, float b, float c) {
    float r;
    asm("min.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
    return r;
}

__device__ __forceinline__ float fmax3(float a, float b, float c) {
    float r;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
    return r;
}

// v[i] for a lane-dependent i in [0, 32): binary select tree (no local memory).
__device__ __forceinline__ uint32_t pick32(const uint32_t (&v)[32], int i) {
    uint32_t w16[16], w8[8], w4[4], w2[2];
#pragma unroll
    for (int t = 0; t < 16; ++t) w16[t] = (i & 16) ? v[t + 16] : v[t];
#pragma unroll
    for (int t = 0; t < 8; ++t) w8[t] = (i & 8) ? w16[t + 8] : w16[t];
#pragma unroll
    for (int t = 0; t < 4; ++t) w4[t] = (i & 4) ? w8[t + 4] : w8[t];
#pragma unroll
    for (int t = 0; t < 2; ++t) w2[t] = (i & 2) ? w4[t + 2] : w4[t];
    return (i & 1) ? w2[1] : w2[0];
}

__device__ __forceinline__ __attribute__((unused)) uint32_t pick16(const uint32_t (&v)[16], int i) {
    uint32_t w8[8], w4[4], w2[2];
#pragma unroll
    for (int t = 0; t < 8; ++t) w8[t] = (i & 8) ? v[t + 8] : v[t];
#pragma unroll
    for (int t = 0; t < 4; ++t) w4[t] = (i & 4) ? w8[t + 4] : w8[t];
#pragma unroll
    for (int t = 0; t < 2; ++t) w2[t] = (i & 2) ? w4[t + 2] : w4[t];
    return (i & 1) ? w2[1] : w2[0];
}
template <int N>
__device__ __forceinline__ uint32_t pickn(const uint32_t (&v)[N], int i) {
    if constexpr (N == 32)
        return pick32(v, i);
    else
        return pick16(v, i);
}

// Shared-memory matrix descriptor: K-major operand, 128-byte swizzle, rows of
// 128 bytes in 8-row (1024-byte) groups as written by TMA.  The start address
// advances by 32 bytes per K=16 step inside the swizzle row.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
    uint64_t d = (uint64_t)((saddr & 0x3FFFFu) >> 4);  // start address
    d |= (uint64_t)1 << 16;                            // leading byte offset (unused here)
    d |= (uint64_t)(1024 >> 4) << 32;                  // stride byte offset: 8 rows x 128 B
    d |= (uint64_t)1 << 46;                            // descriptor version (sm_100 family)
    d |= (uint64_t)2 << 61;                            // 128-byte swizzle
    return d;
}

// Instruction descriptors: D fp32, both operands K-major, N = 256, M = 128;
// kind::f16 with A/B bf16, kind::f8f6f4 with A/B e4m3.
constexpr uint32_t IDESC = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(BN >> 3) << 17) |
                           ((uint32_t)(BM >> 4) << 24);
constexpr uint32_t IDESC_F8 = (1u << 4) | ((uint32_t)(BN >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);

// ------------------------------------------------------ screening row state
// Per point row: the T smallest lower bounds L (sorted, indices J) among
// centroids that could still be the nearest, the smallest upper bound Umin,
// and Lev, the smallest such L that did not fit in the list.
struct ScreenRow {
    float L[TCAND];
    int J[TCAND];
    float umin, lev;
};

__device__ __forceinline__ void screen_init(ScreenRow &s) {
#pragma unroll
    for (int t = 0; t < TCAND; ++t) {
        s.L[t] = INFINITY;
        s.J[t] = 0x7fffffff;
    }
    s.umin = INFINITY;
    s.lev = INFINITY;
}

// Insert (L, j) into the sorted list; what falls off the end is kept in lev.
// (L, j) pairs are ordered by L, then by j.
__device__ __forceinline__ void screen_insert(ScreenRow &s, float L, int j) {
    const bool before3 = L < s.L[3] || (L == s.L[3] && j < s.J[3]);
    if (!before3) {
        s.lev = fminf(s.lev, L);
        return;
    }
    s.lev = fminf(s.lev, s.L[3]);
    if (L < s.L[0] || (L == s.L[0] && j < s.J[0])) {  // a new head: shift the list down
#pragma unroll
        for (int t = TCAND - 1; t > 0; --t) {
            s.L[t] = s.L[t - 1];
            s.J[t] = s.J[t - 1];
        }
        s.L[0] = L;
        s.J[0] = j;
        return;
    }
    float cl = L;
    int cj = j;
#pragma unroll
    for (int t = 0; t < TCAND; ++t) {  // bubble the new pair into place
        const bool lt = cl < s.L[t] || (cl == s.L[t] && cj < s.J[t]);
        const float tl = s.L[t];
        const int tj = s.J[t];
        s.L[t] = lt ? cl : tl;
        s.J[t] = lt ? cj : tj;
        cl = lt ? tl : cl;
        cj = lt ? tj : cj;
    }
}

// Centroid tiles [lo, hi) of point tile rt (every tile, or the tile's
// groups' range in segmented mode; none past the last point tile there).
__device__ __forceinline__ void ct_range(const TcParams &p, int64_t rt, int &lo, int &hi) {
    if (p.seg_ct0) {
        if (rt < p.nrt) {
            lo = p.seg_ct0[rt];
            hi = lo + p.seg_nct[rt];
        } else {
            lo = hi = 0;
        }
    } else {
        lo = 0;
        hi = p.nct;
    }
}

template <int MODE, int NH, bool SEG, int NS, bool PK>
__global__ void __launch_bounds__(tc_threads<NH, PK>(), 1)
    tc_assign_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                     const TcParams p) {
    static_assert(NS == 1 || (NS == 2 && NH % 2 == 0), "two job streams: two epilogue groups");
    static_assert(NS == 1 || MODE == MODE_GEMM ||
                      epi_threads<NH>() / NS >= (MODE == MODE_SCREEN || MODE == MODE_PFRONT ? 128 : 256),
                  "records staged by one epilogue group");
    static_assert(MODE != MODE_PFRONT || !SEG, "the pruning front has no segmented variant");
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t *smem = smem_raw + (base - raw);
    const uint32_t sA = base;
    const uint32_t sB = base + STAGES * A_STAGE;
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + (size_t)STAGES * (A_STAGE + B_STAGE));
    const uint32_t bar0 = smem_u32(bars);
    auto full_bar = [&](int s) { return bar0 + 8u * s; };
    auto empty_bar = [&](int s) { return bar0 + 8u * (STAGES + s); };
    auto tfull_bar = [&](int b) { return bar0 + 8u * (2 * STAGES + b); };
    auto tempty_bar = [&](int b) { return bar0 + 8u * (2 * STAGES + 2 + b); };
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(bars + 2 * STAGES + 4);
    // two more barriers after the TMEM slot: the MMA warp's drain on abort and
    // the injected wait (nothing arrives on either otherwise)
    const uint32_t drain_bar = bar0 + 8u * (2 * STAGES + 5);
    const uint32_t inject_bar = bar0 + 8u * (2 * STAGES + 6);
    // PK: scratch slot i of job stream j is written (count: one arrival per
    // converter warp) / free again (the MMA warp, once the last TMA load
    // from it has landed)
    auto sready_bar = [&](int j, int i) { return bar0 + 8u * (2 * STAGES + 7 + 2 * j + i); };
    auto sfree_bar = [&](int j, int i) { return bar0 + 8u * (2 * STAGES + 11 + 2 * j + i); };
    // PFRONT: 16 bytes after those (word 2 grp + (job & 1)) pass each epilogue
    // group's accumulator wait result to its other warps; the merge buffer
    // starts further on, 256 bytes after tmem_slot
    static_assert(8 * (2 * STAGES + 15) + 16 <= 8 * (2 * STAGES + 4) + 256, "group flags inside the barrier area");
    static_assert(!PK || MODE == MODE_RBQ1 || MODE == MODE_LVQ4, "packed points: 1-bit or LVQ4 codes");
    // PK, LVQ4: lut[b] = e4m3 codes of the two nibbles of byte b (low byte: low nibble)
    uint16_t *lut = reinterpret_cast<uint16_t *>(smem + tc_lut_offset<MODE, NH, NS>());
    if (PK && MODE == MODE_LVQ4)
        for (int i = threadIdx.x; i < 256; i += blockDim.x)
            lut[i] = (uint16_t)(e4m3_of_code(i & 15) | ((uint32_t)e4m3_of_code(i >> 4) << 8));
    // the epilogue's merge buffer starts 256 bytes after tmem_slot (see tc_smem_bytes)

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    volatile int32_t *abort_flag = p.counters + 2;
    constexpr int NSEG = MODE == MODE_GEMM ? GEMM_NSEG : 1;  // K segments per job
    constexpr int KC_ELEMS = f8_mode<MODE>() ? 128 : 64;  // elements per 128-byte row

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(full_bar(s), 1);
            mbar_init(empty_bar(s), 1);  // the MMA warp's commit
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(tfull_bar(b), 1);
            mbar_init(tempty_bar(b), epi_threads<NH>() / NS / 32);  // one arrival per epilogue warp
        }
        mbar_init(drain_bar, 1);
        mbar_init(inject_bar, 1);
        if (PK)
            for (int j = 0; j < NS; ++j)
                for (int i = 0; i < 2; ++i) {
                    mbar_init(sready_bar(j, i), CONV_WARPS);
                    mbar_init(sfree_bar(j, i), 1);
                }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmA)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmB)) : "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_u32(tmem_slot)),
                     "r"(512)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    // CTA b takes the point tiles b, b + grid, b + 2 grid, ...
    const int64_t g0 = (int64_t)blockIdx.x;
    const int64_t gstep = (int64_t)gridDim.x;
    const int64_t ngroups = p.nrt;

    // Job order (producer and MMA issuer walk it identically): stream s takes
    // the CTA's point-tile groups g0 + (s + NS i) gstep; the streams' jobs
    // (point tile, centroid tile) are issued round-robin.
    struct JobStream {
        int64_t g;
        int ct, hi;
    };
    auto stream_seek = [&](JobStream &js) {  // the first job at or after group js.g
        while (js.g < ngroups) {
            int lo, hi;
            ct_range(p, js.g, lo, hi);
            if (lo < hi) {
                js.ct = lo;
                js.hi = hi;
                return;
            }
            js.g += NS * gstep;
        }
    };
    auto stream_advance = [&](JobStream &js) {
        if (++js.ct >= js.hi) {
            js.g += NS * gstep;
            stream_seek(js);
        }
    };
    // the stream of the next job (turn first), or -1 when both are done;
    // streams are indexed by constants only, so they stay in registers
    auto stream_g = [&](const JobStream(&js)[NS], int s) { return s == 0 ? js[0].g : js[NS - 1].g; };
    auto stream_pick = [&](const JobStream(&js)[NS], int turn) {
        if (stream_g(js, turn) < ngroups) return turn;
        const int o = (turn + 1) % NS;
        return stream_g(js, o) < ngroups ? o : -1;
    };
    auto stream_take = [&](JobStream(&js)[NS], int s, int64_t &g, int &ct) {  // the job, then advance
        if (s == 0) {
            g = js[0].g;
            ct = js[0].ct;
            stream_advance(js[0]);
        } else {
            g = js[NS - 1].g;
            ct = js[NS - 1].ct;
            stream_advance(js[NS - 1]);
        }
    };

    if (warp == 0) {
        if (lane == 0) {  // ---------------------------------------- TMA producer
            uint32_t it = 0;
            if (p.inject_wait_ns && !mbar_wait(inject_bar, 0u, abort_flag, p.inject_wait_ns)) goto producer_done;
            {
            JobStream js[NS];
            int64_t ptile[NS];  // PK: each stream's current point tile and tiles taken
            uint32_t pcnt[NS];
            for (int s = 0; s < NS; ++s) {
                js[s].g = g0 + s * gstep;
                ptile[s] = -1;
                pcnt[s] = 0;
                stream_seek(js[s]);
            }
            for (int turn = 0;;) {
                const int sj = stream_pick(js, turn);
                if (sj < 0) break;
                int64_t gj;
                int ct;
                stream_take(js, sj, gj, ct);
                const int64_t rt = gj;
                turn = (sj + 1) % NS;
                int64_t arow0 = rt * BM;
                if (PK) {  // A comes from the stream's scratch slot of this tile
                    uint32_t pc = sj == 0 ? pcnt[0] : pcnt[NS - 1];
                    if ((sj == 0 ? ptile[0] : ptile[NS - 1]) != gj) {  // a new tile: wait for its expansion
                        if (!mbar_wait(sready_bar(sj, pc & 1u), (pc >> 1) & 1u, abort_flag)) goto producer_done;
                        ++pc;
                        if (sj == 0) {
                            ptile[0] = gj;
                            pcnt[0] = pc;
                        } else {
                            ptile[NS - 1] = gj;
                            pcnt[NS - 1] = pc;
                        }
                    }
                    arow0 = (((int64_t)blockIdx.x * NS + sj) * 2 + ((pc - 1u) & 1u)) * BM;
                }
                {
                    for (int kt = 0; kt < NSEG * p.nkc; ++kt, ++it) {
                        const int seg = kt / p.nkc, kc = kt - seg * p.nkc;
                        const int arow = (int)arow0 + (NSEG > 1 ? GEMM_SEG_A[seg] * (int)p.n : 0);
                        const int brow = ct * BN + (NSEG > 1 ? GEMM_SEG_B[seg] * p.k : 0);
                        const uint32_t s = it % STAGES, ph = (it / STAGES) & 1u;
                        if (!mbar_wait(empty_bar(s), ph ^ 1u, abort_flag)) goto producer_done;
                        mbar_expect_tx(full_bar(s), A_STAGE + B_STAGE);
                        tma_load_2d(sA + s * A_STAGE, &tmA, kc * KC_ELEMS, arow, full_bar(s));
                        tma_load_2d(sB + s * B_STAGE, &tmB, kc * KC_ELEMS, brow, full_bar(s));
                    }
                }
            }
            }
        producer_done:
            // Every stage fill issued so far lands before the CTA can exit (after
            // a normal run the MMA warp has consumed them all and this returns at
            // once; after an abort it waits for the copies still in flight).
            for (uint32_t s = 0; s < (uint32_t)STAGES && s < it; ++s) {
                const uint32_t last = s + ((it - 1u - s) / STAGES) * STAGES;
                mbar_drain(full_bar(s), (last / STAGES) & 1u);
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {  // ---------------------------------------- MMA issuer
            uint32_t it = 0, job = 0;
            bool issued = false, gave_up = true;
            uint32_t jc[NS];
            JobStream js[NS];
            int64_t mtile[NS];  // PK: each stream's current point tile and tiles taken
            uint32_t mcnt[NS];
            for (int s = 0; s < NS; ++s) {
                js[s].g = g0 + s * gstep;
                jc[s] = 0;
                mtile[s] = -1;
                mcnt[s] = 0;
                stream_seek(js[s]);
            }
            for (int turn = 0;; ++job) {
                const int sj = stream_pick(js, turn);
                if (sj < 0) break;
                // PK: whether this job is its tile's last, and the tile's scratch slot
                bool tile_last = false;
                uint32_t slot = 0;
                {
                    const int hij = sj == 0 ? js[0].hi : js[NS - 1].hi;
                    int64_t gj;
                    int ctj;
                    stream_take(js, sj, gj, ctj);
                    if (PK) {
                        uint32_t mc = sj == 0 ? mcnt[0] : mcnt[NS - 1];
                        if ((sj == 0 ? mtile[0] : mtile[NS - 1]) != gj) {
                            ++mc;
                            if (sj == 0) {
                                mtile[0] = gj;
                                mcnt[0] = mc;
                            } else {
                                mtile[NS - 1] = gj;
                                mcnt[NS - 1] = mc;
                            }
                        }
                        slot = (mc - 1u) & 1u;
                        tile_last = ctj == hij - 1;
                    }
                }
                turn = (sj + 1) % NS;
                {
                    // NS = 2: stream sj owns accumulator sj; NS = 1: they alternate
                    const uint32_t b = NS == 2 ? (uint32_t)sj : (job & 1u);
                    const uint32_t use = sj == 0 ? jc[0]++ : jc[NS - 1]++;
                    const uint32_t bph = NS == 2 ? (use & 1u) : ((job >> 1) & 1u);
                    if (!mbar_wait(tempty_bar(b), bph ^ 1u, abort_flag)) goto mma_done;
                    tc_fence_after();
                    const uint32_t dcol = tmem + b * BN;
                    for (int kc = 0; kc < NSEG * p.nkc; ++kc, ++it) {
                        const uint32_t s = it % STAGES, ph = (it / STAGES) & 1u;
                        if (!mbar_wait(full_bar(s), ph, abort_flag)) goto mma_done;
                        // PK: the tile's last slice has landed, so no TMA load
                        // reads its scratch slot any more
                        if (PK && tile_last && kc == NSEG * p.nkc - 1) mbar_arrive(sfree_bar(sj, slot));
                        tc_fence_after();
                        const uint64_t ad = sw128_desc(sA + s * A_STAGE);
                        const uint64_t bd = sw128_desc(sB + s * B_STAGE);
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk) {  // 4 x 32-byte K steps per 128-byte row
                            if (f8_mode<MODE>())
                                tc_mma_f8(dcol, ad + 2u * kk, bd + 2u * kk, IDESC_F8, (kc | kk) != 0);
                            else
                                tc_mma(dcol, ad + 2u * kk, bd + 2u * kk, IDESC, (kc | kk) != 0);
                        }
                        issued = true;
                        tc_commit(empty_bar(s));
                    }
                    tc_commit(tfull_bar(b));
                }
            }
            gave_up = false;
        mma_done:
            // After an abort, the MMAs issued so far complete before TMEM is
            // released (after a normal run the epilogue has waited for them all).
            if (gave_up && issued) {
                tc_commit(drain_bar);
                mbar_drain(drain_bar, 0u);
            }
        }
    } else if (PK && warp >= 2 + 4 * NH) {  // -------------------------- converters
        // Walks the producer's job order and expands a tile at its first job,
        // ahead of the producer (every tile the producer meets before a tile
        // this walk waits on has been expanded already, so neither waits on
        // the other): wait until the stream's scratch slot is free (its tile
        // two back has had all its A slices loaded), expand the tile's 128
        // packed rows (bit 1 -> +1.0 = 0x38, bit 0 -> -1.0 = 0xB8, the
        // tensor-core operand 2 xbar - 1; rows past n as -1; LVQ4 nibbles ->
        // their e4m3 integer codes, rows past n as 0) into round16(d)
        // e4m3 bytes a row, then make the writes visible to the TMA (async
        // proxy) and mark the slot ready.  Warp w takes rows w, w + CONV_WARPS,
        // ..., lanes over a row's 32-bit code words; code bits past d meet
        // zero centroid columns (the B map's width is d).
        const int cw = warp - (2 + 4 * NH);
        const int npair = (p.pk_dp + 31) >> 5;  // 32-dimension groups in a scratch row
        JobStream js[NS];
        int64_t ctile[NS];
        uint32_t ccnt[NS];
        for (int s = 0; s < NS; ++s) {
            js[s].g = g0 + s * gstep;
            ctile[s] = -1;
            ccnt[s] = 0;
            stream_seek(js[s]);
        }
        for (int turn = 0;;) {
            const int sj = stream_pick(js, turn);
            if (sj < 0) break;
            int64_t gj;
            int ct;
            stream_take(js, sj, gj, ct);
            turn = (sj + 1) % NS;
            if ((sj == 0 ? ctile[0] : ctile[NS - 1]) == gj) continue;  // not a tile's first job
            const uint32_t i = sj == 0 ? ccnt[0] : ccnt[NS - 1];
            if (sj == 0) {
                ctile[0] = gj;
                ccnt[0] = i + 1;
            } else {
                ctile[NS - 1] = gj;
                ccnt[NS - 1] = i + 1;
            }
            const uint32_t slot = i & 1u;
            if (!mbar_wait(sfree_bar(sj, slot), ((i >> 1) & 1u) ^ 1u, abort_flag)) goto conv_done;
            // the TMA's reads of the slot's previous tile before these writes
            asm volatile("fence.proxy.async.global;" ::: "memory");
            uint8_t *dst = p.pk_scratch + (((size_t)blockIdx.x * NS + sj) * 2 + slot) * BM * p.pk_dp;
            const int64_t r0 = gj * BM;
            constexpr int RB = 4;
            if constexpr (MODE == MODE_RBQ1) {
                // lane q takes code word q of the warp's rows (npair <= 32 for
                // d <= 1024); RB rows' loads in flight before they are expanded
                const bool act = lane < npair;
                for (int rb = 0; rb < BM / CONV_WARPS; rb += RB) {
                    uint32_t w[RB];
#pragma unroll
                    for (int u = 0; u < RB; ++u) {
                        const int64_t row = r0 + cw + CONV_WARPS * (rb + u);
                        w[u] = act && row < p.n ? __ldg(p.pk_codes + row * p.pk_words + lane) : 0u;
                    }
#pragma unroll
                    for (int u = 0; u < RB; ++u) {
                        if (!act) continue;
                        uint8_t *drow = dst + (size_t)(cw + CONV_WARPS * (rb + u)) * p.pk_dp + 32 * lane;
                        *reinterpret_cast<uint4 *>(drow) =
                            make_uint4(pm1_e4m3(w[u]), pm1_e4m3(w[u] >> 4), pm1_e4m3(w[u] >> 8), pm1_e4m3(w[u] >> 12));
                        if (32 * lane + 16 < p.pk_dp)
                            *reinterpret_cast<uint4 *>(drow + 16) = make_uint4(
                                pm1_e4m3(w[u] >> 16), pm1_e4m3(w[u] >> 20), pm1_e4m3(w[u] >> 24), pm1_e4m3(w[u] >> 28));
                    }
                }
            } else {
                // LVQ4: lane q takes nibble words q + 32 t (8 dimensions each; at
                // most 128 words for d <= 1024) of the warp's rows, RB rows' loads
                // in flight, each byte looked up as two e4m3 codes
                const int nq = p.pk_dp >> 3;  // 8-dimension words in a scratch row (<= pk_words)
                for (int rb = 0; rb < BM / CONV_WARPS; rb += RB) {
                    uint32_t w[RB][4];
#pragma unroll
                    for (int u = 0; u < RB; ++u) {
                        const int64_t row = r0 + cw + CONV_WARPS * (rb + u);
#pragma unroll
                        for (int t = 0; t < 4; ++t) {
                            const int q = lane + 32 * t;
                            w[u][t] = q < nq && row < p.n ? __ldg(p.pk_codes + row * p.pk_words + q) : 0u;
                        }
                    }
#pragma unroll
                    for (int u = 0; u < RB; ++u) {
                        uint8_t *drow = dst + (size_t)(cw + CONV_WARPS * (rb + u)) * p.pk_dp;
#pragma unroll
                        for (int t = 0; t < 4; ++t) {
                            const int q = lane + 32 * t;
                            if (q < nq) {
                                const uint32_t v = w[u][t];
                                *reinterpret_cast<uint2 *>(drow + 8 * q) =
                                    make_uint2((uint32_t)lut[v & 255u] | ((uint32_t)lut[(v >> 8) & 255u] << 16),
                                               (uint32_t)lut[(v >> 16) & 255u] | ((uint32_t)lut[v >> 24] << 16));
                            }
                        }
                    }
                }
            }
            asm volatile("fence.proxy.async.global;" ::: "memory");
            __syncwarp();
            if (lane == 0) mbar_arrive(sready_bar(sj, slot));
        }
    conv_done:;
    } else {  // ------------------------------------------------------- epilogue
        constexpr int NHG = NH / NS;     // warps per TMEM lane quarter in a group
        constexpr int GT = epi_threads<NH>() / NS;  // threads per group
        constexpr int SW = BN / NHG;     // columns per slice
        constexpr int MW = merge_words<MODE>();
        const int e = warp - 2;          // 0 .. 4 NH - 1
        const int q = warp & 3;          // TMEM lane quarter this warp may access
        const int grp = (e >> 2) / NHG;  // job stream (and accumulator) of this warp
        const int slice = (e >> 2) % NHG;  // which SW of the 256 columns
        const int rin = q * 32 + lane;   // row within the point tile
        // per group [NHG-1][BM][MW]
        uint32_t *merge = reinterpret_cast<uint32_t *>(tmem_slot + 64) + (size_t)grp * (NHG - 1) * BM * MW;
        // Records of the job's 256 centroids (SCREEN: 128 ||c||^2 pairs; RBQ1:
        // 128 rinfo + 128 rinfoq pairs; SQ8: 256 nc), copied into
        // shared memory at the start of each job from registers that were
        // loaded one job ahead, so the per-column reads are shared-memory
        // broadcasts.  Buffer (job & 1) is rewritten only after every epilogue
        // thread has passed the next job's barrier, i.e. finished reading it.
        uint8_t *rec_base = reinterpret_cast<uint8_t *>(reinterpret_cast<uint32_t *>(tmem_slot + 64) +
                                                        (size_t)(NH - NS) * BM * MW) +
                            (size_t)grp * 2 * REC_BYTES;  // this group's two buffers
        const int te = threadIdx.x - 64 - grp * GT;  // 0 .. GT - 1
        float4 pre4 = make_float4(0.f, 0.f, 0.f, 0.f);
        float2 pre2 = make_float2(0.f, 0.f);
        int32_t pre1 = 0;
        auto rec_load = [&](int ctn) {
            if (MODE == MODE_SCREEN || MODE == MODE_PFRONT) {
                if (te < 128) {
                    const float4 ci = __ldg(p.cinfo + ctn * 128 + te);
                    pre2 = make_float2(ci.x, ci.y);
                } else if (MODE == MODE_PFRONT && te < 130) {  // the tile's 8 chunk minima
                    pre4 = __ldg(reinterpret_cast<const float4 *>(p.pf_cmin + ctn * 8) + (te - 128));
                }
            } else if (f8_mode<MODE>()) {
                if (te < 128) pre4 = __ldg(p.rinfo + ctn * 128 + te);
                else if (te < 256) pre4 = __ldg(p.rinfoq + ctn * 128 + (te - 128));
            } else if (MODE == MODE_SQ8) {
                if (te < 256) pre1 = __ldg(p.nc + ctn * 256 + te);
            }
        };
        auto rec_store = [&](uint32_t buf) {
            uint8_t *rb = rec_base + buf * REC_BYTES;
            if (MODE == MODE_SCREEN || MODE == MODE_PFRONT) {
                if (te < 128) reinterpret_cast<float2 *>(rb)[te] = pre2;
                else if (MODE == MODE_PFRONT && te < 130) reinterpret_cast<float4 *>(rb + 1024)[te - 128] = pre4;
            } else if (f8_mode<MODE>()) {
                if (te < 256) reinterpret_cast<float4 *>(rb)[te] = pre4;
            } else if (MODE == MODE_SQ8) {
                if (te < 256) reinterpret_cast<int32_t *>(rb)[te] = pre1;
            }
        };
        {
            int lo0, hi0;
            ct_range(p, g0 + grp * gstep, lo0, hi0);
            rec_load(lo0);
        }
        // A warp whose barrier wait gave up stops computing but keeps taking part
        // in the named barriers, so the other epilogue warps never wait on it.
        bool dead = false;
        uint32_t job = 0;  // jobs of this group so far (NS = 1: of the CTA)
        unsigned long long pf_alive = 0;  // PFRONT: survivors of this thread's rows
        for (int64_t g = g0 + grp * gstep; g < ngroups; g += NS * gstep) {
            const int64_t rt = g;
            const int64_t row = rt * BM + rin;
            const bool valid = row < p.n;
            ScreenRow sr;
            screen_init(sr);
            int32_t best = 0x7fffffff, besti = 0x7fffffff;
            float fbest = INFINITY;
            float a2 = 0.0f, w2 = 0.0f, rnx2 = 0.0f, rf2 = 0.0f, rpc = 0.0f;
            int32_t nxr = 0;
            // PFRONT: survive iff s~ <= pthr; this slice's sub-list and count
            constexpr int PF_SUB = PF_CAP / NHG;
            float pthr = -INFINITY;
            int pcnt = 0;
            uint16_t *pf_list = nullptr;
            if (MODE == MODE_PFRONT && valid) {
                // finite, so that columns past k (s~ = +inf) never survive
                pthr = fminf(p.pf_thr[row].x, FLT_MAX);
                pf_list = p.pf_cand + row * PF_CAP + slice * PF_SUB;
            }
            // segmented mode: this row's centroid range (ids clamped into bounds)
            int cb = 0, ce = 0x7fffffff;
            if (SEG && valid) {
                int gi = p.seg_group[row];
                gi = gi < 0 ? 0 : (gi >= p.nseg ? p.nseg - 1 : gi);
                cb = p.seg_base[gi];
                ce = p.seg_base[gi + 1];
            }
            int ct_lo, ct_hi;
            ct_range(p, rt, ct_lo, ct_hi);
            int next_lo = 0;
            {
                int nhi;
                ct_range(p, g + NS * gstep, next_lo, nhi);
            }
            if (MODE == MODE_SCREEN) {
                a2 = valid ? 2.0f * p.xinfo[row].x : 0.0f;
                // 2 W_row, W_row = 2 ||x~|| max h' + max z >= every pair's half-width
                w2 = 2.0f * __fmaf_ru(a2, __ldg(p.hz), __ldg(p.hz + 1));
                if (p.warm_row && valid && *p.warm_ok) {
                    // s for the centroid the row had is at most U grown by its move:
                    // s(x, c') <= U + (||c'||^2 - ||c||^2) + 2 ||x|| ||c' - c||, with
                    // ||x|| <= ||x~|| + ||x~ - x||.  The nearest centroid j* has
                    // s~_j* <= s_j* + W_row, so a running minimum started at
                    // Un - W_row keeps the threshold (minimum + 2 W_row) above it.
                    const int2 wr = p.warm_row[row];
                    const float U = __int_as_float(wr.x);
                    if (wr.y >= 0 && wr.y < p.k && U < INFINITY) {
                        const float2 sh = __ldg(p.warm_shift + wr.y);
                        const float2 xi = p.xinfo[row];
                        const float xn = __fadd_ru(xi.x, xi.y);
                        const float Un = __fmaf_ru(2.0f * xn, sh.y, __fadd_ru(U, sh.x));
                        if (Un < INFINITY) sr.umin = __fsub_ru(Un, 0.5f * w2);
                    }
                }
            } else if (MODE == MODE_SQ8) {
                nxr = valid ? p.nx[row] : 0;
            } else if (MODE == MODE_LVQ4) {
                // per row: -2 s_x, -2 b_x, -2 A_x (exact) and N_x
                const float4 f = valid ? p.lvq[row] : make_float4(0.f, 0.f, 0.f, 0.f);
                rpc = __fmul_rn(-2.0f, f.x);
                rf2 = __fmul_rn(-2.0f, f.y);
                a2 = __fmul_rn(-2.0f, f.w);
                rnx2 = f.z;
            } else if (MODE == MODE_RBQ1) {
                rnx2 = valid ? p.nx2[row] : 0.0f;
                rf2 = valid ? __fmul_rn(-2.0f, p.F[row]) : 0.0f;  // exact
                rpc = valid ? (float)(2 * p.popx[row] - p.d) : 0.0f;
            }
            for (int ct = ct_lo; ct < ct_hi; ++ct, ++job) {
                // accumulator b (NS = 2: the group's own; NS = 1: alternating), its
                // use parity, and the record buffer (two per group, alternating)
                const uint32_t b = NS == 2 ? (uint32_t)grp : (job & 1u);
                const uint32_t bph = NS == 2 ? (job & 1u) : ((job >> 1) & 1u);
                const uint32_t rb = job & 1u;
                bool ok = true;
                if (MODE == MODE_PFRONT) {
                    // one warp of the group waits for the accumulator, the others
                    // park at the group barrier (which orders them after it); a
                    // wait that gave up has raised the abort flag
                    volatile uint32_t *grp_ok = reinterpret_cast<volatile uint32_t *>(bars + 2 * STAGES + 15) + 2 * grp + rb;
                    if (slice == 0 && q == 0) {
                        if (!dead) ok = mbar_wait(tfull_bar(b), bph, abort_flag);
                        ok = __all_sync(0xffffffffu, ok) && !dead;
                        if (lane == 0) *grp_ok = ok ? 1u : 0u;
                    }
                    rec_store(rb);
                    asm volatile("bar.sync %0, %1;" ::"r"(2 + grp), "n"(GT) : "memory");
                    dead = dead || *grp_ok == 0u;
                } else {
                    if (!dead) ok = mbar_wait(tfull_bar(b), bph, abort_flag);
                    dead = dead || !__all_sync(0xffffffffu, ok);
                    rec_store(rb);
                    asm volatile("bar.sync %0, %1;" ::"r"(2 + grp), "n"(GT) : "memory");
                }
                rec_load(ct + 1 < ct_hi ? ct + 1 : next_lo);
                if (dead) continue;
                tc_fence_after();
                const uint8_t *rbuf = rec_base + rb * REC_BYTES;
                const uint32_t taddr = tmem + ((uint32_t)(q * 32) << 16) + b * BN + slice * SW;
                const int jh = ct * BN + slice * SW;
                if (MODE == MODE_GEMM) {
                    // write the accumulator row out: 32 columns per TMEM load
#pragma unroll 1
                    for (int c = 0; c < SW / 32; ++c) {
                        const int col0 = jh + c * 32;
                        if (col0 >= p.ydout) break;  // warp-uniform
                        uint32_t v[32];
                        tmem_ld32(taddr + c * 32, v);
                        if (valid) {
                        if (p.y_bf16) {
                            uint16_t *yr = static_cast<uint16_t *>(p.y) + row * p.ydout;
                            if (col0 + 32 <= p.ydout && (p.ydout % 8) == 0) {
                                uint32_t w[16];
#pragma unroll
                                for (int i = 0; i < 16; ++i)
                                    w[i] = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(__uint_as_float(v[2 * i]))) |
                                           ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(__uint_as_float(v[2 * i + 1]))) << 16);
                                uint4 *dst = reinterpret_cast<uint4 *>(yr + col0);
#pragma unroll
                                for (int q4 = 0; q4 < 4; ++q4)
                                    dst[q4] = make_uint4(w[4 * q4], w[4 * q4 + 1], w[4 * q4 + 2], w[4 * q4 + 3]);
                            } else {
                                for (int i = 0; i < 32 && col0 + i < p.ydout; ++i)
                                    yr[col0 + i] = __bfloat16_as_ushort(__float2bfloat16_rn(__uint_as_float(pick32(v, i))));
                            }
                        } else {
                            float *yr = static_cast<float *>(p.y) + row * p.ydout;
                            if (col0 + 32 <= p.ydout && (p.ydout % 4) == 0) {
                                float4 *dst = reinterpret_cast<float4 *>(yr + col0);
#pragma unroll
                                for (int q4 = 0; q4 < 8; ++q4)
                                    dst[q4] = make_float4(__uint_as_float(v[4 * q4]), __uint_as_float(v[4 * q4 + 1]),
                                                          __uint_as_float(v[4 * q4 + 2]), __uint_as_float(v[4 * q4 + 3]));
                            } else {
                                for (int i = 0; i < 32 && col0 + i < p.ydout; ++i)
                                    yr[col0 + i] = __uint_as_float(pick32(v, i));
                            }
                        }
                        }
                    }
                } else if (MODE == MODE_SCREEN) {
                    // chunks of SCR_CW columns (16: the next TMEM load in flight)
                    constexpr int NC = SW / SCR_CW;
                    constexpr int G = SCR_CW / 8;
                    auto chunk = [&](uint32_t(&v)[SCR_CW], int c) {
                        const int j0 = jh + c * SCR_CW;
                        const int cc = slice * SW + c * SCR_CW;  // column offset within the tile
                        // pass 1, two columns per packed op: s~ = ||c||^2 - 2 acc (kept in
                        // v) and the chunk's smallest s~.  Records past k have ||c||^2 =
                        // +inf, so s~ = +inf.
                        float cm[G];
#pragma unroll
                        for (int g = 0; g < G; ++g) {
                            cm[g] = INFINITY;
#pragma unroll
                            for (int i = 8 * g; i < 8 * g + 8; i += 4) {
                                // ||c||^2 of four columns in one 16-byte broadcast load
                                const float4 c4 = reinterpret_cast<const float4 *>(rbuf)[(cc + i) >> 2];
                                const float2 a0 = make_float2(__uint_as_float(v[i]), __uint_as_float(v[i + 1]));
                                const float2 a1 = make_float2(__uint_as_float(v[i + 2]), __uint_as_float(v[i + 3]));
                                const float2 s0 = ffma2(make_float2(-2.0f, -2.0f), a0, make_float2(c4.x, c4.y));
                                const float2 s1 = ffma2(make_float2(-2.0f, -2.0f), a1, make_float2(c4.z, c4.w));
                                cm[g] = fmin3(cm[g], s0.x, s0.y);
                                cm[g] = fmin3(cm[g], s1.x, s1.y);
                                v[i] = __float_as_uint(s0.x);
                                v[i + 1] = __float_as_uint(s0.y);
                                v[i + 2] = __float_as_uint(s1.x);
                                v[i + 3] = __float_as_uint(s1.y);
                            }
                        }
                        if (SEG && (j0 < cb || j0 + SCR_CW > ce)) {
                            // segmented rows whose range cuts this chunk: columns
                            // outside it do not exist for this row
#pragma unroll
                            for (int g = 0; g < G; ++g) {
                                cm[g] = INFINITY;
#pragma unroll
                                for (int i = 8 * g; i < 8 * g + 8; ++i) {
                                    const bool in = j0 + i >= cb && j0 + i < ce;
                                    const float x = in ? __uint_as_float(v[i]) : INFINITY;
                                    v[i] = __float_as_uint(x);
                                    cm[g] = fminf(cm[g], x);
                                }
                            }
                        }
                        float cmin = cm[0];
#pragma unroll
                        for (int g = 1; g < G; ++g) cmin = fminf(cmin, cm[g]);
                        sr.umin = fminf(sr.umin, cmin);
                        const float thr = __fadd_ru(sr.umin, w2);
                        // pass 2 (rare once the running minimum is small): pairs within
                        // 2 W_row of the running minimum of s~ could still be the nearest
                        if (cmin <= thr && cmin < INFINITY) {
                            // only the 8-column groups whose minimum is inside
                            uint32_t mask = 0;
#pragma unroll
                            for (int g = 0; g < G; ++g) {
                                if (cm[g] <= thr && cm[g] < INFINITY) {
#pragma unroll
                                    for (int i = 8 * g; i < 8 * g + 8; ++i)
                                        mask |= (__uint_as_float(v[i]) <= thr ? 1u : 0u) << i;
                                }
                            }
                            if ((mask & (mask - 1u)) == 0u) {
                                // one column within the threshold (the usual case: a new
                                // running minimum): it is the chunk's minimum
                                screen_insert(sr, cmin, j0 + __ffs(mask) - 1);
                            } else {
                                while (mask) {
                                    const int i = __ffs(mask) - 1;
                                    mask &= mask - 1;
                                    screen_insert(sr, __uint_as_float(pickn<SCR_CW>(v, i)), j0 + i);
                                }
                            }
                        }
                    };
                    if constexpr (SCR_CW == 32) {
#pragma unroll 1
                        for (int c = 0; c < NC; ++c) {
                            if (jh + c * 32 >= p.k) break;  // warp-uniform
                            uint32_t v[32];
                            tmem_ld32(taddr + c * 32, v);
                            chunk(v, c);
                        }
                    } else if (jh < p.k) {  // warp-uniform conditions throughout
                        uint32_t va[16], vb[16];
                        tmem_ld16_async(taddr, va);
                        tmem_wait16(va);
#pragma unroll
                        for (int c = 0; c < NC; c += 2) {
                            const bool m1 = c + 1 < NC && jh + (c + 1) * 16 < p.k;
                            if (m1) tmem_ld16_async(taddr + (c + 1) * 16, vb);
                            chunk(va, c);
                            if (!m1) break;
                            tmem_wait16(vb);
                            const bool m2 = c + 2 < NC && jh + (c + 2) * 16 < p.k;
                            if (m2) tmem_ld16_async(taddr + (c + 2) * 16, va);
                            chunk(vb, c + 1);
                            if (!m2) break;
                            tmem_wait16(va);
                        }
                    }
                } else if (MODE == MODE_PFRONT) {
                    // Columns are centroids sorted by ||c_F||^2.  Per 32-column
                    // chunk: a = the largest accumulator (three-input maxima), and
                    // fl(cmin - 2 a) <= fl(||c_j||^2 - 2 acc_j) = s~_j for every
                    // column (rounding is monotone), so a chunk with fl(cmin - 2 a)
                    // > pthr has no survivor.  Otherwise (rare) each column's s~ is
                    // formed and those <= pthr are listed (sorted positions).
                    // Records past k have ||c_F||^2 = +inf.  The slices take
                    // alternate chunks (neighbouring positions, which similar
                    // survivors tend to share, go to different sub-lists).
                    // The warp releases the accumulator right after its last TMEM
                    // load, so the MMA can refill it while that chunk is evaluated.
                    const float *cmins = reinterpret_cast<const float *>(rbuf + 1024);
                    const uint32_t tbase = tmem + ((uint32_t)(q * 32) << 16) + b * BN;
                    int nvc = 0;  // this slice's chunks inside [0, k) (warp-uniform)
                    while (nvc < SW / 32 && ct * BN + (NHG * nvc + slice) * 32 < p.k) ++nvc;
                    if (nvc == 0) {
                        tc_fence_before();
                        __syncwarp();
                        if (lane == 0) mbar_arrive(tempty_bar(b));
                    }
#pragma unroll 1
                    for (int c = 0; c < nvc; ++c) {
                        const int cc = (NHG * c + slice) * 32;  // column offset within the tile
                        const int j0 = ct * BN + cc;
                        uint32_t v[32];
                        tmem_ld32(tbase + cc, v);
                        if (c == nvc - 1) {  // the warp's loads are complete (each thread waited)
                            tc_fence_before();
                            __syncwarp();
                            if (lane == 0) mbar_arrive(tempty_bar(b));
                        }
                        auto f = [&](int i) { return __uint_as_float(v[i]); };
                        float m[11];
#pragma unroll
                        for (int t = 0; t < 10; ++t) m[t] = fmax3(f(3 * t), f(3 * t + 1), f(3 * t + 2));
                        m[10] = fmaxf(f(30), f(31));
                        const float amax = fmax3(fmax3(m[0], m[1], m[2]), fmax3(m[3], m[4], m[5]),
                                                 fmax3(fmax3(m[6], m[7], m[8]), m[9], m[10]));
                        if (__fmaf_rn(-2.0f, amax, cmins[cc >> 5]) <= pthr && pf_list) {
                            uint32_t mask = 0;
#pragma unroll
                            for (int i = 0; i < 32; i += 4) {
                                const float4 c4 = reinterpret_cast<const float4 *>(rbuf)[(cc + i) >> 2];
                                mask |= (__fmaf_rn(-2.0f, f(i), c4.x) <= pthr ? 1u : 0u) << i;
                                mask |= (__fmaf_rn(-2.0f, f(i + 1), c4.y) <= pthr ? 2u : 0u) << i;
                                mask |= (__fmaf_rn(-2.0f, f(i + 2), c4.z) <= pthr ? 4u : 0u) << i;
                                mask |= (__fmaf_rn(-2.0f, f(i + 3), c4.w) <= pthr ? 8u : 0u) << i;
                            }
                            while (mask) {
                                const int i = __ffs(mask) - 1;
                                mask &= mask - 1u;
                                if (pcnt < PF_SUB) pf_list[pcnt] = (uint16_t)(j0 + i);
                                ++pcnt;
                            }
                        }
                    }
                } else if (f8_mode<MODE>()) {
                    // e4m3 modes: chunks of F8_CW columns (F8_CW = 16: the next
                    // chunk's TMEM load in flight while this one is evaluated)
                    constexpr int F8_CW = f8_cw<MODE>();
                    constexpr int NC = SW / F8_CW;
                    constexpr int G = F8_CW / 8;
                    auto chunk = [&](const uint32_t(&v)[F8_CW], int c) {
                        const int j0 = jh + c * F8_CW;
                        const int cc = slice * SW + c * F8_CW;
                        float gb[G];
                        int gi[G];
#pragma unroll
                        for (int g = 0; g < G; ++g) {
                            asm volatile("" ::: "memory");
                            gb[g] = INFINITY;
                            gi[g] = 0x7fffffff;
#pragma unroll
                            for (int i = 8 * g; i < 8 * g + 8; i += 2) {
                                const float4 r0 = reinterpret_cast<const float4 *>(rbuf)[(cc + i) >> 1];
                                const float4 r1 = reinterpret_cast<const float4 *>(rbuf)[128 + ((cc + i) >> 1)];
                                // the accumulator is the exact integer dot product (LVQ4:
                                // P = <xbar, ybar>; 1-bit: 2P - sum ybar, from +-1 codes)
                                const float2 P2 = make_float2(__uint_as_float(v[i]), __uint_as_float(v[i + 1]));
                                float2 est;
                                if (MODE == MODE_LVQ4) {
                                    // Eq. final:lvq: key = fma(b_y, -2 A_x, N_y),
                                    // fma(G_y, -2 b_x, .), fma(-2 s_x, s_y P, .)
                                    est = ffma2(make_float2(r0.x, r0.y), make_float2(a2, a2), make_float2(r1.z, r1.w));
                                    est = ffma2(make_float2(r0.z, r0.w), make_float2(rf2, rf2), est);
                                    const float2 t = fmul2(make_float2(r1.x, r1.y), P2);
                                    est = ffma2(make_float2(rpc, rpc), t, est);
                                } else {
                                    // Eq. final:rabitq in Eq. rabitq_l2: u = fma(sd, 2P -
                                    // sum ybar, bd pc), est = fma(-2F, u, nx2 + ny2)
                                    const float2 t = fmul2(make_float2(r0.x, r0.y), make_float2(rpc, rpc));
                                    const float2 u = ffma2(make_float2(r0.z, r0.w), P2, t);
                                    const float2 nn = fadd2(make_float2(rnx2, rnx2), make_float2(r1.z, r1.w));
                                    est = ffma2(make_float2(rf2, rf2), u, nn);
                                }
                                if (SEG && (j0 < cb || j0 + F8_CW > ce)) {  // columns outside the row's group
                                    if (j0 + i < cb || j0 + i >= ce) est.x = INFINITY;
                                    if (j0 + i + 1 < cb || j0 + i + 1 >= ce) est.y = INFINITY;
                                }
                                if (est.x < gb[g]) {
                                    gb[g] = est.x;
                                    gi[g] = j0 + i;
                                }
                                if (est.y < gb[g]) {
                                    gb[g] = est.y;
                                    gi[g] = j0 + i + 1;
                                }
                            }
                        }
                        // the groups hold increasing columns: the earlier wins ties
#pragma unroll
                        for (int g = 0; g < G; ++g)
                            if (gb[g] < fbest) {
                                fbest = gb[g];
                                besti = gi[g];
                            }
                    };
                    if constexpr (F8_CW == 32) {
#pragma unroll 1
                        for (int c = 0; c < NC; ++c) {
                            if (jh + c * 32 >= p.k) break;  // warp-uniform
                            uint32_t v[32];
                            tmem_ld32(taddr + c * 32, v);
                            chunk(v, c);
                        }
                    } else if (jh < p.k) {  // warp-uniform conditions throughout
                        uint32_t va[16], vb[16];
                        tmem_ld16_async(taddr, va);
                        tmem_wait16(va);
#pragma unroll
                        for (int c = 0; c < NC; c += 2) {
                            const bool m1 = c + 1 < NC && jh + (c + 1) * 16 < p.k;
                            if (m1) tmem_ld16_async(taddr + (c + 1) * 16, vb);
                            chunk(va, c);
                            if (!m1) break;
                            tmem_wait16(vb);
                            const bool m2 = c + 2 < NC && jh + (c + 2) * 16 < p.k;
                            if (m2) tmem_ld16_async(taddr + (c + 2) * 16, va);
                            chunk(vb, c + 1);
                            if (!m2) break;
                            tmem_wait16(va);
                        }
                    }
                } else
#pragma unroll 1
                for (int c = 0; c < SW / 32; ++c) {
                    const int j0 = jh + c * 32;
                    const int cc = slice * SW + c * 32;  // column offset within the tile
                    if (j0 >= p.k) break;  // warp-uniform
                    uint32_t v[32];
                    tmem_ld32(taddr + c * 32, v);
                    if (MODE == MODE_SQ8) {
#pragma unroll
                        for (int i = 0; i < 32; ++i) {
                            const int32_t dot = __float2int_rn(__uint_as_float(v[i]));
                            const int32_t dd = nxr + reinterpret_cast<const int32_t *>(rbuf)[cc + i] - 2 * dot;
                            if (dd < best && (!SEG || (j0 + i >= cb && j0 + i < ce))) {
                                best = dd;
                                besti = j0 + i;
                            }
                        }
                    }
                }
                // the warp's TMEM loads are complete (each thread waited on
                // them); one arrival for the warp releases its share (PFRONT:
                // released after its last load already)
                if (MODE != MODE_PFRONT) {
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(tempty_bar(b));
                }
            }
            // merge the column slices of each row: slices 1.. publish, slice 0 finishes
            // (single buffer: a publisher rewrites its slot only at the end of
            // the next point tile, after slice 0 has passed that tile's first
            // job barrier, i.e. after it has read this one)
            if (MODE == MODE_GEMM) continue;  // no per-row reduction across slices
            if (slice > 0) {
                uint32_t *slot = merge + ((slice - 1) * BM + rin) * MW;
                if (MODE == MODE_SCREEN) {
#pragma unroll
                    for (int t = 0; t < TCAND; ++t) {
                        slot[t] = __float_as_uint(sr.L[t]);
                        slot[TCAND + t] = (uint32_t)sr.J[t];
                    }
                    slot[2 * TCAND] = __float_as_uint(sr.umin);
                    slot[2 * TCAND + 1] = __float_as_uint(sr.lev);
                } else if (MODE == MODE_SQ8) {
                    slot[0] = (uint32_t)best;
                    slot[1] = (uint32_t)besti;
                } else if (MODE == MODE_PFRONT) {
                    slot[0] = (uint32_t)pcnt;
                } else {
                    slot[0] = __float_as_uint(fbest);
                    slot[1] = (uint32_t)besti;
                }
            }
            asm volatile("bar.sync %0, %1;" ::"r"(NS == 2 ? 4 + grp : 1), "n"(GT) : "memory");
            if (MODE == MODE_PFRONT && slice == 0 && valid && !dead) {
                // The row's survivors: one (the seed, whose pruned distance
                // every pruned pair provably exceeds) decides the row; 2 ..
                // PF_CAP go to the CUDA-core finish; more, or none
                // (impossible while the bounds hold), to pruning over all k.
                int tot = pcnt, one = pcnt == 1 ? 0 : -1;
                bool over = pcnt > PF_SUB;
                uint32_t packed = (uint32_t)min(pcnt, 255);
#pragma unroll
                for (int h = 1; h < NHG; ++h) {
                    const int ch = (int)merge[((h - 1) * BM + rin) * MW];
                    if (ch == 1) one = h;
                    tot += ch;
                    over = over || ch > PF_SUB;
                    packed |= (uint32_t)min(ch, 255) << (8 * h);
                }
                pf_alive += (unsigned long long)tot;
                const int seed = p.pf_seed[row];
                if (!over && tot == 1 && one >= 0 && p.pf_perm[p.pf_cand[row * PF_CAP + one * PF_SUB]] == seed) {
                    p.assign[row] = seed;
                    const float u = p.pf_thr[row].y;  // the seed's distance (or, kept bounds, a bound of it)
                    if (p.dist) p.dist[row] = u;
                    if (p.pf_wrow) p.pf_wrow[row] = make_int2(__float_as_int(u), seed);
                } else if (!over && tot >= 2) {
                    p.pf_cnt[row] = (int32_t)packed;
                    p.resc_rows[atomicAdd(p.counters, 1)] = (int32_t)row;
                } else {
                    p.fall_rows[atomicAdd(p.counters + 1, 1)] = (int32_t)row;
                }
            }
            if (MODE != MODE_PFRONT && slice == 0 && valid && !dead) {
                // slices in increasing column order; ties resolve to the lower index
#pragma unroll
                for (int h = 1; h < NHG; ++h) {
                    const uint32_t *slot = merge + ((h - 1) * BM + rin) * MW;
                    if (MODE == MODE_SCREEN) {
                        sr.umin = fminf(sr.umin, __uint_as_float(slot[2 * TCAND]));
                        sr.lev = fminf(sr.lev, __uint_as_float(slot[2 * TCAND + 1]));
#pragma unroll
                        for (int t = 0; t < TCAND; ++t)
                            screen_insert(sr, __uint_as_float(slot[t]), (int)slot[TCAND + t]);
                    } else if (MODE == MODE_SQ8) {
                        const int32_t ob = (int32_t)slot[0], oi = (int32_t)slot[1];
                        if (ob < best || (ob == best && oi < besti)) {
                            best = ob;
                            besti = oi;
                        }
                    } else {
                        const float ob = __uint_as_float(slot[0]);
                        const int32_t oi = (int32_t)slot[1];
                        if (ob < fbest || (ob == fbest && oi < besti)) {
                            fbest = ob;
                            besti = oi;
                        }
                    }
                }
                if (MODE == MODE_SCREEN) {
                    // The nearest centroid j* has s~_j* <= min s~ + 2 W_row (its own
                    // and the argmin's intervals), so it is a kept candidate unless the
                    // list overflowed (Lev inside the threshold).
                    const float thr = __fadd_ru(sr.umin, w2);
                    int ncert = 0;
#pragma unroll
                    for (int t = 0; t < TCAND; ++t) ncert += (sr.L[t] <= thr) ? 1 : 0;
                    const bool overflow = !(sr.lev > thr);
                    int nk = ncert;
                    int kj[TCAND];
#pragma unroll
                    for (int t = 0; t < TCAND; ++t) kj[t] = sr.J[t];
                    if (!overflow && ncert >= 2) {
                        // refine with each candidate's own interval [s~ - w, s~ + w],
                        // w = 2 ||x~|| h'_j + z_j (rounded outwards)
                        float lo[TCAND], umin = INFINITY;
#pragma unroll
                        for (int t = 0; t < TCAND; ++t) {
                            lo[t] = INFINITY;
                            if (t < ncert) {
                                const int j = sr.J[t];
                                const float4 ci = __ldg(p.cinfo + (j >> 1));
                                const float2 cz = __ldg(p.cinfoz + (j >> 1));
                                const float w = __fmaf_ru(a2, (j & 1) ? ci.w : ci.z, (j & 1) ? cz.y : cz.x);
                                umin = fminf(umin, __fadd_ru(sr.L[t], w));
                                lo[t] = __fsub_rd(sr.L[t], w);
                            }
                        }
                        nk = 0;
#pragma unroll
                        for (int t = 0; t < TCAND; ++t)
                            if (t < ncert && lo[t] <= umin) kj[nk++] = sr.J[t];
                    }
                    const int first = kj[0] < p.k ? kj[0] : 0;
                    p.assign[row] = first;
                    if (p.warm_row) {
                        // SKM_FLAG_WARM: a decided row keeps U = s~ + W_row >= s for
                        // its centroid; rows left to the fp32 passes keep none
                        int2 wr = make_int2(__float_as_int(INFINITY), -1);
                        if (!overflow && nk == 1) {
                            float Lj = INFINITY;
#pragma unroll
                            for (int t = 0; t < TCAND; ++t)
                                if (sr.J[t] == kj[0]) Lj = fminf(Lj, sr.L[t]);
                            wr = make_int2(__float_as_int(__fadd_ru(Lj, 0.5f * w2)), kj[0]);
                        }
                        p.warm_row[row] = wr;
                    }
                    if (!overflow && nk == 1) {
                        // decided by the screen
                    } else if (!overflow && nk >= 2) {
                        int32_t *cr = p.cand + row * (TCAND + 1);
#pragma unroll
                        for (int t = 0; t < TCAND; ++t) cr[t] = kj[t];
                        cr[TCAND] = nk;
                        p.resc_rows[atomicAdd(&p.counters[0], 1)] = (int32_t)row;
                    } else {
                        p.fall_rows[atomicAdd(&p.counters[1], 1)] = (int32_t)row;
                    }
                } else if (MODE == MODE_SQ8) {
                    p.assign[row] = besti;
                    if (p.dist) p.dist[row] = (float)best;
                } else if (MODE == MODE_LVQ4) {
                    p.assign[row] = besti;
                    if (p.dist) p.dist[row] = __fadd_rn(rnx2, fbest);
                } else {
                    p.assign[row] = besti;
                    if (p.dist) p.dist[row] = fbest;
                }
            }
        }
        if (MODE == MODE_PFRONT) {
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) pf_alive += __shfl_xor_sync(0xffffffffu, pf_alive, o);
            if (lane == 0 && pf_alive) atomicAdd(p.pf_ctr, pf_alive);
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(512)
                     : "memory");
    }
}

// ------------------------------------------------------------- preparation
// fp32 points -> bf16 screening copy (row stride dp) and per-row
// (||x~||, ||x~ - x||), both rounded up.  One warp per row.  The squares are
// summed in fp32 (each lane sequentially, then an xor tree): a sum of m
// non-negative terms carries a relative error below (m - 1) 2^-24 / (1 -
// (m - 1) 2^-24), so the sums are scaled up by 1 + (m + 2) 2^-23 (rounded
// up) before the upward-rounded square root.  x~_i - x_i is exact in fp32.
__device__ __forceinline__ float sumsq_upper_norm(float s, int terms) {
    const float grow = 1.0f + (float)(terms + 2) * 0x1p-23f;
    return __fsqrt_ru(__fmul_ru(s, grow));
}

constexpr int PREP_UNROLL = 8;

__global__ void screen_prep_f32_kernel(const float *__restrict__ X, int64_t n, int d, int dp,
                                       __nv_bfloat16 *__restrict__ xs, float2 *__restrict__ xinfo,
                                       unsigned int *__restrict__ rho_max_bits) {
    const int lane = threadIdx.x & 31;
    const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int W = (d + 31) >> 5;
    const int terms = W + 5;  // longest chain of roundings: per-lane terms + 5 tree levels
    float rho_local = 0.0f;
    for (int64_t r = warp; r < n; r += nw) {
        float a2 = 0.0f, r2 = 0.0f;
        for (int w0 = 0; w0 < W; w0 += PREP_UNROLL) {
            float v[PREP_UNROLL];
#pragma unroll
            for (int u = 0; u < PREP_UNROLL; ++u) {
                const int i = 32 * (w0 + u) + lane;
                v[u] = (i < d) ? __ldg(X + r * d + i) : 0.0f;
            }
#pragma unroll
            for (int u = 0; u < PREP_UNROLL; ++u) {
                const int i = 32 * (w0 + u) + lane;
                if (i < d) {
                    const __nv_bfloat16 xb = __float2bfloat16_rn(v[u]);
                    xs[r * dp + i] = xb;
                    const float xf = __bfloat162float(xb);
                    const float e = __fsub_rn(xf, v[u]);
                    a2 = __fmaf_rn(xf, xf, a2);
                    r2 = __fmaf_rn(e, e, r2);
                }
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            a2 = __fadd_rn(a2, __shfl_xor_sync(0xffffffffu, a2, o));
            r2 = __fadd_rn(r2, __shfl_xor_sync(0xffffffffu, r2, o));
        }
        if (lane == 0) {
            const float an = sumsq_upper_norm(a2, terms);
            const float rn = sumsq_upper_norm(r2, terms);
            xinfo[r] = make_float2(an, rn);
            // ratio ||x~ - x|| / ||x~|| (rounded up); x~ = 0 only when x = 0
            const float rho = an > 0.0f ? __fdiv_ru(rn, an) : 0.0f;
            rho_local = (rho == rho) ? fmaxf(rho_local, rho) : INFINITY;  // NaN (inf data): no bound
        }
    }
    // one atomic per warp; non-negative floats order like their bit patterns
    if (lane == 0 && rho_local > 0.0f) atomicMax(rho_max_bits, __float_as_uint(rho_local));
}

// bf16 points: optional padded copy (when the row stride is not a multiple of
// 16 bytes) and (||x||, 0): the points are the screening operand exactly.
__global__ void screen_prep_bf16_kernel(const uint16_t *__restrict__ X, int64_t n, int d, int dp,
                                        uint16_t *__restrict__ xs, float2 *__restrict__ xinfo) {
    const int lane = threadIdx.x & 31;
    const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int terms = (d + 31) / 32 + 5;
    for (int64_t r = warp; r < n; r += nw) {
        float a2 = 0.0f;
        for (int i = lane; i < d; i += 32) {
            const uint16_t v = X[r * d + i];
            if (xs) xs[r * dp + i] = v;
            const float xf = __uint_as_float(((uint32_t)v) << 16);
            a2 = __fmaf_rn(xf, xf, a2);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) a2 = __fadd_rn(a2, __shfl_xor_sync(0xffffffffu, a2, o));
        if (lane == 0) xinfo[r] = make_float2(sumsq_upper_norm(a2, terms), 0.0f);
    }
}

// SQ8 codes -> centred bf16 (code - 128, exact) and centred ||x||^2 (exact).
__global__ void screen_prep_sq8_kernel(const uint8_t *__restrict__ X, int64_t n, int d, int dp,
                                       __nv_bfloat16 *__restrict__ xs, int32_t *__restrict__ nx) {
    const int lane = threadIdx.x & 31;
    const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    for (int64_t r = warp; r < n; r += nw) {
        int32_t s = 0;
        for (int i = lane; i < d; i += 32) {
            const int32_t v = (int32_t)X[r * d + i] - 128;
            xs[r * dp + i] = __int2bfloat16_rn(v);
            s += v * v;
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
        if (lane == 0) nx[r] = s;
    }
}

// Centroids (fp32) -> bf16 operand + (||c||^2, h', z, 0) with
// h' = e + (eps_acc + eps_s) (||c|| + e) + rho_max ||c||, e = ||c~ - c||,
// z = eps_s ||c||^2, where rho_max >= ||x~ - x|| / ||x~|| over all points, so
// |s~ - s| <= 2 ||x~|| h' + z = w (the half-width of the pair's interval).
// Records j in [k, kp) get ||c||^2 = +inf so they never matter.  The operand
// and the records cover the first dr dimensions (dr = d, or the pruning
// front's prefix).  Layout:
// column pair p = (2p, 2p+1) -> cinfo[p] = (||c||^2 x2, h' x2), cinfoz[p] = (z x2);
// hz_bits (zeroed by the caller) receives max h' and max z over j < k.
//
// SKM_FLAG_WARM (cprev non-NULL): also shift[j] = (||c_j||^2 - ||cprev_j||^2,
// ||c_j - cprev_j||), each rounded up (fp64 sums of products of fp32 values,
// plus a margin far above their rounding), then cprev_j = c_j; thread 0
// publishes in *warm_ok whether the stamp names this n, d and k (the bounds
// and cprev then belong to these points; with cgen, also cprev's generation,
// which it then advances) and clears the stamp until this call completes.
__global__ void cprep_f32_kernel(const float *__restrict__ C, int k, int kp, int d, int dp, int dr,
                                 float eps_acc, float eps_s, const float *__restrict__ rho_max,
                                 __nv_bfloat16 *__restrict__ cs, float4 *__restrict__ cinfo,
                                 float2 *__restrict__ cinfoz, unsigned int *__restrict__ hz_bits,
                                 float *__restrict__ cprev, float2 *__restrict__ shift,
                                 int64_t *__restrict__ warm_hdr, int64_t n, int32_t *__restrict__ warm_ok,
                                 int64_t *__restrict__ cgen) {
    const int lane = threadIdx.x & 31;
    const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int nw = (gridDim.x * blockDim.x) >> 5;
    const double rho = (double)*rho_max;
    if (cprev && blockIdx.x == 0 && threadIdx.x == 0) {
        // cgen (the pruning front): cprev's generation, which the stamp must
        // name too (bounds taken against exactly these previous centroids)
        const int64_t g = cgen ? *cgen : 0;
        *warm_ok = warm_hdr[0] == WARM_MAGIC && warm_hdr[1] == n && warm_hdr[2] == d && warm_hdr[3] == k &&
                   (!cgen || warm_hdr[4] == g);
        warm_hdr[0] = 0;
        if (cgen) *cgen = g + 1;
    }
    float *cf = reinterpret_cast<float *>(cinfo);
    float *zf = reinterpret_cast<float *>(cinfoz);
    for (int j = warp; j < kp; j += nw) {
        const int pp = j >> 1, o = j & 1;
        if (j >= k) {
            if (lane == 0) {
                cf[4 * pp + o] = INFINITY;
                cf[4 * pp + 2 + o] = 0.0f;
                zf[2 * pp + o] = 0.0f;
            }
            continue;
        }
        double c2 = 0.0, e2 = 0.0, p2 = 0.0, dd = 0.0, dn = 0.0;
        const int iend = cprev ? d : dr;
        for (int i = lane; i < iend; i += 32) {
            const float c = C[(int64_t)j * d + i];
            if (i < dr) {
                const __nv_bfloat16 cb = __float2bfloat16_rn(c);
                cs[(int64_t)j * dp + i] = cb;
                const double cf = (double)__bfloat162float(cb);
                c2 += (double)c * (double)c;
                e2 += (cf - (double)c) * (cf - (double)c);
            }
            if (cprev) {
                const double cq = (double)cprev[(int64_t)j * d + i];
                p2 += cq * cq;
                dd += ((double)c - cq) * ((double)c - cq);
                dn += ((double)c - cq) * ((double)c + cq);
                cprev[(int64_t)j * d + i] = c;
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            c2 += __shfl_xor_sync(0xffffffffu, c2, o);
            e2 += __shfl_xor_sync(0xffffffffu, e2, o);
            if (cprev) {
                p2 += __shfl_xor_sync(0xffffffffu, p2, o);
                dd += __shfl_xor_sync(0xffffffffu, dd, o);
                dn += __shfl_xor_sync(0xffffffffu, dn, o);
            }
        }
        if (cprev && lane == 0) {
            const double margin = 1e-12 * (c2 + p2);
            shift[j] = make_float2(__double2float_ru(dn + margin), __double2float_ru(sqrt(dd + margin) * (1.0 + 1e-12)));
        }
        if (lane == 0) {
            const double up = 1.0 + 1e-6;
            const double cn = sqrt(c2) * up, e = sqrt(e2) * up;
            const double g = (cn + e) * up;
            const double h = (e + ((double)eps_acc + (double)eps_s) * g + rho * cn) * up;
            const double z = (double)eps_s * c2 * up;
            cf[4 * pp + o] = __double2float_rn(c2);
            const float hf = __double2float_ru(h), zf1 = __double2float_ru(z);
            cf[4 * pp + 2 + o] = hf;
            zf[2 * pp + o] = zf1;
            // maxima over the centroids (non-negative: bits order like values)
            atomicMax(hz_bits, __float_as_uint(hf));
            atomicMax(hz_bits + 1, __float_as_uint(zf1));
        }
    }
}

// Pruning front: the centroids' positions sorted (by buckets) by ||c_F||^2,
// so that the 32 columns of a chunk have nearly the same norm.  One block:
// the finite keys' range, PF_NB equal buckets, an exclusive scan of their
// counts, then each centroid takes the next position of its bucket (the
// order within a bucket is whatever the atomics give: the survivors' lists
// then differ in order only, which the argmin does not see).
constexpr int PF_NB = 4096;
__global__ void __launch_bounds__(1024) pf_sort_kernel(const float4 *__restrict__ cinfo, int k, int kp,
                                                       int32_t *__restrict__ perm) {
    __shared__ unsigned int cnt[PF_NB];
    __shared__ float red[2][32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const float *cf = reinterpret_cast<const float *>(cinfo);
    auto key = [&](int j) { return cf[4 * (j >> 1) + (j & 1)]; };
    float lo = INFINITY, hi = -INFINITY;
    for (int j = threadIdx.x; j < k; j += blockDim.x) {
        const float v = key(j);
        if (v < INFINITY && v == v) {
            lo = fminf(lo, v);
            hi = fmaxf(hi, v);
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, o));
        hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, o));
    }
    if (lane == 0) {
        red[0][warp] = lo;
        red[1][warp] = hi;
    }
    for (int b = threadIdx.x; b < PF_NB; b += blockDim.x) cnt[b] = 0u;
    __syncthreads();
    lo = red[0][lane];
    hi = red[1][lane];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, o));
        hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, o));
    }
    const float scale = hi > lo ? (float)PF_NB / (hi - lo) : 0.0f;
    auto bucket = [&](float v) {
        if (!(v < INFINITY) || !(v == v)) return PF_NB - 1;
        const int b = (int)((v - lo) * scale);
        return b < 0 ? 0 : (b >= PF_NB ? PF_NB - 1 : b);
    };
    for (int j = threadIdx.x; j < k; j += blockDim.x) atomicAdd(&cnt[bucket(key(j))], 1u);
    __syncthreads();
    // exclusive scan: four buckets a thread, then the warps' and the block's sums
    unsigned int c4[4], s = 0;
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        c4[u] = cnt[4 * threadIdx.x + u];
        s += c4[u];
    }
    unsigned int inc = s;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const unsigned int t = __shfl_up_sync(0xffffffffu, inc, o);
        if (lane >= o) inc += t;
    }
    __shared__ unsigned int wsum[32];
    if (lane == 31) wsum[warp] = inc;
    __syncthreads();
    if (warp == 0) {
        unsigned int w = wsum[lane], wi = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const unsigned int t = __shfl_up_sync(0xffffffffu, wi, o);
            if (lane >= o) wi += t;
        }
        wsum[lane] = wi - w;  // exclusive
    }
    __syncthreads();
    unsigned int run = wsum[warp] + inc - s;
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        cnt[4 * threadIdx.x + u] = run;
        run += c4[u];
    }
    __syncthreads();
    for (int j = threadIdx.x; j < k; j += blockDim.x) perm[atomicAdd(&cnt[bucket(key(j))], 1u)] = j;
    for (int pos = k + threadIdx.x; pos < kp; pos += blockDim.x) perm[pos] = 0;  // padding: a valid index
}

// The sorted operand rows (F bf16 each), records (||c_F||^2, h') and each
// 32-position chunk's smallest ||c_F||^2 (positions past k: +inf).  One warp
// per chunk.
__global__ void pf_gather_kernel(const uint16_t *__restrict__ cs0, const float4 *__restrict__ cinfo0, int k, int kp,
                                 int F, const int32_t *__restrict__ perm, uint16_t *__restrict__ cs,
                                 float4 *__restrict__ cinfo, float *__restrict__ cmin) {
    const int lane = threadIdx.x & 31;
    const int64_t w0 = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const float *cf0 = reinterpret_cast<const float *>(cinfo0);
    float *cf = reinterpret_cast<float *>(cinfo);
    for (int64_t w = w0; w < kp / 32; w += nw) {
        const int pos = (int)(32 * w) + lane;
        const int j = pos < k ? perm[pos] : -1;
        const float cn = j >= 0 ? cf0[4 * (j >> 1) + (j & 1)] : INFINITY;
        const float h = j >= 0 ? cf0[4 * (j >> 1) + 2 + (j & 1)] : 0.0f;
        cf[4 * (pos >> 1) + (pos & 1)] = cn;
        cf[4 * (pos >> 1) + 2 + (pos & 1)] = h;
        float m = cn;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) m = fminf(m, __shfl_xor_sync(0xffffffffu, m, o));
        if (lane == 0) cmin[w] = m;
        // rows of F bf16 (F % 4 == 0): lanes over 8-byte words
        for (int r = 0; r < 32; ++r) {
            const int jr = __shfl_sync(0xffffffffu, j, r);
            if (jr < 0) break;  // warp-uniform: positions past k are last
            const uint2 *src = reinterpret_cast<const uint2 *>(cs0 + (int64_t)jr * F);
            uint2 *dst = reinterpret_cast<uint2 *>(cs + ((int64_t)32 * w + r) * F);
            for (int q = lane; q < F / 4; q += 32) dst[q] = src[q];
        }
    }
}

__global__ void cprep_sq8_kernel(const uint8_t *__restrict__ C, int k, int kp, int d, int dp,
                                 __nv_bfloat16 *__restrict__ cs, int32_t *__restrict__ nc) {
    const int lane = threadIdx.x & 31;
    const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int nw = (gridDim.x * blockDim.x) >> 5;
    for (int j = warp; j < kp; j += nw) {
        if (j >= k) {  // padding records: never the nearest
            if (lane == 0) nc[j] = 0x3fffffff;
            continue;
        }
        int32_t s = 0;
        for (int i = lane; i < d; i += 32) {
            const int32_t v = (int32_t)C[(int64_t)j * d + i] - 128;
            cs[(int64_t)j * dp + i] = __int2bfloat16_rn(v);
            s += v * v;
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
        if (lane == 0) nc[j] = s;
    }
}

// RBQ1 points: sign bits -> e4m3 bytes 2 xbar - 1 (bit 1 -> +1.0 = 0x38, bit 0
// -> -1.0 = 0xB8), row stride dp bytes (columns past d are never read: the
// tensor map's width is d).  One thread per 32-bit code word writes 32 bytes.
__global__ void screen_prep_rbq1_kernel(const uint32_t *__restrict__ codes, int64_t n, int d,
                                        int dp, uint8_t *__restrict__ xs) {
    const int W = (d + 31) >> 5;
    const int64_t total = n * W;
    for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < total;
         t += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = t / W;
        const int w = (int)(t - r * W);
        const uint32_t bits = codes[t];
        uint8_t *dst = xs + r * dp + 32 * w;
        const int nb = min(32, d - 32 * w);
        if (nb == 32 && (dp % 16) == 0) {
            uint4 o[2];
            uint32_t *ow = reinterpret_cast<uint32_t *>(o);
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                uint32_t v = 0;
#pragma unroll
                for (int u = 0; u < 4; ++u) v |= (((bits >> (4 * q + u)) & 1u) ? 0x38u : 0xB8u) << (8 * u);
                ow[q] = v;
            }
            reinterpret_cast<uint4 *>(dst)[0] = o[0];
            reinterpret_cast<uint4 *>(dst)[1] = o[1];
        } else {
            for (int u = 0; u < nb; ++u) dst[u] = ((bits >> u) & 1u) ? 0x38 : 0xB8;
        }
    }
}

// Per-centroid estimator terms -> column-pair records for the tensor
// epilogue: bs[p] = (bd x2, sd x2), qn[p] = (-sum ybar x2, ||c - m||^2 x2);
// columns past k get ||c - m||^2 = +inf (never the nearest).
__global__ void pack_rbq1_pairs_kernel(const Rbq1CInfo *__restrict__ info, int k, int kp,
                                       float4 *__restrict__ bs, float4 *__restrict__ qn) {
    const int pp = blockIdx.x * blockDim.x + threadIdx.x;
    if (2 * pp >= kp) return;
    float b[2], sc[2], q[2], n2[2];
#pragma unroll
    for (int o = 0; o < 2; ++o) {
        const int j = 2 * pp + o;
        if (j < k) {
            const Rbq1CInfo in = info[j];
            b[o] = in.bd;
            sc[o] = in.sd;
            q[o] = -(float)in.sumy;
            n2[o] = in.ny2;
        } else {
            b[o] = 0.0f;
            sc[o] = 0.0f;
            q[o] = 0.0f;
            n2[o] = INFINITY;
        }
    }
    bs[pp] = make_float4(b[0], b[1], sc[0], sc[1]);
    qn[pp] = make_float4(q[0], q[1], n2[0], n2[1]);
}

// ------------------------------------------------------------ fp32 rescoring
template <typename TX>
__device__ __forceinline__ float ldx(const TX *p);
template <>
__device__ __forceinline__ float ldx<float>(const float *p) {
    return __ldg(p);
}
template <>
__device__ __forceinline__ float ldx<uint16_t>(const uint16_t *p) {
    return __uint_as_float(((uint32_t)__ldg(p)) << 16);
}

template <typename TX>
__device__ __forceinline__ float warp_sqdist(const TX *x, const float *c, int d, int lane) {
    float s = 0.0f;
    for (int i = lane; i < d; i += 32) {
        const float t = __fsub_rn(ldx<TX>(x + i), __ldg(c + i));
        s = __fmaf_rn(t, t, s);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    return s;
}

// One warp per listed row: exact fp32 distances to its screen candidates.
template <typename TX>
// (count: the call's counters, [0] rows listed, [2] the screen's abort flag.)
// SKM_FLAG_WARM: thread 0 stamps the workspace's bounds as complete for this
// n, d and k unless the screen gave up.
__global__ void rescore_kernel(const TX *__restrict__ X, int d, const float *__restrict__ C,
                               const int32_t *__restrict__ rows, const int32_t *__restrict__ count,
                               const int32_t *__restrict__ cand, int32_t *__restrict__ assign,
                               int64_t *__restrict__ warm_hdr, int64_t n, int k) {
    const int lane = threadIdx.x & 31;
    const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int64_t cnt = *count;
    if (warm_hdr && blockIdx.x == 0 && threadIdx.x == 0 && count[2] == 0) {
        warm_hdr[1] = n;
        warm_hdr[2] = d;
        warm_hdr[3] = k;
        __threadfence();
        warm_hdr[0] = WARM_MAGIC;
    }
    for (int64_t i = warp; i < cnt; i += nw) {
        const int64_t r = rows[i];
        const int32_t *cr = cand + r * (TCAND + 1);
        const int nc = cr[TCAND];
        float bd = INFINITY;
        int bj = 0x7fffffff;
        for (int t = 0; t < nc; ++t) {
            const int j = cr[t];
            const float dd = warp_sqdist<TX>(X + r * d, C + (int64_t)j * d, d, lane);
            if (dd < bd || (dd == bd && j < bj)) {
                bd = dd;
                bj = j;
            }
        }
        if (lane == 0) assign[r] = bj;
    }
}

// dist[r] = fp32 sum of squared differences to the assigned centroid.
template <typename TX>
__global__ void assigned_dist_kernel(const TX *__restrict__ X, int64_t n, int d,
                                     const float *__restrict__ C, const int32_t *__restrict__ assign,
                                     float *__restrict__ dist) {
    const int lane = threadIdx.x & 31;
    const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    for (int64_t r = warp; r < n; r += nw) {
        const float dd = warp_sqdist<TX>(X + r * d, C + (int64_t)assign[r] * d, d, lane);
        if (lane == 0) dist[r] = dd;
    }
}

__global__ void add_stats_kernel(const int32_t *__restrict__ counters, int64_t *__restrict__ stats) {
    stats[0] += counters[0];
    stats[1] += counters[1];
    stats[2] |= counters[2];
}

// ---------------------------------------------------------- segmented mode
// Centroid tiles of each point tile: the union of its rows' group ranges
// (min and max group over the tile's rows, ids clamped into [0, nseg)).
__global__ void seg_tiles_kernel(const int32_t *__restrict__ group, const int32_t *__restrict__ base, int nseg,
                                 int64_t n, int64_t nrt, int32_t *__restrict__ ct0, int32_t *__restrict__ nct) {
    const int lane = threadIdx.x & 31;
    const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    for (int64_t rt = warp; rt < nrt; rt += nw) {
        int gmin = 0x7fffffff, gmax = -1;
        for (int i = lane; i < BM; i += 32) {
            const int64_t r = rt * BM + i;
            if (r < n) {
                int g = group[r];
                g = g < 0 ? 0 : (g >= nseg ? nseg - 1 : g);
                gmin = min(gmin, g);
                gmax = max(gmax, g);
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            gmin = min(gmin, __shfl_xor_sync(0xffffffffu, gmin, o));
            gmax = max(gmax, __shfl_xor_sync(0xffffffffu, gmax, o));
        }
        if (lane == 0) {
            const int lo = base[gmin], hi = base[gmax + 1];
            const int t0 = lo / BN;
            const int t1 = hi > lo ? (hi + BN - 1) / BN : t0 + 1;
            ct0[rt] = t0;
            nct[rt] = t1 - t0;
        }
    }
}

// Segmented fallback: one warp per listed row scans its own group's range in
// fp32 (direct differences), ties to the lowest index.
template <typename TX>
__global__ void seg_rows_exact_kernel(const TX *__restrict__ X, int d, const float *__restrict__ C,
                                      const int32_t *__restrict__ rows, const int32_t *__restrict__ count,
                                      const int32_t *__restrict__ group, const int32_t *__restrict__ base,
                                      int nseg, int32_t *__restrict__ assign) {
    const int lane = threadIdx.x & 31;
    const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int64_t cnt = *count;
    for (int64_t t = warp; t < cnt; t += nw) {
        const int64_t r = rows[t];
        int g = group[r];
        g = g < 0 ? 0 : (g >= nseg ? nseg - 1 : g);
        const int cb = base[g], ce = base[g + 1];
        float bd = INFINITY;
        int bj = cb;
        for (int j = cb; j < ce; ++j) {
            const float dd = warp_sqdist<TX>(X + r * d, C + (int64_t)j * d, d, lane);
            if (dd < bd) {
                bd = dd;
                bj = j;
            }
        }
        if (lane == 0) assign[r] = bj;
    }
}

// ------------------------------------------------------------------ host side
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

// 2D map over [rows][cols] of 2-byte (bf16) or 1-byte (e4m3, as uint8)
// elements with row stride `stride_elems`; box = box_rows x 128 bytes.
int make_map(CUtensorMap *m, const void *ptr, int64_t rows, int cols, int stride_elems,
             int box_rows, int elem_bytes) {
    auto fn = encode_fn();
    if (!fn) return set_error(SKM_ERR_CUDA, "cuTensorMapEncodeTiled entry point not found");
    cuuint64_t gdim[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t gstride[1] = {(cuuint64_t)stride_elems * elem_bytes};
    cuuint32_t box[2] = {(cuuint32_t)(128 / elem_bytes), (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    const CUtensorMapDataType dt =
        elem_bytes == 2 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_UINT8;
    CUresult r = fn(m, dt, 2, const_cast<void *>(ptr), gdim, gstride, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return set_error(SKM_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", (int)r);
    return SKM_OK;
}

int device_sms() {
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    return sms > 0 ? sms : 148;
}

template <int MODE, bool SEG, bool PK>
int launch_tc_kind(const void *xs, int64_t n, int dp, int d, const void *cs, int k, const TcParams &p0,
                   cudaStream_t st, int dpb);

// packed: xs is the 1-bit codes [n][ceil(d/32)] or the LVQ4 nibble words
// [n][ceil(d/8)] (MODE_RBQ1 / MODE_LVQ4)
// (dpb: the centroid operand's row stride when it differs from dp)
template <int MODE>
int launch_tc(const void *xs, int64_t n, int dp, int d, const void *cs, int k, const TcParams &p0,
              cudaStream_t st, bool packed = false, int dpb = -1) {
    if (dpb < 0) dpb = dp;
    if constexpr (MODE == MODE_RBQ1 || MODE == MODE_LVQ4) {
        if (packed) {
            if (p0.seg_group) return launch_tc_kind<MODE, true, true>(xs, n, dp, d, cs, k, p0, st, dpb);
            return launch_tc_kind<MODE, false, true>(xs, n, dp, d, cs, k, p0, st, dpb);
        }
    }
    if constexpr (MODE != MODE_PFRONT)
        if (p0.seg_group) return launch_tc_kind<MODE, true, false>(xs, n, dp, d, cs, k, p0, st, dpb);
    return launch_tc_kind<MODE, false, false>(xs, n, dp, d, cs, k, p0, st, dpb);
}

// One persistent CTA per SM (at most one point tile per CTA when there are
// fewer tiles than SMs).
template <int MODE, bool SEG, bool PK>
int launch_tc_kind(const void *xs, int64_t n, int dp, int d, const void *cs, int k, const TcParams &p0,
                   cudaStream_t st, int dpb) {
    constexpr int NH = TC_NH[MODE];
    constexpr int NS = TC_NS[MODE];
    constexpr size_t SMEM = tc_smem_bytes<MODE, NH, NS>();
    static_assert(SMEM <= 227 * 1024, "shared memory per CTA");
    auto kern = tc_assign_kernel<MODE, NH, SEG, NS, PK>;
    const int segi = SEG ? 1 : 0, pki = PK ? 1 : 0;
    // the dynamic shared memory attribute, set once per device
    constexpr int MAXDEV = 64;
    static std::mutex mu;
    static bool attr_set[6][2][2][MAXDEV] = {};
    int dev = 0;
    SKM_CUDA_TRY(cudaGetDevice(&dev));
    {
        std::lock_guard<std::mutex> lock(mu);
        if (dev >= MAXDEV || !attr_set[MODE][segi][pki][dev]) {
            SKM_CUDA_TRY(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SMEM));
            if (dev < MAXDEV) attr_set[MODE][segi][pki][dev] = true;
        }
    }
    CUtensorMap ma, mb;
    const int eb = f8_mode<MODE>() ? 1 : 2;
    // GEMM mode: the A and B parts are stacked (rows [part][n], [part][k])
    const int parts = MODE == MODE_GEMM ? 3 : 1;
    // PK: the A slices come from the CTAs' expansion scratch
    int grid = (int)std::min<int64_t>(device_sms(), cdiv(n, BM));
    if (PK) {
        grid = std::min(grid, PK_MAX_CTAS);
        SKM_TRY(make_map(&ma, p0.pk_scratch, (int64_t)grid * NS * 2 * BM, d, dp, BM, eb));
    } else {
        SKM_TRY(make_map(&ma, xs, parts * n, d, dp, BM, eb));
    }
    SKM_TRY(make_map(&mb, cs, (int64_t)parts * k, d, dpb, BN, eb));
    TcParams p = p0;
    p.n = n;
    p.nrt = cdiv(n, BM);
    p.k = k;
    p.nct = (int)cdiv(k, BN);
    p.nkc = (int)cdiv(d, 128 / eb);
    p.inject_wait_ns = fault_take(SKM_FAULT_WAIT) ? 1000000ull : 0ull;  // 1 ms
    tc_timer_mark(st, 0);
    kern<<<grid, tc_threads<NH, PK>(), SMEM, st>>>(ma, mb, p);
    tc_timer_mark(st, 1);
    SKM_CUDA_TRY(launched());
    return SKM_OK;
}

int grid_warps(int64_t items) {
    int64_t b = (items * 32 + 255) / 256;
    const int64_t cap = 152LL * 8;
    return (int)(b < 1 ? 1 : (b > cap ? cap : b));
}

inline int round8(int d) { return (d + 7) & ~7; }
inline int round16(int d) { return (d + 15) & ~15; }
// 1-bit codes the tensor-core kernel can read packed (rows a multiple of 16
// bytes, 16-byte aligned); it does so unless the caller supplies the e4m3
// screening copy
inline bool rbq1_packed(int d, const void *x) {
    return d <= TC_RBQ1_MAX_D && ((d + 31) / 32) % 4 == 0 && ((uintptr_t)x & 15) == 0;
}
// the same for LVQ4 nibble words (then round16(d) <= 8 ceil(d/8): every word
// a converter reads lies inside the row)
inline bool lvq4_packed(int d, const void *x) {
    return d <= TC_LVQ4_MAX_D && ((d + 7) / 8) % 4 == 0 && ((uintptr_t)x & 15) == 0;
}

}  // namespace

// ------------------------------------------------------------- public (internal)
size_t tc_screen_bytes(int repr, int64_t n, int d, const void *x) {
    Carver cv(nullptr, 0);
    const int dp = round8(d);
    switch (repr) {
    case SKM_REPR_F32:
        cv.take<uint16_t>((size_t)n * dp);
        cv.take<float2>(n);
        cv.take<float>(1);
        break;
    case SKM_REPR_SQ8:
        if (d > TC_SQ8_MAX_D) return 0;
        cv.take<uint16_t>((size_t)n * dp);
        cv.take<int32_t>(n);
        break;
    case SKM_REPR_BF16:
        if (d % 8 != 0 || ((uintptr_t)x & 15) != 0) cv.take<uint16_t>((size_t)n * dp);
        cv.take<float2>(n);
        cv.take<float>(1);
        break;
    case SKM_REPR_RBQ1:
        if (d > TC_RBQ1_MAX_D) return 0;
        cv.take<uint8_t>((size_t)n * round16(d));
        break;
    case SKM_REPR_LVQ4:
        if (d > TC_LVQ4_MAX_D) return 0;
        cv.take<uint8_t>((size_t)n * round16(d));
        break;
    default:
        return 0;
    }
    return cv.off;
}

struct ScreenView {
    const void *xs = nullptr;
    const float2 *xinfo = nullptr;
    const float *rho_max = nullptr;  // max over points of ||x~ - x|| / ||x~||
    const int32_t *nx = nullptr;
    bool packed = false;  // RBQ1: xs is the packed codes
};

static ScreenView screen_view(int repr, int64_t n, int d, const void *x, const void *screen) {
    ScreenView v;
    Carver cv(const_cast<void *>(screen), SIZE_MAX);
    const int dp = round8(d);
    switch (repr) {
    case SKM_REPR_F32:
        v.xs = cv.take<uint16_t>((size_t)n * dp);
        v.xinfo = cv.take<float2>(n);
        v.rho_max = cv.take<float>(1);
        break;
    case SKM_REPR_SQ8:
        v.xs = cv.take<uint16_t>((size_t)n * dp);
        v.nx = cv.take<int32_t>(n);
        break;
    case SKM_REPR_BF16:
        if (d % 8 != 0 || ((uintptr_t)x & 15) != 0)
            v.xs = cv.take<uint16_t>((size_t)n * dp);
        else
            v.xs = x;
        v.xinfo = cv.take<float2>(n);
        v.rho_max = cv.take<float>(1);
        break;
    case SKM_REPR_RBQ1:
        if (!screen) {  // no copy: the codes are read packed
            v.xs = x;
            v.packed = true;
            break;
        }
        v.xs = cv.take<uint8_t>((size_t)n * round16(d));
        break;
    case SKM_REPR_LVQ4:
        if (!screen) {  // no copy: the codes are read packed
            v.xs = x;
            v.packed = true;
            break;
        }
        v.xs = cv.take<uint8_t>((size_t)n * round16(d));
        break;
    }
    return v;
}

int tc_screen_prep(const skm_data *x, void *screen, cudaStream_t st) {
    const int64_t n = x->n;
    const int d = x->d, dp = round8(d);
    ScreenView v = screen_view(x->repr, n, d, x->x, screen);
    const int g = grid_warps(n);
    if (v.rho_max) SKM_CUDA_TRY(cudaMemsetAsync((void *)v.rho_max, 0, sizeof(float), st));
    switch (x->repr) {
    case SKM_REPR_F32:
        screen_prep_f32_kernel<<<g, 256, 0, st>>>(static_cast<const float *>(x->x), n, d, dp,
                                                  (__nv_bfloat16 *)v.xs, (float2 *)v.xinfo,
                                                  (unsigned int *)v.rho_max);
        break;
    case SKM_REPR_SQ8:
        screen_prep_sq8_kernel<<<g, 256, 0, st>>>(static_cast<const uint8_t *>(x->x), n, d, dp,
                                                  (__nv_bfloat16 *)v.xs, (int32_t *)v.nx);
        break;
    case SKM_REPR_BF16:
        screen_prep_bf16_kernel<<<g, 256, 0, st>>>(static_cast<const uint16_t *>(x->x), n, d, dp,
                                                   v.xs == x->x ? nullptr : (uint16_t *)v.xs,
                                                   (float2 *)v.xinfo);
        break;
    case SKM_REPR_RBQ1: {
        int64_t blocks = (n * words_of(d) + 255) / 256;
        if (blocks > 152 * 8) blocks = 152 * 8;
        screen_prep_rbq1_kernel<<<(int)blocks, 256, 0, st>>>(static_cast<const uint32_t *>(x->x), n,
                                                             d, round16(d), (uint8_t *)v.xs);
        break;
    }
    case SKM_REPR_LVQ4:
        SKM_CUDA_TRY(launch_lvq4_expand(static_cast<const uint32_t *>(x->x), n, d, (uint8_t *)v.xs, round16(d), st));
        return SKM_OK;
    default:
        return set_error(SKM_ERR_INVALID_ARG, "no screening copy for repr %d", x->repr);
    }
    SKM_CUDA_TRY(launched());
    return SKM_OK;
}

bool tc_reads_packed(int repr, int d, const void *x) {
    return (repr == SKM_REPR_RBQ1 && rbq1_packed(d, x)) || (repr == SKM_REPR_LVQ4 && lvq4_packed(d, x));
}

void tc_plan(int repr, int64_t n, int d, int k, const void *x, const void *screen, bool warm, Carver &cv,
             TcAssignBufs &b) {
    b.stats = cv.take<int64_t>(4);
    b.counters = cv.take<int32_t>(8);  // [4], [5]: SCREEN max h', max z (float bits)
    if (repr < 0) return;  // statistics only
    const int dp = round8(d);
    const bool dense = repr == SKM_REPR_F32 || repr == SKM_REPR_BF16 ||
                       (repr == SKM_REPR_RBQ1 && d <= TC_RBQ1_MAX_D) ||
                       (repr == SKM_REPR_LVQ4 && d <= TC_LVQ4_MAX_D) ||
                       (repr == SKM_REPR_SQ8 && d <= TC_SQ8_MAX_D);
    if (!dense) return;
    const bool pk = !screen && ((repr == SKM_REPR_RBQ1 && rbq1_packed(d, x)) ||
                                (repr == SKM_REPR_LVQ4 && lvq4_packed(d, x)));
    if (!screen && !pk) {
        const size_t sb = tc_screen_bytes(repr, n, d, x);
        b.screen = cv.take<uint8_t>(sb);
    }
    const size_t kp = (size_t)cdiv(k, BN) * BN;  // per-centroid records padded to whole tiles
    if (repr == SKM_REPR_LVQ4) {
        if (pk)  // read packed: per-CTA expansion slots (two per job stream)
            b.pk_scratch = cv.take<uint8_t>((size_t)std::min<int64_t>(PK_MAX_CTAS, cdiv(n, BM)) * TC_NS[MODE_LVQ4] *
                                            2 * BM * round16(d));
        b.cs = reinterpret_cast<uint16_t *>(cv.take<uint8_t>((size_t)k * round16(d)));
        b.linfo = cv.take<float4>(k);
        b.rpair_bs = cv.take<float4>(kp / 2);
        b.rpair_qn = cv.take<float4>(kp / 2);
        return;
    }
    if (repr == SKM_REPR_RBQ1) {
        if (pk)  // read packed: per-CTA expansion slots (two per job stream)
            b.pk_scratch = cv.take<uint8_t>((size_t)std::min<int64_t>(PK_MAX_CTAS, cdiv(n, BM)) * TC_NS[MODE_RBQ1] *
                                            2 * BM * round16(d));
        b.cs = reinterpret_cast<uint16_t *>(cv.take<uint8_t>((size_t)k * round16(d)));
        b.rinfo = cv.take<Rbq1CInfo>(k);
        b.rpair_bs = cv.take<float4>(kp / 2);
        b.rpair_qn = cv.take<float4>(kp / 2);
        return;
    }
    b.cs = cv.take<uint16_t>((size_t)k * dp);
    if (repr == SKM_REPR_SQ8) {
        b.nc = cv.take<int32_t>(kp);
    } else {
        if (warm) {
            b.warm_hdr = cv.take<int64_t>(4);
            b.warm_row = cv.take<int2>(n);
            b.warm_cprev = cv.take<float>((size_t)k * d);
            b.warm_shift = cv.take<float2>(k);
        }
        b.cinfo = cv.take<float4>(kp / 2);
        b.cinfoz = cv.take<float2>(kp / 2);
        b.cand = cv.take<int32_t>((size_t)n * (TCAND + 1));
        b.resc_rows = cv.take<int32_t>(n);
        b.fall_rows = cv.take<int32_t>(n);
        b.fall_keys = cv.take<unsigned long long>(n);
    }
}

bool tc_pfront_ok(int repr, int d, const void *x) {
    return repr == SKM_REPR_BF16 && d >= 2 * PF_DIMS && d <= 1024 && d % 8 == 0 && ((uintptr_t)x & 15) == 0;
}

void tc_plan_pfront(int64_t n, int d, int k, bool warm, Carver &cv, TcAssignBufs &b) {
    const size_t kp = (size_t)cdiv(k, BN) * BN;
    b.pf_seed = cv.take<int32_t>(n);
    if (warm) {  // bounds kept across calls
        b.pf_whdr = cv.take<int64_t>(8);
        b.pf_cgen = cv.take<int64_t>(1);
        b.pf_wrow = cv.take<int2>(n);
        b.pf_xn = cv.take<float2>(n);
        b.pf_cprev = cv.take<float>((size_t)k * d);
        b.pf_shift = cv.take<float2>(k);
    }
    b.cs = cv.take<uint16_t>((size_t)k * PF_DIMS);  // sorted by ||c_F||^2
    b.cinfo = cv.take<float4>(kp / 2);
    b.cinfoz = cv.take<float2>(kp / 2);
    b.pf_cs0 = cv.take<uint16_t>((size_t)k * PF_DIMS);  // centroid order
    b.pf_cinfo0 = cv.take<float4>(kp / 2);
    b.pf_perm = cv.take<int32_t>(kp);
    b.pf_cmin = cv.take<float>(kp / 32);
    b.pf_thr = cv.take<float2>(n);
    b.pf_cand = cv.take<uint16_t>((size_t)n * PF_CAP);
    b.pf_cnt = cv.take<int32_t>(n);
    b.resc_rows = cv.take<int32_t>(n);
    b.fall_rows = cv.take<int32_t>(n);
}

// Exact dimension pruning with a tensor-core front (Section 3.1
// "SuperKMeans": a GEMM over the front dimensions, then pruning on the
// survivors).  The pruned distance of the method is the fp32 sum of 32-
// dimension block partials, in order, of (x_i - c_i)^2; a centroid may be
// dropped once a lower bound of it exceeds the row's seed distance (the
// distance to its previous centroid), which every argmin and tie is below.
//   1. centroids: bf16 operand and bound records over the first PF_DIMS
//      dimensions (the screen's interval terms, with prefix norms);
//   2. rows: the seed distance and the threshold on s~ over the front
//      (k_prune.cu);
//   3. tcgen05 over the front: survivors listed per row; a row whose one
//      survivor is its seed is decided;
//   4. CUDA cores: the listed rows' survivors evaluated block by block, and
//      rows whose lists overflowed pruned over all k.
// The result is the same as the CUDA-core pruning kernels' bit for bit.
// End of a front call: the call's list counts into the pruning statistics
// ([4] finished rows, [5] rows pruned over all k; cumulative in skm_fit) and,
// with kept bounds (hdr), the stamp when no wait gave up (every row's bound
// was then written).
__global__ void pf_done_kernel(int64_t *__restrict__ hdr, const int32_t *__restrict__ counters,
                               unsigned long long *__restrict__ ctr, int64_t n, int d, int k,
                               const int64_t *__restrict__ cgen) {
    ctr[4] += (unsigned long long)counters[0];
    ctr[5] += (unsigned long long)counters[1];
    if (hdr && counters[2] == 0) {
        hdr[1] = n;
        hdr[2] = d;
        hdr[3] = k;
        hdr[4] = *cgen;  // the bounds are against the centroids of this generation
        __threadfence();
        hdr[0] = WARM_MAGIC;
    }
}

// A call on centroids prepared by another workspace's call this step
// (shared): this workspace's bounds apply when its stamp names these n, d, k
// and the generation the shared previous centroids had before that
// preparation advanced it.
__global__ void pf_stamp_kernel(int64_t *__restrict__ hdr, int64_t n, int d, int k,
                                const int64_t *__restrict__ cgen, int32_t *__restrict__ warm_ok) {
    *warm_ok = hdr[0] == WARM_MAGIC && hdr[1] == n && hdr[2] == d && hdr[3] == k && hdr[4] == *cgen - 1;
    hdr[0] = 0;
}

int tc_assign_pfront(const skm_data *x, const float *C, int k, const int32_t *prev, int32_t *assign, float *dist,
                     TcAssignBufs &b, unsigned long long *ctr, cudaStream_t st, const TcAssignBufs *sh) {
    // SKM_FLAG_WARM: bounds kept across calls (the previous call's state applies
    // when its stamp matches; distances wanted: exact seed distances this call).
    // sh: the centroid side (operand, records, sort, moves) was prepared this
    // step by an earlier call in the workspace sh, on the same centroids.
    const bool warm = (x->flags & SKM_FLAG_WARM) && b.pf_whdr && (!sh || sh->pf_cgen);
    const TcAssignBufs &cb = sh ? *sh : b;  // the centroid side
    const int64_t n = x->n;
    const int d = x->d;
    constexpr int F = PF_DIMS;
    const int kp = (int)(cdiv(k, BN) * BN);
    SKM_CUDA_TRY(cudaMemsetAsync(b.counters, 0, sizeof(int32_t) * 8, st));
    if (!sh) {
        const float eps_acc = (float)(((F / BK) * (BK / 16) + 4) * 0x1p-18);
        const float eps_s = 0x1p-21f;
        // bf16 points are their own operand: no residual term (counters[7] = 0.0f)
        cprep_f32_kernel<<<grid_warps(kp), 256, 0, st>>>(C, k, kp, d, F, F, eps_acc, eps_s,
                                                         reinterpret_cast<const float *>(b.counters + 7),
                                                         (__nv_bfloat16 *)b.pf_cs0, b.pf_cinfo0, b.cinfoz,
                                                         reinterpret_cast<unsigned int *>(b.counters + 4),
                                                         warm ? b.pf_cprev : nullptr, b.pf_shift, b.pf_whdr, n,
                                                         b.counters + 6, warm ? b.pf_cgen : nullptr);
        SKM_CUDA_TRY(launched());
        // columns sorted by ||c_F||^2 (a chunk's columns then share a tight bound)
        pf_sort_kernel<<<1, 1024, 0, st>>>(b.pf_cinfo0, k, kp, b.pf_perm);
        SKM_CUDA_TRY(launched());
        pf_gather_kernel<<<std::max(1, std::min(kp / 32 / 8, 152 * 8)), 256, 0, st>>>(b.pf_cs0, b.pf_cinfo0, k, kp, F,
                                                                                      b.pf_perm, b.cs, b.cinfo,
                                                                                      b.pf_cmin);
        SKM_CUDA_TRY(launched());
    } else if (warm) {
        pf_stamp_kernel<<<1, 1, 0, st>>>(b.pf_whdr, n, d, k, sh->pf_cgen, b.counters + 6);
        SKM_CUDA_TRY(launched());
    }
    const uint16_t *X = static_cast<const uint16_t *>(x->x);
    PfRows rows;
    rows.thr = b.pf_thr;
    rows.seed = b.pf_seed;
    if (warm) {
        rows.xn = b.pf_xn;
        rows.wrow = b.pf_wrow;
        rows.shift = cb.pf_shift;
        rows.warm_ok = b.counters + 6;
    }
    SKM_CUDA_TRY(launch_prune_front_prep(X, n, d, F, C, k, prev, reinterpret_cast<const float *>(cb.counters + 4),
                                         rows, dist != nullptr, ctr, st));
    TcParams p{};
    p.cinfo = cb.cinfo;
    p.counters = b.counters;
    p.assign = assign;
    p.dist = dist;
    p.resc_rows = b.resc_rows;
    p.fall_rows = b.fall_rows;
    p.pf_thr = b.pf_thr;
    p.pf_cand = b.pf_cand;
    p.pf_cnt = b.pf_cnt;
    p.pf_seed = b.pf_seed;
    p.pf_ctr = ctr;
    p.pf_wrow = rows.wrow;
    p.pf_perm = cb.pf_perm;
    p.pf_cmin = cb.pf_cmin;
    SKM_TRY(launch_tc<MODE_PFRONT>(X, n, d, F, cb.cs, k, p, st, false, F));
    constexpr int nsub = TC_NH[MODE_PFRONT] / TC_NS[MODE_PFRONT];
    SKM_CUDA_TRY(launch_prune_finish(X, d, C, b.pf_thr, b.pf_cand, b.pf_cnt, PF_CAP, nsub, cb.pf_perm, b.resc_rows,
                                     b.counters, assign, dist, rows.wrow, ctr, st));
    SKM_CUDA_TRY(launch_prune_rows_cta(X, d, C, k, rows, b.fall_rows, b.counters + 1, assign, dist, ctr + 6, st));
    add_stats_kernel<<<1, 1, 0, st>>>(b.counters, b.stats);
    SKM_CUDA_TRY(launched());
    pf_done_kernel<<<1, 1, 0, st>>>(warm ? b.pf_whdr : nullptr, b.counters, ctr, n, d, k, cb.pf_cgen);
    SKM_CUDA_TRY(launched());
    return SKM_OK;
}

int tc_init_stats(TcAssignBufs &b, cudaStream_t st) {
    SKM_CUDA_TRY(cudaMemsetAsync(b.stats, 0, sizeof(int64_t) * 4, st));
    return SKM_OK;
}

// point tiles' centroid-tile ranges for a segmented call (none otherwise)
static int seg_setup(const TcSeg *seg, int64_t n, TcParams &p, cudaStream_t st) {
    if (!seg) return SKM_OK;
    const int64_t nrt = cdiv(n, BM);
    int64_t blocks = (nrt * 32 + 255) / 256;
    if (blocks > 152 * 8) blocks = 152 * 8;
    seg_tiles_kernel<<<(int)(blocks < 1 ? 1 : blocks), 256, 0, st>>>(seg->group, seg->base, seg->nseg, n, nrt,
                                                                    seg->ct0, seg->nct);
    SKM_CUDA_TRY(launched());
    p.seg_ct0 = seg->ct0;
    p.seg_nct = seg->nct;
    p.seg_group = seg->group;
    p.seg_base = seg->base;
    p.nseg = seg->nseg;
    return SKM_OK;
}

int tc_assign_float(const skm_data *x, const float *C, int k, int32_t *assign, float *dist,
                    TcAssignBufs &b, cudaStream_t st, const TcSeg *seg) {
    const int64_t n = x->n;
    const int d = x->d, dp = round8(d);
    const bool bf16 = x->repr == SKM_REPR_BF16;
    const void *screen = x->screen;
    if (!screen) {
        skm_data tmp = *x;
        SKM_TRY(tc_screen_prep(&tmp, b.screen, st));
        screen = b.screen;
    }
    ScreenView v = screen_view(x->repr, n, d, x->x, screen);
    const int nkc = (int)cdiv(d, BK);
    const float eps_acc = (float)((nkc * (BK / 16) + 4) * 0x1p-18);
    const float eps_s = 0x1p-21f;
    const int kp = (int)(cdiv(k, BN) * BN);
    SKM_CUDA_TRY(cudaMemsetAsync(b.counters, 0, sizeof(int32_t) * 8, st));
    // SKM_FLAG_WARM (not in segmented calls): bounds carried between calls
    const bool warm = !seg && (x->flags & SKM_FLAG_WARM) && b.warm_hdr;
    cprep_f32_kernel<<<grid_warps(kp), 256, 0, st>>>(C, k, kp, d, dp, d, eps_acc, eps_s, v.rho_max,
                                                     (__nv_bfloat16 *)b.cs, b.cinfo, b.cinfoz,
                                                     reinterpret_cast<unsigned int *>(b.counters + 4),
                                                     warm ? b.warm_cprev : nullptr, b.warm_shift, b.warm_hdr, n,
                                                     b.counters + 6, nullptr);
    SKM_CUDA_TRY(launched());
    TcParams p{};
    p.cinfo = b.cinfo;
    p.hz = reinterpret_cast<const float *>(b.counters + 4);
    p.cinfoz = b.cinfoz;
    p.xinfo = v.xinfo;
    p.cand = b.cand;
    p.resc_rows = b.resc_rows;
    p.fall_rows = b.fall_rows;
    p.counters = b.counters;
    p.assign = assign;
    if (warm) {
        p.warm_row = b.warm_row;
        p.warm_shift = b.warm_shift;
        p.warm_ok = b.counters + 6;
    }
    SKM_TRY(seg_setup(seg, n, p, st));
    SKM_TRY(launch_tc<MODE_SCREEN>(v.xs, n, dp, d, b.cs, k, p, st));
    int64_t *hdr = warm ? b.warm_hdr : nullptr;
    const int gw = grid_warps(n);
    if (bf16) {
        const uint16_t *X = static_cast<const uint16_t *>(x->x);
        rescore_kernel<uint16_t><<<gw, 256, 0, st>>>(X, d, C, b.resc_rows, b.counters, b.cand, assign, hdr, n, k);
        SKM_CUDA_TRY(launched());
        if (seg) {
            seg_rows_exact_kernel<uint16_t><<<gw, 256, 0, st>>>(X, d, C, b.fall_rows, b.counters + 1, seg->group,
                                                                seg->base, seg->nseg, assign);
            SKM_CUDA_TRY(launched());
        } else {
            SKM_CUDA_TRY(launch_assign_exact_rows(X, 1, b.fall_rows, b.counters + 1, n, d, C, k, assign,
                                                  nullptr, b.fall_keys, st));
        }
        if (dist) {
            assigned_dist_kernel<uint16_t><<<gw, 256, 0, st>>>(X, n, d, C, assign, dist);
            SKM_CUDA_TRY(launched());
        }
    } else {
        const float *X = static_cast<const float *>(x->x);
        rescore_kernel<float><<<gw, 256, 0, st>>>(X, d, C, b.resc_rows, b.counters, b.cand, assign, hdr, n, k);
        SKM_CUDA_TRY(launched());
        if (seg) {
            seg_rows_exact_kernel<float><<<gw, 256, 0, st>>>(X, d, C, b.fall_rows, b.counters + 1, seg->group,
                                                             seg->base, seg->nseg, assign);
            SKM_CUDA_TRY(launched());
        } else {
            SKM_CUDA_TRY(launch_assign_exact_rows(X, 0, b.fall_rows, b.counters + 1, n, d, C, k, assign,
                                                  nullptr, b.fall_keys, st));
        }
        if (dist) {
            assigned_dist_kernel<float><<<gw, 256, 0, st>>>(X, n, d, C, assign, dist);
            SKM_CUDA_TRY(launched());
        }
    }
    add_stats_kernel<<<1, 1, 0, st>>>(b.counters, b.stats);
    SKM_CUDA_TRY(launched());
    return SKM_OK;
}

int tc_assign_sq8(const skm_data *x, const uint8_t *C, int k, int32_t *nx_plain,
                  int32_t *nc_plain, int32_t *assign, float *dist, TcAssignBufs &b,
                  cudaStream_t st, const TcSeg *seg) {
    const int64_t n = x->n;
    const int d = x->d, dp = round8(d);
    if (d > TC_SQ8_MAX_D) {  // the bf16 accumulation is exact only up to d = 1024
        if (seg) return set_error(SKM_ERR_UNSUPPORTED, "segmented SQ8 assignment needs d <= %d", TC_SQ8_MAX_D);
        const uint8_t *X = static_cast<const uint8_t *>(x->x);
        SKM_CUDA_TRY(launch_row_sqnorm_u8(X, n, d, nx_plain, st));
        SKM_CUDA_TRY(launch_row_sqnorm_u8(C, k, d, nc_plain, st));
        SKM_CUDA_TRY(launch_assign_sq8_simt(X, n, d, C, k, nx_plain, nc_plain, assign, dist, st));
        return SKM_OK;
    }
    const void *screen = x->screen;
    if (!screen) {
        skm_data tmp = *x;
        SKM_TRY(tc_screen_prep(&tmp, b.screen, st));
        screen = b.screen;
    }
    ScreenView v = screen_view(x->repr, n, d, x->x, screen);
    const int kp = (int)(cdiv(k, BN) * BN);
    cprep_sq8_kernel<<<grid_warps(kp), 256, 0, st>>>(C, k, kp, d, dp, (__nv_bfloat16 *)b.cs, b.nc);
    SKM_CUDA_TRY(launched());
    SKM_CUDA_TRY(cudaMemsetAsync(b.counters, 0, sizeof(int32_t) * 4, st));
    TcParams p{};
    p.counters = b.counters;
    p.assign = assign;
    p.nx = v.nx;
    p.nc = b.nc;
    p.dist = dist;
    SKM_TRY(seg_setup(seg, n, p, st));
    SKM_TRY(launch_tc<MODE_SQ8>(v.xs, n, dp, d, b.cs, k, p, st));
    add_stats_kernel<<<1, 1, 0, st>>>(b.counters, b.stats);
    SKM_CUDA_TRY(launched());
    return SKM_OK;
}

int tc_assign_rbq1(const skm_data *x, const float *C, int k, int32_t *assign, float *dist,
                   TcAssignBufs &b, cudaStream_t st, const TcSeg *seg) {
    const int64_t n = x->n;
    const int d = x->d, dp = round16(d);
    const void *screen = x->screen;
    // without a caller copy the codes are read packed where their layout allows
    if (!screen && !rbq1_packed(d, x->x)) {
        skm_data tmp = *x;
        SKM_TRY(tc_screen_prep(&tmp, b.screen, st));
        screen = b.screen;
    }
    ScreenView v = screen_view(x->repr, n, d, x->x, screen);
    const int kp = (int)(cdiv(k, BN) * BN);
    if (x->flags & SKM_FLAG_SYMMETRIC)
        SKM_CUDA_TRY(launch_rbq1_cprep_sym(C, k, d, x->m, reinterpret_cast<uint8_t *>(b.cs), dp, nullptr, b.rinfo,
                                           st));
    else
        SKM_CUDA_TRY(launch_rbq1_cprep_tc(C, k, d, x->m, reinterpret_cast<uint8_t *>(b.cs), dp, b.rinfo,
                                          st));
    pack_rbq1_pairs_kernel<<<(kp / 2 + 255) / 256, 256, 0, st>>>(b.rinfo, k, kp, b.rpair_bs,
                                                                 b.rpair_qn);
    SKM_CUDA_TRY(launched());
    SKM_CUDA_TRY(cudaMemsetAsync(b.counters, 0, sizeof(int32_t) * 4, st));
    TcParams p{};
    p.counters = b.counters;
    p.assign = assign;
    p.dist = dist;
    p.rinfo = b.rpair_bs;
    p.rinfoq = b.rpair_qn;
    p.nx2 = x->nx2;
    p.F = x->F;
    p.popx = x->popx;
    p.d = d;
    if (v.packed) {
        p.pk_codes = static_cast<const uint32_t *>(x->x);
        p.pk_scratch = b.pk_scratch;
        p.pk_words = words_of(d);
        p.pk_dp = dp;
    }
    SKM_TRY(seg_setup(seg, n, p, st));
    SKM_TRY(launch_tc<MODE_RBQ1>(v.xs, n, dp, d, b.cs, k, p, st, v.packed));
    add_stats_kernel<<<1, 1, 0, st>>>(b.counters, b.stats);
    SKM_CUDA_TRY(launched());
    return SKM_OK;
}

int tc_assign_lvq4(const skm_data *x, const float *C, int k, int32_t *assign, float *dist,
                   TcAssignBufs &b, cudaStream_t st, const TcSeg *seg) {
    const int64_t n = x->n;
    const int d = x->d, dp = round16(d);
    const void *screen = x->screen;
    // without a caller copy the codes are read packed where their layout allows
    if (!screen && !lvq4_packed(d, x->x)) {
        SKM_TRY(tc_screen_prep(x, b.screen, st));
        screen = b.screen;
    }
    ScreenView v = screen_view(x->repr, n, d, x->x, screen);
    const int kp = (int)(cdiv(k, BN) * BN);
    SKM_CUDA_TRY(launch_lvq4_cprep(C, k, d, reinterpret_cast<uint8_t *>(b.cs), dp, nullptr, b.linfo, st));
    SKM_CUDA_TRY(launch_lvq4_pack_pairs(b.linfo, k, kp, b.rpair_bs, b.rpair_qn, st));
    SKM_CUDA_TRY(cudaMemsetAsync(b.counters, 0, sizeof(int32_t) * 4, st));
    TcParams p{};
    p.counters = b.counters;
    p.assign = assign;
    p.dist = dist;
    p.rinfo = b.rpair_bs;
    p.rinfoq = b.rpair_qn;
    p.lvq = reinterpret_cast<const float4 *>(x->lvq);
    p.d = d;
    if (v.packed) {
        p.pk_codes = static_cast<const uint32_t *>(x->x);
        p.pk_scratch = b.pk_scratch;
        p.pk_words = lvq4_words(d);
        p.pk_dp = dp;
    }
    SKM_TRY(seg_setup(seg, n, p, st));
    SKM_TRY(launch_tc<MODE_LVQ4>(v.xs, n, dp, d, b.cs, k, p, st, v.packed));
    add_stats_kernel<<<1, 1, 0, st>>>(b.counters, b.stats);
    SKM_CUDA_TRY(launched());
    return SKM_OK;
}

// ------------------------------------------------------------- projection
namespace {
// fp32 v -> bf16 parts v1 + v2 + v3 (each the round-to-nearest-even bf16 of
// the remainder; the remainders are exact in fp32)
__device__ __forceinline__ void split3(float v, uint16_t &a, uint16_t &b, uint16_t &c) {
    const __nv_bfloat16 h1 = __float2bfloat16_rn(v);
    const float r1 = __fsub_rn(v, __bfloat162float(h1));
    const __nv_bfloat16 h2 = __float2bfloat16_rn(r1);
    const float r2 = __fsub_rn(r1, __bfloat162float(h2));
    a = __bfloat16_as_ushort(h1);
    b = __bfloat16_as_ushort(h2);
    c = __bfloat16_as_ushort(__float2bfloat16_rn(r2));
}

// rows [0, n) of X - mean -> A parts [3][n][dp] (8 dimensions per thread)
__global__ void proj_split_x_kernel(const float *__restrict__ X, int64_t n, int d, const float *__restrict__ mu,
                                    int dp, uint16_t *__restrict__ A) {
    const int no = dp / 8;
    const int64_t total = n * no;
    const size_t part = (size_t)n * dp;
    for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < total; t += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = t / no;
        const int i0 = (int)(t - r * no) * 8;
        uint32_t w[3][4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            uint16_t a[2], b[2], c[2];
#pragma unroll
            for (int u = 0; u < 2; ++u) {
                const int i = i0 + 2 * q + u;
                float v = 0.0f;
                if (i < d) v = mu ? __fsub_rn(X[r * d + i], mu[i]) : X[r * d + i];
                split3(v, a[u], b[u], c[u]);
            }
            w[0][q] = (uint32_t)a[0] | ((uint32_t)a[1] << 16);
            w[1][q] = (uint32_t)b[0] | ((uint32_t)b[1] << 16);
            w[2][q] = (uint32_t)c[0] | ((uint32_t)c[1] << 16);
        }
#pragma unroll
        for (int s3 = 0; s3 < 3; ++s3)
            *reinterpret_cast<uint4 *>(A + s3 * part + r * dp + i0) = make_uint4(w[s3][0], w[s3][1], w[s3][2], w[s3][3]);
    }
}

// P [d][dout] -> B parts [3][dout][dp] (transposed: K-major rows per output column)
__global__ void proj_split_p_kernel(const float *__restrict__ P, int d, int dout, int dp, uint16_t *__restrict__ B) {
    const int64_t total = (int64_t)dout * dp;
    const size_t part = (size_t)dout * dp;
    for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < total; t += (int64_t)gridDim.x * blockDim.x) {
        const int j = (int)(t / dp), i = (int)(t - (int64_t)j * dp);
        uint16_t a = 0, b = 0, c = 0;
        if (i < d) split3(P[(int64_t)i * dout + j], a, b, c);
        B[t] = a;
        B[part + t] = b;
        B[2 * part + t] = c;
    }
}
}  // namespace

size_t tc_project_ws_min(int d, int dout) {
    const size_t dp = (size_t)round8(d);
    return 256 + 3 * (size_t)dout * dp * 2 + 256 + 3 * (size_t)BM * dp * 2 + 256 + 64;
}

size_t tc_project_ws_full(int64_t n, int d, int dout) {
    const size_t dp = (size_t)round8(d);
    return 256 + 3 * (size_t)dout * dp * 2 + 256 + 3 * (size_t)n * dp * 2 + 256 + 64;
}

int tc_project(const float *X, int64_t n, int d, const float *mean, const float *P, int dout, int out_bf16, void *Y,
               void *ws, size_t ws_bytes, cudaStream_t st) {
    const int dp = round8(d);
    Carver cv(ws, ws_bytes);
    int32_t *counters = cv.take<int32_t>(16);
    uint16_t *B = cv.take<uint16_t>((size_t)3 * dout * dp);
    const size_t used = cv.off + 256;
    int64_t rows = ws_bytes > used ? (int64_t)((ws_bytes - used) / ((size_t)3 * dp * 2)) : 0;
    if (rows >= n) rows = n;
    else rows = (rows / BM) * BM;
    if (rows < 1) return set_error(SKM_ERR_NO_MEMORY, "projection workspace too small");
    uint16_t *A = cv.take<uint16_t>((size_t)3 * rows * dp);
    if (cv.off > ws_bytes) return set_error(SKM_ERR_NO_MEMORY, "projection workspace too small");
    {
        int64_t blocks = ((int64_t)dout * dp + 255) / 256;
        if (blocks > 152 * 8) blocks = 152 * 8;
        proj_split_p_kernel<<<(unsigned)blocks, 256, 0, st>>>(P, d, dout, dp, B);
        SKM_CUDA_TRY(launched());
    }
    SKM_CUDA_TRY(cudaMemsetAsync(counters, 0, sizeof(int32_t) * 16, st));
    for (int64_t r0 = 0; r0 < n; r0 += rows) {
        const int64_t nr = n - r0 < rows ? n - r0 : rows;
        int64_t blocks = (nr * (dp / 8) + 255) / 256;
        if (blocks > 152 * 16) blocks = 152 * 16;
        proj_split_x_kernel<<<(unsigned)blocks, 256, 0, st>>>(X + r0 * d, nr, d, mean, dp, A);
        SKM_CUDA_TRY(launched());
        TcParams p{};
        p.counters = counters;
        p.y = out_bf16 ? (void *)(static_cast<uint16_t *>(Y) + r0 * dout) : (void *)(static_cast<float *>(Y) + r0 * dout);
        p.y_bf16 = out_bf16;
        p.ydout = dout;
        p.d = d;
        SKM_TRY(launch_tc<MODE_GEMM>(A, nr, dp, d, B, dout, p, st));
    }
    return SKM_OK;
}

int tc_read_stats(const TcAssignBufs &b, skm_stats *st_host, cudaStream_t st) {
    int64_t h[4] = {0, 0, 0, 0};
    SKM_CUDA_TRY(cudaMemcpyAsync(h, b.stats, sizeof(h), cudaMemcpyDeviceToHost, st));
    SKM_CUDA_TRY(cudaStreamSynchronize(st));
    if (st_host) {
        st_host->rescored_rows = h[0];
        st_host->fallback_rows = h[1];
    }
    if (h[2]) return set_error(SKM_ERR_TIMEOUT, "a tensor-core pipeline wait exceeded its limit");
    return SKM_OK;
}

}  // namespace skm
