// Tensor-core assignment for the dense representations (F32, BF16, SQ8):
// buffers and entry points used by skm_abi.cu (implemented in k_tc.cu).
#pragma once
#include "skm_internal.cuh"

namespace skm {

// Above this d the fp32 accumulator of the bf16-encoded SQ8 dot product can
// exceed 2^24 and stop being exact; SQ8 then uses the __dp4a kernel.
constexpr int TC_SQ8_MAX_D = 1024;
// The e4m3 1-bit path rounds its accumulator to the integer P; up to this d
// (P < 2^14) the accumulation error stays far below 1/2.  Beyond it the
// AND + popcount kernel is used.
constexpr int TC_RBQ1_MAX_D = 1024;
// LVQ4 on the same e4m3 path: P <= 225 d stays below 2^18 up to this d; beyond
// it the __dp4a kernel is used.
constexpr int TC_LVQ4_MAX_D = 1024;

struct TcAssignBufs {
    int64_t *stats = nullptr;     // [0] rescored rows, [1] fallback rows, [2] timeout (cumulative)
    int32_t *counters = nullptr;  // per call: [0] rescore list, [1] fallback list, [2] abort flag
    uint8_t *screen = nullptr;    // screening copy built per call when the caller gave none
    uint8_t *pk_scratch = nullptr;  // RBQ1 read packed: per-CTA tile expansion slots
    // F32/BF16 with SKM_FLAG_WARM: stamp of the last complete call (magic, n,
    // d, k), per row (bound bits, centroid), the previous centroids, and per
    // centroid (||c'||^2 - ||c||^2, ||c' - c||) rounded up
    int64_t *warm_hdr = nullptr;
    int2 *warm_row = nullptr;
    float *warm_cprev = nullptr;
    float2 *warm_shift = nullptr;
    uint16_t *cs = nullptr;       // centroid operand, bf16 [k][round8(d)]
    float4 *cinfo = nullptr;      // F32/BF16: per-column-pair bound terms
    float2 *cinfoz = nullptr;
    int32_t *nc = nullptr;        // SQ8: centred ||c||^2
    Rbq1CInfo *rinfo = nullptr;   // RBQ1: per-centroid estimator terms
    float4 *linfo = nullptr;      // LVQ4: per-centroid (s, b, N, G)
    float4 *rpair_bs = nullptr;   // RBQ1 / LVQ4: column-pair records (padded)
    float4 *rpair_qn = nullptr;
    int32_t *cand = nullptr;      // F32/BF16: [n][5] screen candidates + count
    int32_t *resc_rows = nullptr;
    int32_t *fall_rows = nullptr;
    unsigned long long *fall_keys = nullptr;  // F32/BF16: per fallback row, (dist bits, index)
    // BF16 with SKM_FLAG_PRUNE (tensor-core front): per row (threshold, seed
    // distance), survivor lists, per listed row the sub-lists' counts
    float2 *pf_thr = nullptr;
    uint16_t *pf_cand = nullptr;
    int32_t *pf_cnt = nullptr;
    // ... and the centroid operand / records in centroid order (the sorted
    // copies are cs / cinfo), the sort's permutation and chunk minima
    uint16_t *pf_cs0 = nullptr;
    float4 *pf_cinfo0 = nullptr;
    int32_t *pf_perm = nullptr;
    float *pf_cmin = nullptr;
    int32_t *pf_seed = nullptr;  // per row: the seed centroid
    // ... with SKM_FLAG_WARM: stamp (magic, n, d, k, the generation of the
    // previous centroids the bounds were taken against), per row (bound bits,
    // centroid) and the prefix norms, the previous centroids and their moves
    int64_t *pf_whdr = nullptr;
    int64_t *pf_cgen = nullptr;  // generation of pf_cprev (advanced by each preparation)
    int2 *pf_wrow = nullptr;
    float2 *pf_xn = nullptr;
    float *pf_cprev = nullptr;
    float2 *pf_shift = nullptr;
};

// Segmented assignment: rows sorted by group, row r only takes centroids
// [base[g], base[g + 1]) of g = group[r]; ct0 / nct: workspace of one int32
// per 128-row point tile.
struct TcSeg {
    const int32_t *group = nullptr;
    const int32_t *base = nullptr;
    int nseg = 0;
    int32_t *ct0 = nullptr;
    int32_t *nct = nullptr;
};

size_t tc_screen_bytes(int repr, int64_t n, int d, const void *x);
int tc_screen_prep(const skm_data *x, void *screen, cudaStream_t st);
// whether the 1-bit / LVQ4 tensor-core assignment reads these codes packed
// when no screening copy is given
bool tc_reads_packed(int repr, int d, const void *x);
void tc_plan(int repr, int64_t n, int d, int k, const void *x, const void *screen, bool warm, Carver &cv,
             TcAssignBufs &b);
int tc_init_stats(TcAssignBufs &b, cudaStream_t st);
// Exact dimension pruning of bf16 points with the first dimensions on tensor
// cores (used when a seed assignment is given): whether these points can take
// it, its workspace, and the call.  ctr: the pruning counters ([0] pairs alive
// after the front, [1] complete, [2] 32-dimension blocks evaluated on CUDA
// cores, [3] front dimensions, [4] rows finished on CUDA cores, [5] rows
// pruned over all k, [6..8] the latter's own counters, [9] k).
bool tc_pfront_ok(int repr, int d, const void *x);
void tc_plan_pfront(int64_t n, int d, int k, bool warm, Carver &cv, TcAssignBufs &b);
// sh: the centroid side was prepared by an earlier call this step in the
// workspace sh, on the same centroids (only this call's rows are done here).
int tc_assign_pfront(const skm_data *x, const float *C, int k, const int32_t *prev, int32_t *assign, float *dist,
                     TcAssignBufs &b, unsigned long long *ctr, cudaStream_t st, const TcAssignBufs *sh = nullptr);
int tc_assign_float(const skm_data *x, const float *C, int k, int32_t *assign, float *dist,
                    TcAssignBufs &b, cudaStream_t st, const TcSeg *seg = nullptr);
// nx_plain / nc_plain: buffers for the __dp4a path (d > TC_SQ8_MAX_D), filled here.
int tc_assign_sq8(const skm_data *x, const uint8_t *C, int k, int32_t *nx_plain,
                  int32_t *nc_plain, int32_t *assign, float *dist, TcAssignBufs &b,
                  cudaStream_t st, const TcSeg *seg = nullptr);
// RBQ1 on tensor cores (e4m3 operands, exact integer P, same fp32 epilogue
// as the AND+popcount kernel).
int tc_assign_rbq1(const skm_data *x, const float *C, int k, int32_t *assign, float *dist,
                   TcAssignBufs &b, cudaStream_t st, const TcSeg *seg = nullptr);
// LVQ4 on tensor cores (e4m3 codes, exact integer P, Eq. final:lvq epilogue).
int tc_assign_lvq4(const skm_data *x, const float *C, int k, int32_t *assign, float *dist,
                   TcAssignBufs &b, cudaStream_t st, const TcSeg *seg = nullptr);
// Y = (X - mean) P on tensor cores with fp32 accuracy (bf16 parts, six
// products); ws: at least tc_project_ws_min (rows are then processed in chunks),
// tc_project_ws_full for one pass.
size_t tc_project_ws_min(int d, int dout);
size_t tc_project_ws_full(int64_t n, int d, int dout);
int tc_project(const float *X, int64_t n, int d, const float *mean, const float *P, int dout, int out_bf16, void *Y,
               void *ws, size_t ws_bytes, cudaStream_t st);
// Copies the cumulative statistics; returns SKM_ERR_TIMEOUT if a pipeline
// wait gave up.  Synchronises the stream.
int tc_read_stats(const TcAssignBufs &b, skm_stats *st_host, cudaStream_t st);

}  // namespace skm
