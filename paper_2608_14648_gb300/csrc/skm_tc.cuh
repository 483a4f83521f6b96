// Assignment for the dense representations (F32, BF16, SQ8): buffers and
// entry points used by skm_abi.cu.
#pragma once
#include "skm_internal.cuh"

namespace skm {

struct TcAssignBufs {
    int64_t *stats = nullptr;  // [0] rescored rows, [1] fallback rows (cumulative)
};

void tc_plan(int repr, int64_t n, int d, int k, Carver &cv, TcAssignBufs &b);
int tc_assign_float(const skm_data *x, const float *C, int k, int32_t *assign, float *dist,
                    TcAssignBufs &b, cudaStream_t st);
int tc_assign_sq8(const skm_data *x, const uint8_t *C, int k, const int32_t *nx,
                  const int32_t *nc, int32_t *assign, float *dist, TcAssignBufs &b,
                  cudaStream_t st);
void tc_read_stats(const TcAssignBufs &b, skm_stats *st_host, cudaStream_t st);

}  // namespace skm
