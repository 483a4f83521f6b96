// Assignment for the dense representations.
#include "skm_tc.cuh"

namespace skm {

void tc_plan(int repr, int64_t n, int d, int k, Carver &cv, TcAssignBufs &b) {
    (void)repr; (void)n; (void)d; (void)k;
    b.stats = cv.take<int64_t>(2);
}

int tc_assign_float(const skm_data *x, const float *C, int k, int32_t *assign, float *dist,
                    TcAssignBufs &b, cudaStream_t st) {
    (void)b;
    if (x->repr == SKM_REPR_BF16)
        SKM_CUDA_TRY(launch_assign_exact_bf16(static_cast<const uint16_t *>(x->x), x->n, x->d, C, k,
                                              assign, dist, st));
    else
        SKM_CUDA_TRY(launch_assign_exact_f32(static_cast<const float *>(x->x), x->n, x->d, C, k,
                                             assign, dist, st));
    return SKM_OK;
}

int tc_assign_sq8(const skm_data *x, const uint8_t *C, int k, const int32_t *nx,
                  const int32_t *nc, int32_t *assign, float *dist, TcAssignBufs &b,
                  cudaStream_t st) {
    (void)b;
    SKM_CUDA_TRY(launch_assign_sq8_simt(static_cast<const uint8_t *>(x->x), x->n, x->d, C, k, nx,
                                        nc, assign, dist, st));
    return SKM_OK;
}

void tc_read_stats(const TcAssignBufs &b, skm_stats *st_host, cudaStream_t st) {
    (void)b; (void)st; (void)st_host;
}

}  // namespace skm
