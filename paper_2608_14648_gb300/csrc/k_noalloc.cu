// skm_assign_rbq1_noalloc: the 1-bit (RabitQ) assignment with its per-call
// scratch held in a fixed device array instead of a caller workspace.
//
// Some callers cannot allocate device memory: code that runs inside a host
// engine which owns every byte of device memory through its own pool or a
// fixed budget, and latency-critical paths where cudaMalloc/cudaFree (which
// may synchronise the whole device) are not acceptable.  This entry point
// needs nothing from them but the inputs and outputs.
//
// The scratch is the per-centroid SQ4 bit planes (k * ceil(d/32) uint4) and
// the per-centroid estimator terms (k records of 16 bytes), the same data
// skm_assign builds in its workspace.  It lives in one file-scope device array
// of 2.25 MiB that every GPU which loads the library keeps until exit.
#include "skm_internal.cuh"

namespace skm {
namespace {

constexpr size_t NOALLOC_PLANE_WORDS = 131072;  // uint4 entries: 2 MiB
constexpr int NOALLOC_MAX_K = 16384;            // centroid records: 256 KiB
constexpr size_t NOALLOC_BYTES = NOALLOC_PLANE_WORDS * sizeof(uint4) + NOALLOC_MAX_K * sizeof(Rbq1CInfo);

static __device__ __align__(256) unsigned char g_rbq1_scratch[NOALLOC_BYTES];

// Device address of g_rbq1_scratch in the current context, looked up on
// every call (cudaGetSymbolAddress allocates nothing), so the address stays
// right after the context is torn down and the module loaded again.
int scratch_address(void **out) {
    void *p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_rbq1_scratch);
    if (e != cudaSuccess || !p)
        return set_error(SKM_ERR_CUDA, "cudaGetSymbolAddress(g_rbq1_scratch) failed: %s", cudaGetErrorString(e));
    *out = p;
    return SKM_OK;
}

}  // namespace
}  // namespace skm

using namespace skm;

extern "C" int skm_assign_rbq1_noalloc(const skm_data *x, const float *C, int k, int32_t *assign,
                                       float *dist, void *stream) {
    if (!x || x->repr != SKM_REPR_RBQ1)
        return set_error(SKM_ERR_INVALID_ARG, "skm_assign_rbq1_noalloc needs RBQ1 points");
    if (x->flags & SKM_FLAG_SYMMETRIC)
        return set_error(SKM_ERR_UNSUPPORTED, "skm_assign_rbq1_noalloc: the asymmetric estimate only");
    if (!x->x || !x->nx2 || !x->F || !x->popx || !x->m || !C || !assign)
        return set_error(SKM_ERR_INVALID_ARG, "NULL pointer");
    if (x->d < 1 || x->d > 4096 || x->n < 1 || x->n > (int64_t(1) << 24))
        return set_error(SKM_ERR_INVALID_ARG, "bad shape n=%lld d=%d", (long long)x->n, x->d);
    if (k < 1) return set_error(SKM_ERR_INVALID_ARG, "k = %d", k);
    const size_t words = (size_t)k * words_of(x->d);
    if (k > NOALLOC_MAX_K || words > NOALLOC_PLANE_WORDS)
        return set_error(SKM_ERR_UNSUPPORTED,
                         "skm_assign_rbq1_noalloc: k = %d, d = %d needs %zu plane words; the fixed "
                         "scratch holds k <= %d and k * ceil(d/32) <= %zu",
                         k, x->d, words, NOALLOC_MAX_K, NOALLOC_PLANE_WORDS);
    void *base = nullptr;
    SKM_TRY(scratch_address(&base));
    uint4 *planes = static_cast<uint4 *>(base);
    Rbq1CInfo *info = reinterpret_cast<Rbq1CInfo *>(static_cast<unsigned char *>(base) +
                                                    NOALLOC_PLANE_WORDS * sizeof(uint4));
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    // every record and plane word the assignment reads for these k centroids
    // is rewritten here, so nothing from an earlier call needs clearing
    SKM_CUDA_TRY(launch_rbq1_cprep(C, k, x->d, x->m, planes, info, st));
    SKM_CUDA_TRY(launch_assign_rbq1(static_cast<const uint32_t *>(x->x), x->nx2, x->F, x->popx, x->n,
                                    x->d, planes, info, k, assign, dist, st));
    return SKM_OK;
}
