// skm_lloyd_step_host: one Lloyd iteration (Section 2.3, STEP 2 then STEP 3)
// of points that live in host memory.
//
// The points cross the host link once per iteration, so the step is built as
// a copy/compute pipeline: the rows are cut into `chunks` ranges; range i is
// copied host -> device on the caller's copy stream into one of R = 3 range
// buffers of the workspace while the compute stream assigns and sums range
// i - 1 (and i - 2); a buffer is refilled only after the compute stream has
// finished with it and has sent the range's assignments back.  The cluster
// sums of the ranges go into one set of partial sums (the sharded form of
// skm_update), an optional caller hook exchanges them (the one multi-process
// exchange per iteration), and the finalised centroids go back to the host.
// Everything is composed from the library's own entry points (skm_assign,
// skm_update, skm_update_finalize) on device views of the range buffers; with
// pruning, the ranges after the first reuse the first range's centroid-side
// preparation of the tensor-core front.
#include <vector>

#include "skm_internal.cuh"

namespace skm {
namespace {

constexpr int RING = 3;
constexpr int MAX_CHUNKS = 256;
constexpr int RED = 304;

int64_t host_row_bytes(const skm_data *x) {
    switch (x->repr) {
    case SKM_REPR_F32: return (int64_t)x->d * 4;
    case SKM_REPR_BF16: return (int64_t)x->d * 2;
    case SKM_REPR_SQ8: return (int64_t)x->d;
    default: return 0;
    }
}

int host_check(const skm_step_host_config *cfg, const skm_data *x) {
    if (!cfg || !x) return set_error(SKM_ERR_INVALID_ARG, "cfg and x are required");
    if (x->repr != SKM_REPR_F32 && x->repr != SKM_REPR_BF16 && x->repr != SKM_REPR_SQ8)
        return set_error(SKM_ERR_UNSUPPORTED, "skm_lloyd_step_host: F32, BF16 or SQ8 points (repr %d)", x->repr);
    if (x->flags != 0) return set_error(SKM_ERR_UNSUPPORTED, "skm_lloyd_step_host: no flags (got %d)", x->flags);
    if (x->d < 1 || x->d > 4096 || x->n < 1 || x->n >= (int64_t(1) << 31))
        return set_error(SKM_ERR_INVALID_ARG, "bad shape n=%lld d=%d", (long long)x->n, x->d);
    if (cfg->k < 1 || cfg->k > 65536 || (int64_t)cfg->k > x->n)
        return set_error(SKM_ERR_INVALID_ARG, "k = %d outside [1, min(n, 65536)]", cfg->k);
    if (cfg->chunks < 1 || cfg->chunks > MAX_CHUNKS)
        return set_error(SKM_ERR_INVALID_ARG, "chunks = %d outside [1, %d]", cfg->chunks, MAX_CHUNKS);
    if (x->screen) return set_error(SKM_ERR_INVALID_ARG, "skm_lloyd_step_host: x->screen must be NULL");
    if (cfg->prune && (!cfg->warm || x->repr != SKM_REPR_BF16))
        return set_error(SKM_ERR_UNSUPPORTED, "skm_lloyd_step_host: prune needs warm and BF16 points");
    return SKM_OK;
}

// Device view of `rows` rows of the representation at `base`.
skm_data view_of(const skm_data *x, const void *base, int64_t rows) {
    skm_data v = *x;
    v.x = base;
    v.n = rows;
    v.screen = nullptr;
    return v;
}

struct HostBufs {
    uint8_t *ring[RING] = {};
    int32_t *assign[RING] = {};
    float *dist[RING] = {};
    void *C = nullptr;
    void *partial = nullptr;
    int64_t *counts = nullptr;
    double *red = nullptr, *chunk_sum = nullptr, *total = nullptr;
    uint8_t *ws_a = nullptr, *ws_u = nullptr;
    size_t ws_a_bytes = 0, ws_u_bytes = 0;
    size_t ws_a_stride = 0;  // warm: range i's assignment workspace at ws_a + i * ws_a_stride
};

bool host_warm(const skm_step_host_config *cfg, const skm_data *x) {
    return cfg->warm && (x->repr == SKM_REPR_F32 || x->repr == SKM_REPR_BF16);
}

void plan_host(const skm_step_host_config *cfg, const skm_data *x, Carver &cv, HostBufs &b) {
    const int64_t rc = cdiv(x->n, cfg->chunks);
    const int64_t rb = host_row_bytes(x);
    const int k = cfg->k, d = x->d;
    const int nr = (int)std::min<int64_t>(RING, cfg->chunks);
    for (int s = 0; s < nr; ++s) {
        b.ring[s] = cv.take<uint8_t>((size_t)(rc * rb));
        b.assign[s] = cv.take<int32_t>((size_t)rc);
        b.dist[s] = cv.take<float>((size_t)rc);
    }
    b.C = cv.take<uint8_t>((size_t)k * d * (x->repr == SKM_REPR_SQ8 ? 1 : 4));
    if (!cfg->partial) b.partial = cv.take<uint8_t>((size_t)k * d * 8);
    if (!cfg->counts) b.counts = cv.take<int64_t>((size_t)k);
    b.red = cv.take<double>(RED);
    b.chunk_sum = cv.take<double>(MAX_CHUNKS);
    b.total = cv.take<double>(1);
    // the entry points' own workspaces for a range of rc rows (reused by
    // every range: the compute stream runs them one after another)
    skm_data probe = view_of(x, reinterpret_cast<const void *>(256), rc);
    if (host_warm(cfg, x)) probe.flags |= SKM_FLAG_WARM;
    if (cfg->prune) probe.flags |= SKM_FLAG_PRUNE;
    b.ws_a_bytes = skm_workspace_size(0, &probe, k);
    probe.flags = 0;
    b.ws_u_bytes = skm_workspace_size(1, &probe, k);
    // warm: one assignment workspace per range (each keeps its rows' bounds)
    b.ws_a_stride = (b.ws_a_bytes + 255) & ~size_t(255);
    b.ws_a = cv.take<uint8_t>(host_warm(cfg, x) ? b.ws_a_stride * (size_t)cfg->chunks : b.ws_a_bytes);
    b.ws_u = cv.take<uint8_t>(b.ws_u_bytes);
}

}  // namespace
}  // namespace skm

using namespace skm;

extern "C" size_t skm_step_host_workspace_size(const skm_step_host_config *cfg, const skm_data *x) {
    if (host_check(cfg, x) != SKM_OK) return 0;
    Carver cv(nullptr, 0);
    HostBufs b;
    plan_host(cfg, x, cv, b);
    if (b.ws_a_bytes == 0 || b.ws_u_bytes == 0) return 0;
    return cv.off;
}

extern "C" int skm_lloyd_step_host(const skm_step_host_config *cfg, const skm_data *x, const void *C_host,
                                   void *C_host_out, int32_t *assign_host, int64_t *counts_host,
                                   double *objective_host, void *ws, size_t ws_bytes, void *stream) {
    SKM_TRY(host_check(cfg, x));
    if (!x->x || !C_host || !C_host_out || !assign_host)
        return set_error(SKM_ERR_INVALID_ARG, "x->x, C_host, C_host_out and assign_host are required");
    if (!ws) return set_error(SKM_ERR_INVALID_ARG, "workspace is NULL");
    if (((uintptr_t)ws & 255) != 0) return set_error(SKM_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
    Carver cv(ws, ws_bytes);
    HostBufs b;
    plan_host(cfg, x, cv, b);
    if (b.ws_a_bytes == 0 || b.ws_u_bytes == 0) return SKM_ERR_INVALID_ARG;  // message set by skm_workspace_size
    if (fault_take(SKM_FAULT_WORKSPACE))
        return set_error(SKM_ERR_NO_MEMORY, "injected fault: workspace reported too small");
    if (cv.off > ws_bytes)
        return set_error(SKM_ERR_NO_MEMORY, "workspace too small: need %zu bytes, got %zu", cv.off, ws_bytes);
    {
        // the points must be page-locked: a pageable source would make every
        // range copy a synchronous staged copy
        cudaPointerAttributes at;
        const cudaError_t e = cudaPointerGetAttributes(&at, x->x);
        if (e != cudaSuccess || at.type != cudaMemoryTypeHost) {
            (void)cudaGetLastError();
            return set_error(SKM_ERR_INVALID_ARG, "x->x must be page-locked host memory");
        }
    }
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    cudaStream_t cp = cfg->copy_stream ? static_cast<cudaStream_t>(cfg->copy_stream) : st;
    const int64_t n = x->n;
    const int k = cfg->k, d = x->d, nchunk = cfg->chunks;
    const int64_t rc = cdiv(n, nchunk), rb = host_row_bytes(x);
    const int nr = (int)std::min<int64_t>(RING, nchunk);
    void *partial = cfg->partial ? cfg->partial : b.partial;
    int64_t *counts = cfg->counts ? cfg->counts : b.counts;
    const size_t cbytes = (size_t)k * d * (x->repr == SKM_REPR_SQ8 ? 1 : 4);
    const char *xh = static_cast<const char *>(x->x);
    const bool warm = host_warm(cfg, x);

    cudaEvent_t landed[RING], freed[RING];
    int made = 0;
    int rc_status = SKM_OK;
    auto fail = [&](int s) {
        if (rc_status == SKM_OK) rc_status = s;
        return s;
    };
    for (; made < nr; ++made) {
        if (cudaEventCreateWithFlags(&landed[made], cudaEventDisableTiming) != cudaSuccess) break;
        if (cudaEventCreateWithFlags(&freed[made], cudaEventDisableTiming) != cudaSuccess) {
            cudaEventDestroy(landed[made]);
            break;
        }
    }
    if (made < nr) fail(set_error(SKM_ERR_CUDA, "cudaEventCreate failed"));

    auto run = [&]() -> int {
        SKM_CUDA_TRY(cudaMemcpyAsync(b.C, C_host, cbytes, cudaMemcpyHostToDevice, st));
        SKM_CUDA_TRY(cudaMemsetAsync(partial, 0, (size_t)k * d * 8, st));
        SKM_CUDA_TRY(cudaMemsetAsync(counts, 0, sizeof(int64_t) * (size_t)k, st));
        if (cp != st) {  // the copy stream starts after the caller's earlier work on `stream`
            SKM_CUDA_TRY(cudaEventRecord(freed[0], st));
            SKM_CUDA_TRY(cudaStreamWaitEvent(cp, freed[0], 0));
        }
        for (int i = 0; i < nchunk; ++i) {
            const int s = i % nr;
            const int64_t r0 = (int64_t)i * rc;
            const int64_t rows = std::min<int64_t>(rc, n - r0);
            if (rows <= 0) break;
            if (i >= nr) SKM_CUDA_TRY(cudaStreamWaitEvent(cp, freed[s], 0));
            SKM_CUDA_TRY(cudaMemcpyAsync(b.ring[s], xh + r0 * rb, (size_t)(rows * rb), cudaMemcpyHostToDevice, cp));
            if (cfg->prune)  // the range's seeds: the previous call's assignments
                SKM_CUDA_TRY(cudaMemcpyAsync(b.assign[s], assign_host + r0, sizeof(int32_t) * (size_t)rows,
                                             cudaMemcpyHostToDevice, cp));
            SKM_CUDA_TRY(cudaEventRecord(landed[s], cp));
            SKM_CUDA_TRY(cudaStreamWaitEvent(st, landed[s], 0));
            skm_data v = view_of(x, b.ring[s], rows);
            uint8_t *wsa = b.ws_a;
            if (warm) {  // this range's own workspace: its rows' bounds from the previous call
                v.flags |= SKM_FLAG_WARM;
                wsa = b.ws_a + (size_t)i * b.ws_a_stride;
            }
            if (cfg->prune) v.flags |= SKM_FLAG_PRUNE;
            if (cfg->prune && warm && i > 0) {
                // the centroid side of the pruning front was prepared by range
                // 0's call (same centroids, its workspace): this range's rows only
                skm_data v0 = view_of(x, b.ring[0], std::min<int64_t>(rc, n));
                v0.flags = v.flags;
                SKM_TRY(assign_range_shared(&v, b.C, k, b.assign[s], b.assign[s], objective_host ? b.dist[s] : nullptr,
                                            wsa, b.ws_a_bytes, &v0, b.ws_a, b.ws_a_bytes, st));
            } else {
                SKM_TRY(skm_assign(&v, b.C, k, cfg->prune ? b.assign[s] : nullptr, b.assign[s],
                                   objective_host ? b.dist[s] : nullptr, wsa, b.ws_a_bytes, st));
            }
            v.flags = 0;
            SKM_TRY(skm_update(&v, b.assign[s], k, nullptr, counts, partial, b.ws_u, b.ws_u_bytes, st));
            if (objective_host) {
                const int nblk = (int)std::min<int64_t>(RED, rows);
                SKM_CUDA_TRY(launch_sum_float_to_double(b.dist[s], rows, b.red, nblk, st));
                SKM_CUDA_TRY(launch_sum_double(b.red, nblk, b.chunk_sum + i, st));
            }
            SKM_CUDA_TRY(cudaMemcpyAsync(assign_host + r0, b.assign[s], sizeof(int32_t) * (size_t)rows,
                                         cudaMemcpyDeviceToHost, st));
            SKM_CUDA_TRY(cudaEventRecord(freed[s], st));
        }
        if (cfg->exchange) {
            if (cfg->exchange(partial, counts, cfg->user, stream) != 0)
                return set_error(SKM_ERR_EXCHANGE, "the exchange hook reported a failure");
        }
        SKM_TRY(skm_update_finalize(x, partial, counts, k, b.C, stream));
        SKM_CUDA_TRY(cudaMemcpyAsync(C_host_out, b.C, cbytes, cudaMemcpyDeviceToHost, st));
        if (counts_host)
            SKM_CUDA_TRY(cudaMemcpyAsync(counts_host, counts, sizeof(int64_t) * (size_t)k, cudaMemcpyDeviceToHost, st));
        if (objective_host) {
            SKM_CUDA_TRY(launch_sum_double(b.chunk_sum, (int64_t)cdiv(n, rc), b.total, st));
            SKM_CUDA_TRY(cudaMemcpyAsync(objective_host, b.total, sizeof(double), cudaMemcpyDeviceToHost, st));
        }
        return SKM_OK;
    };
    if (rc_status == SKM_OK) fail(run());
    // whatever was enqueued completes before the events go away and the call
    // returns (the outputs are then in host memory)
    const cudaError_t e1 = cudaStreamSynchronize(st);
    const cudaError_t e2 = cp != st ? cudaStreamSynchronize(cp) : cudaSuccess;
    for (int s = 0; s < made; ++s) {
        cudaEventDestroy(landed[s]);
        cudaEventDestroy(freed[s]);
    }
    if (rc_status != SKM_OK) return rc_status;
    if (e1 != cudaSuccess || e2 != cudaSuccess)
        return set_error(SKM_ERR_CUDA, "stream synchronize failed: %s",
                         cudaGetErrorString(e1 != cudaSuccess ? e1 : e2));
    return SKM_OK;
}
