// adapld_semantic_topk_static(): the semantic fallback without a caller
// workspace.  Its scratch (counters, the row plan and the partial top-k slots
// of the semantic kernel) lives in one file-scope device array instead.
//
// Who needs this: host code that can pass device pointers for its inputs and
// outputs but cannot obtain any extra device memory for the library -- for
// example a plugin inside a serving process whose GPU memory is entirely owned
// by another allocator (a cudaMalloc there would bypass that allocator's
// budget and implicitly synchronise the device), or a caller whose API has no
// slot for a workspace buffer.  This entry point calls no cudaMalloc, cudaFree
// or allocating library routine.
#include <mutex>

#include "checks.h"

using namespace adapld;

namespace {

// The scratch array.  Every GPU that loads the library reserves it until the
// process exits.  In host code the name is only a host-side stand-in: the
// device address comes from cudaGetSymbolAddress (see scratch_address).
static __device__ __align__(256) unsigned char g_semantic_scratch[ADAPLD_STATIC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_mutex;
void *g_address[kMaxDevices] = {};

// Device address of g_semantic_scratch on the current device, looked up once
// per device (with that device current) and cached.
int scratch_address(void **out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return ADAPLD_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_mutex);
    if (g_address[dev] == nullptr) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_semantic_scratch) != cudaSuccess || p == nullptr)
            return ADAPLD_ERR_CUDA;
        g_address[dev] = p;
    }
    *out = g_address[dev];
    return ADAPLD_OK;
}

// Only what the semantic path uses: the status word and the per-sequence
// completion counters (cleared every call), the plan and the slots.
Workspace static_layout(void *base, int32_t B) {
    Workspace w{};
    char *p = (char *)base;
    w.dev_status = (int32_t *)p;
    w.done2 = w.dev_status + 2;
    w.counters_bytes = sizeof(int32_t) * (2 + (size_t)B);
    size_t off = align_up(w.counters_bytes, 256);
    w.plan = (int64_t *)(p + off);
    off = align_up(off + sizeof(int64_t) * ((size_t)B + 1), 256);
    w.slots2 = (int32_t *)(p + off);
    off = align_up(off + sizeof(int32_t) * ((size_t)B + kMaxGrid2) * kSlotInts, 256);
    w.total_bytes = off;
    w.C1 = w.S4 = w.W = 1;
    return w;
}

}  // namespace

extern "C" int adapld_semantic_topk_static(const uint16_t *reps, int64_t ld, int32_t d,
                                           const uint16_t *query, const int32_t *lengths,
                                           const uint8_t *active, int32_t B, int32_t k, float tau,
                                           int32_t *cand, float *score, int32_t *n_cand,
                                           adapld_stream_t stream) {
    if (!reps || !query || !lengths || !cand || !score || !n_cand) return ADAPLD_ERR_NULL;
    if (B > ADAPLD_STATIC_MAX_B) return ADAPLD_ERR_STATIC_LIMIT;
    // the same checks, in the same order, as adapld_semantic_topk()
    ADAPLD_TRY(check_shape(B, ld));
    ADAPLD_TRY(check_dim(d));
    if (!aligned16(reps) || !aligned16(query)) return ADAPLD_ERR_ALIGN;
    ADAPLD_TRY(check_k(k));
    ADAPLD_TRY(check_tau(tau));
    void *base = nullptr;
    const int rc = scratch_address(&base);
    if (rc != ADAPLD_OK) return rc;
    const Workspace w = static_layout(base, B);
    if (w.total_bytes > ADAPLD_STATIC_SCRATCH_BYTES) return ADAPLD_ERR_STATIC_LIMIT;
    cudaStream_t s = (cudaStream_t)stream;
    if (cudaMemsetAsync(w.dev_status, 0, w.counters_bytes, s) != cudaSuccess)
        return ADAPLD_ERR_CUDA;
    SemLaunch a{reps, ld, d, query, lengths, active, B, k, tau, cand, score, n_cand,
                nullptr, false};
    return launch_semantic(a, w, s) == cudaSuccess ? ADAPLD_OK : ADAPLD_ERR_CUDA;
}

extern "C" int adapld_semantic_topk_static_status(int32_t *status, adapld_stream_t stream) {
    if (!status) return ADAPLD_ERR_NULL;
    void *base = nullptr;
    const int rc = scratch_address(&base);
    if (rc != ADAPLD_OK) return rc;
    // the status word is the first int32 of the array (static_layout)
    cudaStream_t s = (cudaStream_t)stream;
    if (cudaMemcpyAsync(status, base, sizeof(int32_t), cudaMemcpyDeviceToHost, s) != cudaSuccess)
        return ADAPLD_ERR_CUDA;
    return cudaStreamSynchronize(s) == cudaSuccess ? ADAPLD_OK : ADAPLD_ERR_CUDA;
}
