// phsa_sparse_attn_bwd_noalloc: the backward pass with its scratch memory in a
// fixed, library-owned device array instead of a caller-supplied workspace.
//
// Some callers cannot allocate device memory at the point where they run the
// backward pass: a serving or training engine that reserves all of HBM for its
// own pools at start-up and forbids later allocations, a plugin interface whose
// execute step may not allocate, or a hot loop that cannot afford the implicit
// device synchronisation of cudaMalloc/cudaFree. This entry point needs no
// allocation from anyone: the scratch lives in a file-scope device array that
// every GPU holds for as long as the library stays loaded.
//
// Limits and sharing: the array holds kScratchBytes (64 MiB); shapes whose
// phsa_sparse_attn_bwd_workspace() exceeds that are rejected with
// PHSA_ERR_WORKSPACE before anything is launched. All calls on a device share
// the one array and it keeps the last call's contents; the launch sequence
// clears the part that must start at zero (the pair bitmap) on every call and
// writes every other part before reading it. Two calls whose work overlaps on
// the GPU (for example on two streams) race on the array and give wrong
// results; serialise them.
#include <mutex>

#include "phsa_common.cuh"
#include "phsa_internal.h"

namespace {

constexpr size_t kScratchBytes = size_t(64) << 20;
static __device__ __align__(256) unsigned char g_bwd_scratch[kScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
void* g_scratch_ptr[kMaxDevices] = {nullptr};

// Device address of the scratch array on the current device. The address of
// a __device__ array is per device and only the runtime knows it, so it is
// looked up once per device (with that device current) and cached.
cudaError_t scratch_for_current_device(void** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lk(g_scratch_mu);
    if (!g_scratch_ptr[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_bwd_scratch);
        if (e != cudaSuccess) return e;
        g_scratch_ptr[dev] = p;
    }
    *out = g_scratch_ptr[dev];
    return cudaSuccess;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

extern "C" int phsa_sparse_attn_bwd_noalloc(const void* Q, const void* K, const void* V,
                                            const void* O, const void* dO, const float* lse,
                                            const int32_t* block_idx, const int32_t* block_cnt,
                                            phsa_shape s, int topk, float sm_scale, void* dQ,
                                            void* dK, void* dV, void* stream) {
    // The same checks, in the same order and with the same codes, as
    // phsa_sparse_attn_bwd; only the workspace check differs (the fixed array).
    const int rc = phsa::validate_bwd(s, topk);
    if (rc != PHSA_OK) return rc;
    if (!(sm_scale > 0.f) || !isfinite(sm_scale)) return PHSA_ERR_INVALID_ARG;
    if (s.B == 0 || s.L == 0) return PHSA_OK;
    if (!Q || !K || !V || !O || !dO || !lse || !block_idx || !block_cnt || !dQ || !dK || !dV)
        return PHSA_ERR_INVALID_ARG;
    const void* ptrs[] = {Q, K, V, O, dO, dQ, dK, dV};
    for (const void* p : ptrs)
        if (!aligned16(p)) return PHSA_ERR_INVALID_ARG;
    if (phsa::bwd_layout(s, topk).total > kScratchBytes) return PHSA_ERR_WORKSPACE;
    void* ws = nullptr;
    if (scratch_for_current_device(&ws) != cudaSuccess) return PHSA_ERR_CUDA;
    int* st = phsa::device_status_word();
    if (!st) return PHSA_ERR_CUDA;
    return phsa::status_of(phsa::launch_attn_bwd(Q, K, V, O, dO, lse, block_idx, block_cnt, s,
                                                 topk, sm_scale, ws, dQ, dK, dV, st,
                                                 static_cast<cudaStream_t>(stream)));
}
