// The C ABI (include/phsa.h): argument validation, the per-device status
// word, and dispatch to the kernel launchers.
#include <mutex>

#include "phsa_common.cuh"
#include "phsa_internal.h"

namespace {

// One status word per device, in a file-scope device variable (no allocation).
__device__ int g_device_status = 0;

constexpr int kMaxDevices = 64;
std::mutex g_mu;
int* g_status_ptr[kMaxDevices] = {nullptr};

// Device address of the status word on the current device (looked up once).
int* status_ptr() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_status_ptr[dev]) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_device_status) != cudaSuccess) return nullptr;
        g_status_ptr[dev] = static_cast<int*>(p);
    }
    return g_status_ptr[dev];
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Common shape checks; returns PHSA_OK or an error code. Block sizes 16 and
// 32 are accepted only where any_block is set (every call but the host-buffer
// step; the backward adds its own condition).
int check_shape(const phsa_shape& s, bool any_block = false) {
    if (s.B < 0 || s.L < 0 || s.Hq <= 0 || s.Hkv <= 0 || s.D <= 0 || s.block_size <= 0)
        return PHSA_ERR_INVALID_ARG;
    if (s.Hq % s.Hkv != 0) return PHSA_ERR_INVALID_ARG;
    if (s.D != phsa::kD) return PHSA_ERR_UNSUPPORTED;
    const int bm = s.block_size;
    if (any_block ? (bm != 16 && bm != 32 && bm != 64) : bm != phsa::kM) return PHSA_ERR_UNSUPPORTED;
    const int G = s.Hq / s.Hkv;
    if (G != 1 && G != 2) return PHSA_ERR_UNSUPPORTED;
    const long long nqb = ((long long)s.L + bm - 1) / bm;
    if ((long long)s.B * s.Hkv * nqb > 0x7fffffffLL) return PHSA_ERR_UNSUPPORTED;
    if ((long long)s.B * s.Hq > 0x7fffffffLL / (s.L > 0 ? s.L : 1)) return PHSA_ERR_UNSUPPORTED;
    if (s.B > 65535 * 8 || (long long)s.B * s.Hkv > 65535) return PHSA_ERR_UNSUPPORTED;
    return PHSA_OK;
}

bool empty(const phsa_shape& s) { return s.B == 0 || s.L == 0; }

int from_cuda(cudaError_t e) { return e == cudaSuccess ? PHSA_OK : PHSA_ERR_CUDA; }

int check_topk(const phsa_shape& s, int topk) {
    if (topk < 1) return PHSA_ERR_INVALID_ARG;
    if (topk > 4096) return PHSA_ERR_UNSUPPORTED;
    (void)s;
    return PHSA_OK;
}

// The backward takes block sizes 16 and 32 for GQA pairs (two query heads
// per KV head, the tcgen05 kernels) when their lists fit in shared memory.
int check_bwd(const phsa_shape& s, int topk) {
    int rc = check_shape(s, true);
    if (rc != PHSA_OK) return rc;
    if ((rc = check_topk(s, topk)) != PHSA_OK) return rc;
    if (s.block_size != phsa::kM && (s.Hq != 2 * s.Hkv || !phsa::dq_tc_fits(topk, s.block_size)))
        return PHSA_ERR_UNSUPPORTED;
    return PHSA_OK;
}

}  // namespace

namespace phsa {
// The status word of the current device, for entry points in other files.
int* device_status_word() { return status_ptr(); }
int validate_shape(const phsa_shape& s) { return check_shape(s); }
int validate_bwd(const phsa_shape& s, int topk) { return check_bwd(s, topk); }
int validate_topk(const phsa_shape& s, int topk) { return check_topk(s, topk); }
int status_of(cudaError_t e) { return from_cuda(e); }
}  // namespace phsa

extern "C" {

int phsa_build_block_repr(const void* K, const uint8_t* punct_mask, phsa_shape s, float lambda,
                          void* Krepr, void* stream) {
    int rc = check_shape(s, true);
    if (rc != PHSA_OK) return rc;
    if (!(lambda >= 0.f && lambda <= 1.f)) return PHSA_ERR_INVALID_ARG;
    if (empty(s) || s.L < s.block_size) return PHSA_OK;  // no full block: nothing to write
    if (!K || !punct_mask || !Krepr || !aligned16(K) || !aligned16(Krepr))
        return PHSA_ERR_INVALID_ARG;
    return from_cuda(phsa::launch_block_repr(K, punct_mask, s, lambda, Krepr,
                                             static_cast<cudaStream_t>(stream)));
}

int phsa_select_blocks(const void* Q, const void* Krepr, phsa_shape s, phsa_select_params p,
                       int32_t* block_idx, int32_t* block_cnt, void* stream) {
    int rc = check_shape(s, true);
    if (rc != PHSA_OK) return rc;
    if ((rc = check_topk(s, p.topk)) != PHSA_OK) return rc;
    if (p.n_init < 0 || p.n_local < 1 || p.topk < p.n_init + p.n_local) return PHSA_ERR_INVALID_ARG;
    if (p.aggregation != PHSA_AGG_SOFTMAX_SUM && p.aggregation != PHSA_AGG_MAX_LOGIT)
        return PHSA_ERR_INVALID_ARG;
    if (!(p.sm_scale > 0.f) || !isfinite(p.sm_scale)) return PHSA_ERR_INVALID_ARG;
    if (empty(s)) return PHSA_OK;
    const bool need_repr = s.L >= 2 * s.block_size;  // some query block has a candidate
    if (!Q || !block_idx || !block_cnt || !aligned16(Q) || (need_repr && (!Krepr || !aligned16(Krepr))))
        return PHSA_ERR_INVALID_ARG;
    if (phsa::select_smem_bytes(s, p.topk) > phsa::kMaxDynSmem) return PHSA_ERR_UNSUPPORTED;
    return from_cuda(phsa::launch_select_blocks(Q, Krepr, s, p, block_idx, block_cnt, status_ptr(),
                                                static_cast<cudaStream_t>(stream)));
}

int phsa_sparse_attn_fwd(const void* Q, const void* K, const void* V, const int32_t* block_idx,
                         const int32_t* block_cnt, phsa_shape s, int topk, float sm_scale,
                         void* O, float* lse, void* stream) {
    int rc = check_shape(s, true);
    if (rc != PHSA_OK) return rc;
    if ((rc = check_topk(s, topk)) != PHSA_OK) return rc;
    if (!(sm_scale > 0.f) || !isfinite(sm_scale)) return PHSA_ERR_INVALID_ARG;
    if (empty(s)) return PHSA_OK;
    if (!Q || !K || !V || !block_idx || !block_cnt || !O || !lse) return PHSA_ERR_INVALID_ARG;
    if (!aligned16(Q) || !aligned16(K) || !aligned16(V) || !aligned16(O))
        return PHSA_ERR_INVALID_ARG;
    int* st = status_ptr();
    if (!st) return PHSA_ERR_CUDA;
    return from_cuda(phsa::launch_attn_fwd(Q, K, V, block_idx, block_cnt, s, topk, sm_scale, O,
                                           lse, st, static_cast<cudaStream_t>(stream)));
}

size_t phsa_sparse_attn_bwd_workspace(phsa_shape s, int topk) {
    if (check_bwd(s, topk) != PHSA_OK) return 0;
    if (empty(s)) return 0;
    return phsa::bwd_layout(s, topk).total;
}

int phsa_sparse_attn_bwd(const void* Q, const void* K, const void* V, const void* O,
                         const void* dO, const float* lse, const int32_t* block_idx,
                         const int32_t* block_cnt, phsa_shape s, int topk, float sm_scale,
                         void* workspace, size_t workspace_bytes, void* dQ, void* dK, void* dV,
                         void* stream) {
    const int rc = check_bwd(s, topk);
    if (rc != PHSA_OK) return rc;
    if (!(sm_scale > 0.f) || !isfinite(sm_scale)) return PHSA_ERR_INVALID_ARG;
    if (empty(s)) return PHSA_OK;
    if (!Q || !K || !V || !O || !dO || !lse || !block_idx || !block_cnt || !dQ || !dK || !dV)
        return PHSA_ERR_INVALID_ARG;
    const void* ptrs[] = {Q, K, V, O, dO, dQ, dK, dV};
    for (const void* p : ptrs)
        if (!aligned16(p)) return PHSA_ERR_INVALID_ARG;
    if (!workspace || !aligned16(workspace) ||
        workspace_bytes < phsa::bwd_layout(s, topk).total)
        return PHSA_ERR_WORKSPACE;
    int* st = status_ptr();
    if (!st) return PHSA_ERR_CUDA;
    return from_cuda(phsa::launch_attn_bwd(Q, K, V, O, dO, lse, block_idx, block_cnt, s, topk,
                                           sm_scale, workspace, dQ, dK, dV, st,
                                           static_cast<cudaStream_t>(stream)));
}

int phsa_decode_update_repr(const void* K, const uint8_t* punct_mask, const int32_t* seq_lens,
                            phsa_shape s, float lambda, void* Krepr, void* stream) {
    int rc = check_shape(s, true);
    if (rc != PHSA_OK) return rc;
    if (!(lambda >= 0.f && lambda <= 1.f)) return PHSA_ERR_INVALID_ARG;
    if (empty(s) || s.L < s.block_size) return PHSA_OK;  // no block can fill
    if (!K || !punct_mask || !seq_lens || !Krepr || !aligned16(K) || !aligned16(Krepr))
        return PHSA_ERR_INVALID_ARG;
    int* st = status_ptr();
    if (!st) return PHSA_ERR_CUDA;
    return from_cuda(phsa::launch_decode_repr(K, punct_mask, seq_lens, s, lambda, Krepr, st,
                                              static_cast<cudaStream_t>(stream)));
}

int phsa_decode_select(const void* q, const void* Krepr, const int32_t* seq_lens, phsa_shape s,
                       phsa_select_params p, int32_t* block_idx, int32_t* block_cnt,
                       void* stream) {
    int rc = check_shape(s, true);
    if (rc != PHSA_OK) return rc;
    if ((rc = check_topk(s, p.topk)) != PHSA_OK) return rc;
    if (p.n_init < 0 || p.n_local < 1 || p.topk < p.n_init + p.n_local) return PHSA_ERR_INVALID_ARG;
    if (p.aggregation != PHSA_AGG_SOFTMAX_SUM && p.aggregation != PHSA_AGG_MAX_LOGIT)
        return PHSA_ERR_INVALID_ARG;
    if (!(p.sm_scale > 0.f) || !isfinite(p.sm_scale)) return PHSA_ERR_INVALID_ARG;
    if (empty(s)) return PHSA_OK;
    const bool need_repr = s.L >= 2 * s.block_size;  // some length can have a candidate
    if (!q || !seq_lens || !block_idx || !block_cnt || !aligned16(q) ||
        (need_repr && (!Krepr || !aligned16(Krepr))))
        return PHSA_ERR_INVALID_ARG;
    if (phsa::decode_select_smem_bytes(s, p.topk) > phsa::kMaxDynSmem) return PHSA_ERR_UNSUPPORTED;
    int* st = status_ptr();
    if (!st) return PHSA_ERR_CUDA;
    return from_cuda(phsa::launch_decode_select(q, Krepr, seq_lens, s, p, block_idx, block_cnt, st,
                                                static_cast<cudaStream_t>(stream)));
}

int phsa_decode_attn(const void* q, const void* K, const void* V, const int32_t* block_idx,
                     const int32_t* block_cnt, const int32_t* seq_lens, phsa_shape s, int topk,
                     float sm_scale, void* O, float* lse, void* stream) {
    int rc = check_shape(s, true);
    if (rc != PHSA_OK) return rc;
    if ((rc = check_topk(s, topk)) != PHSA_OK) return rc;
    if (!(sm_scale > 0.f) || !isfinite(sm_scale)) return PHSA_ERR_INVALID_ARG;
    if (s.B == 0) return PHSA_OK;
    if (!q || !K || !V || !block_idx || !block_cnt || !seq_lens || !O || !lse)
        return PHSA_ERR_INVALID_ARG;
    if (!aligned16(q) || !aligned16(K) || !aligned16(V) || !aligned16(O))
        return PHSA_ERR_INVALID_ARG;
    if (phsa::decode_attn_smem_bytes(s, topk) > phsa::kMaxDynSmem) return PHSA_ERR_UNSUPPORTED;
    int* st = status_ptr();
    if (!st) return PHSA_ERR_CUDA;
    return from_cuda(phsa::launch_decode_attn(q, K, V, block_idx, block_cnt, seq_lens, s, topk,
                                              sm_scale, O, lse, st,
                                              static_cast<cudaStream_t>(stream)));
}

int phsa_decode_step(const void* q, const void* K, const void* V, const uint8_t* punct_mask,
                     const int32_t* seq_lens, phsa_shape s, float lambda, phsa_select_params p,
                     void* Krepr, int32_t* block_idx, int32_t* block_cnt, void* O, float* lse,
                     void* stream) {
    int rc = check_shape(s, true);
    if (rc != PHSA_OK) return rc;
    if ((rc = check_topk(s, p.topk)) != PHSA_OK) return rc;
    if (!(lambda >= 0.f && lambda <= 1.f)) return PHSA_ERR_INVALID_ARG;
    if (p.n_init < 0 || p.n_local < 1 || p.topk < p.n_init + p.n_local) return PHSA_ERR_INVALID_ARG;
    if (p.aggregation != PHSA_AGG_SOFTMAX_SUM && p.aggregation != PHSA_AGG_MAX_LOGIT)
        return PHSA_ERR_INVALID_ARG;
    if (!(p.sm_scale > 0.f) || !isfinite(p.sm_scale)) return PHSA_ERR_INVALID_ARG;
    if (s.B == 0) return PHSA_OK;
    if (!q || !K || !V || !punct_mask || !seq_lens || !block_idx || !block_cnt || !O || !lse ||
        (s.L >= s.block_size && !Krepr))
        return PHSA_ERR_INVALID_ARG;
    if (!aligned16(q) || !aligned16(K) || !aligned16(V) || !aligned16(O) ||
        (Krepr && !aligned16(Krepr)))
        return PHSA_ERR_INVALID_ARG;
    if (phsa::decode_select_smem_bytes(s, p.topk) > phsa::kMaxDynSmem ||
        phsa::decode_attn_smem_bytes(s, p.topk) > phsa::kMaxDynSmem)
        return PHSA_ERR_UNSUPPORTED;
    int* st = status_ptr();
    if (!st) return PHSA_ERR_CUDA;
    cudaStream_t cs = static_cast<cudaStream_t>(stream);
    cudaError_t e = phsa::launch_decode_select(q, Krepr, seq_lens, s, p, block_idx, block_cnt, st, cs);
    if (e != cudaSuccess) return PHSA_ERR_CUDA;
    return from_cuda(phsa::launch_decode_attn_repr(q, K, V, block_idx, block_cnt, seq_lens, s,
                                                   p.topk, p.sm_scale, O, lse, punct_mask, lambda,
                                                   s.L >= s.block_size ? Krepr : nullptr, st,
                                                   cs));
}

int phsa_punct_mask(const int32_t* ids, int64_t n, const int32_t* punct_ids, int n_punct,
                    uint8_t* mask, void* stream) {
    if (n < 0 || n_punct < 0) return PHSA_ERR_INVALID_ARG;
    if (n_punct > 4096) return PHSA_ERR_UNSUPPORTED;
    if (n == 0) return PHSA_OK;
    if (!ids || !mask || (n_punct > 0 && !punct_ids)) return PHSA_ERR_INVALID_ARG;
    return from_cuda(phsa::launch_punct_mask(ids, n, punct_ids, n_punct, mask,
                                             static_cast<cudaStream_t>(stream)));
}

int phsa_decode_append(const void* k_new, const void* v_new, const uint8_t* flag_new,
                       const int32_t* seq_lens, phsa_shape s, void* K, void* V,
                       uint8_t* punct_mask, void* stream) {
    int rc = check_shape(s, true);
    if (rc != PHSA_OK) return rc;
    if (s.B == 0) return PHSA_OK;
    if (!k_new || !v_new || !seq_lens || !K || !V || (flag_new && !punct_mask))
        return PHSA_ERR_INVALID_ARG;
    if (!aligned16(k_new) || !aligned16(v_new) || !aligned16(K) || !aligned16(V))
        return PHSA_ERR_INVALID_ARG;
    int* st = status_ptr();
    if (!st) return PHSA_ERR_CUDA;
    return from_cuda(phsa::launch_decode_append(k_new, v_new, flag_new, seq_lens, s, K, V,
                                                punct_mask, st,
                                                static_cast<cudaStream_t>(stream)));
}

int phsa_prefill_append(const void* k_chunk, const void* v_chunk, const uint8_t* flag_chunk,
                        const int32_t* seq_lens, int chunk_len, phsa_shape s, float lambda,
                        void* K, void* V, uint8_t* punct_mask, void* Krepr, void* stream) {
    int rc = check_shape(s, true);
    if (rc != PHSA_OK) return rc;
    if (!(lambda >= 0.f && lambda <= 1.f)) return PHSA_ERR_INVALID_ARG;
    if (chunk_len < 0 || chunk_len > s.L) return PHSA_ERR_INVALID_ARG;
    if (s.B == 0 || chunk_len == 0) return PHSA_OK;
    if (!k_chunk || !v_chunk || !seq_lens || !K || !V || !punct_mask ||
        (s.L >= s.block_size && !Krepr))
        return PHSA_ERR_INVALID_ARG;
    if (!aligned16(k_chunk) || !aligned16(v_chunk) || !aligned16(K) || !aligned16(V) ||
        (Krepr && !aligned16(Krepr)))
        return PHSA_ERR_INVALID_ARG;
    int* st = status_ptr();
    if (!st) return PHSA_ERR_CUDA;
    return from_cuda(phsa::launch_prefill_append(k_chunk, v_chunk, flag_chunk, seq_lens, chunk_len,
                                                 s, lambda, K, V, punct_mask, Krepr, st,
                                                 static_cast<cudaStream_t>(stream)));
}

int phsa_get_device_status(void* stream) {
    if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess)
        return PHSA_ERR_CUDA;
    int* st = status_ptr();
    if (!st) return PHSA_ERR_CUDA;
    int v = 0;
    if (cudaMemcpy(&v, st, sizeof v, cudaMemcpyDeviceToHost) != cudaSuccess) return PHSA_ERR_CUDA;
    const int zero = 0;
    if (cudaMemcpy(st, &zero, sizeof zero, cudaMemcpyHostToDevice) != cudaSuccess)
        return PHSA_ERR_CUDA;
    return v;
}

int phsa_selftest_tcgen05(const void* A, const void* B, const void* V, float* S, float* O,
                          void* stream) {
    if (!A || !B || !V || !S || !O) return PHSA_ERR_INVALID_ARG;
    if (!aligned16(A) || !aligned16(B) || !aligned16(V)) return PHSA_ERR_INVALID_ARG;
    int* st = status_ptr();
    if (!st) return PHSA_ERR_CUDA;
    return from_cuda(phsa::launch_tc_selftest(A, B, V, S, O, st, static_cast<cudaStream_t>(stream)));
}

const char* phsa_status_string(int code) {
    switch (code) {
        case PHSA_OK: return "PHSA_OK";
        case PHSA_ERR_INVALID_ARG: return "PHSA_ERR_INVALID_ARG: invalid argument";
        case PHSA_ERR_UNSUPPORTED: return "PHSA_ERR_UNSUPPORTED: unsupported shape or parameter";
        case PHSA_ERR_CUDA: return "PHSA_ERR_CUDA: CUDA runtime error";
        case PHSA_ERR_TIMEOUT: return "PHSA_ERR_TIMEOUT: a bounded device wait expired";
        case PHSA_ERR_DEVICE_INDEX: return "PHSA_ERR_DEVICE_INDEX: invalid block index skipped";
        case PHSA_ERR_WORKSPACE: return "PHSA_ERR_WORKSPACE: workspace missing or too small";
        default: return "unknown phsa status";
    }
}

const char* phsa_version(void) { return "0.1.0"; }

}  // extern "C"
