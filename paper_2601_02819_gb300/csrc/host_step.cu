// phsa_step_host: the whole path (stage (a), (b), the forward of (c) and its
// backward pass) for tensors in host memory. The copies in and out run on two
// streams owned by the library, one per direction, and are ordered against
// the kernels on the caller's stream by events, so that each stage starts as
// soon as its own inputs have arrived and each result leaves as soon as it is
// final. Per workspace the library keeps the events of the last call, so that
// a later call on the same workspace waits for it and calls on different
// workspaces overlap.
#include <mutex>
#include <unordered_map>

#include "phsa_common.cuh"
#include "phsa_internal.h"

namespace {

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

// Byte offsets of the device copies inside the caller's workspace.
struct StepLayout {
    size_t Q, K, V, dO, mask, Kr, idx, cnt, O, lse, dQ, dK, dV, bwd, total;
    size_t q_bytes, kv_bytes, mask_bytes, idx_bytes, cnt_bytes, lse_bytes;
};

StepLayout step_layout(const phsa_shape& s, int topk) {
    StepLayout l{};
    const size_t B = (size_t)s.B, L = (size_t)s.L, D = (size_t)s.D;
    const size_t T = L / (size_t)s.block_size, NQB = (L + s.block_size - 1) / s.block_size;
    l.q_bytes = B * s.Hq * L * D * 2;
    l.kv_bytes = B * s.Hkv * L * D * 2;
    l.mask_bytes = B * L;
    l.idx_bytes = B * s.Hkv * NQB * (size_t)topk * 4;
    l.cnt_bytes = B * s.Hkv * NQB * 4;
    l.lse_bytes = B * s.Hq * L * 4;
    size_t off = 0;
    auto take = [&](size_t bytes) {
        const size_t o = off;
        off = align256(off + bytes);
        return o;
    };
    l.Q = take(l.q_bytes);
    l.K = take(l.kv_bytes);
    l.V = take(l.kv_bytes);
    l.dO = take(l.q_bytes);
    l.mask = take(l.mask_bytes);
    l.Kr = take(B * s.Hkv * T * D * 2);
    l.idx = take(l.idx_bytes);
    l.cnt = take(l.cnt_bytes);
    l.O = take(l.q_bytes);
    l.lse = take(l.lse_bytes);
    l.dQ = take(l.q_bytes);
    l.dK = take(l.kv_bytes);
    l.dV = take(l.kv_bytes);
    l.bwd = take(phsa::bwd_layout(s, topk).total);
    l.total = off;
    return l;
}

constexpr int kMaxDevices = 64;

struct CopyStreams {
    cudaStream_t in = nullptr, out = nullptr;
};

// Events of the last call on one workspace: K and mask in, Q in, V in, dO
// in, forward done, dQ done, backward done, copies out done.
enum { E_K, E_Q, E_V, E_DO, E_FWD, E_DQ, E_BWD, E_DONE, kWsEvents };
struct WsEvents {
    bool used = false;
    cudaEvent_t e[kWsEvents] = {};
};

std::mutex g_mu;
CopyStreams g_streams[kMaxDevices];
std::unordered_map<const void*, WsEvents> g_ws;

cudaError_t copy_streams(int dev, CopyStreams& out) {
    CopyStreams& c = g_streams[dev];
    if (!c.in) {
        cudaError_t e = cudaStreamCreateWithFlags(&c.in, cudaStreamNonBlocking);
        if (e != cudaSuccess) return e;
        if ((e = cudaStreamCreateWithFlags(&c.out, cudaStreamNonBlocking)) != cudaSuccess) {
            cudaStreamDestroy(c.in);
            c.in = nullptr;
            return e;
        }
    }
    out = c;
    return cudaSuccess;
}

cudaError_t ws_events(const void* ws, WsEvents*& out) {
    auto it = g_ws.find(ws);
    if (it == g_ws.end()) {
        WsEvents ev;
        for (int i = 0; i < kWsEvents; ++i) {
            const cudaError_t e = cudaEventCreateWithFlags(&ev.e[i], cudaEventDisableTiming);
            if (e != cudaSuccess) {
                for (int j = 0; j < i; ++j) cudaEventDestroy(ev.e[j]);
                return e;
            }
        }
        it = g_ws.emplace(ws, ev).first;
    }
    out = &it->second;
    return cudaSuccess;
}

#define STEP_CK(call)                                   \
    do {                                                \
        if ((call) != cudaSuccess) return PHSA_ERR_CUDA; \
    } while (0)

}  // namespace

extern "C" {

size_t phsa_step_host_workspace(phsa_shape s, int topk) {
    if (phsa::validate_shape(s) != PHSA_OK || phsa::validate_topk(s, topk) != PHSA_OK) return 0;
    if (s.B == 0 || s.L == 0) return 0;
    return step_layout(s, topk).total;
}

int phsa_step_host(const void* Q, const void* K, const void* V, const void* dO,
                   const uint8_t* punct_mask, phsa_shape s, float lambda, phsa_select_params p,
                   void* O, float* lse, void* dQ, void* dK, void* dV, int32_t* block_idx,
                   int32_t* block_cnt, void* workspace, size_t workspace_bytes, void* done_event,
                   void* stream) {
    int rc = phsa::validate_shape(s);
    if (rc != PHSA_OK) return rc;
    if ((rc = phsa::validate_topk(s, p.topk)) != PHSA_OK) return rc;
    if (!(lambda >= 0.f && lambda <= 1.f)) return PHSA_ERR_INVALID_ARG;
    if (p.n_init < 0 || p.n_local < 1 || p.topk < p.n_init + p.n_local) return PHSA_ERR_INVALID_ARG;
    if (p.aggregation != PHSA_AGG_SOFTMAX_SUM && p.aggregation != PHSA_AGG_MAX_LOGIT)
        return PHSA_ERR_INVALID_ARG;
    if (!(p.sm_scale > 0.f) || !isfinite(p.sm_scale)) return PHSA_ERR_INVALID_ARG;
    if (phsa::select_smem_bytes(s, p.topk) > phsa::kMaxDynSmem) return PHSA_ERR_UNSUPPORTED;
    cudaStream_t cs = static_cast<cudaStream_t>(stream);
    cudaEvent_t done_ev = static_cast<cudaEvent_t>(done_event);
    if (s.B == 0 || s.L == 0) {
        if (done_ev) STEP_CK(cudaEventRecord(done_ev, cs));
        return PHSA_OK;
    }
    if (!Q || !K || !V || !dO || !punct_mask) return PHSA_ERR_INVALID_ARG;
    const StepLayout l = step_layout(s, p.topk);
    if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u) != 0 ||
        workspace_bytes < l.total)
        return PHSA_ERR_WORKSPACE;
    int* status = phsa::device_status_word();
    int dev = 0;
    if (!status || cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
        return PHSA_ERR_CUDA;

    std::lock_guard<std::mutex> lk(g_mu);
    CopyStreams cp;
    WsEvents* ev = nullptr;
    STEP_CK(copy_streams(dev, cp));
    STEP_CK(ws_events(workspace, ev));
    uint8_t* w = static_cast<uint8_t*>(workspace);
    auto in = [&](size_t off, const void* src, size_t bytes) {
        return cudaMemcpyAsync(w + off, src, bytes, cudaMemcpyHostToDevice, cp.in);
    };
    auto out = [&](void* dst, size_t off, size_t bytes) {
        return dst ? cudaMemcpyAsync(dst, w + off, bytes, cudaMemcpyDeviceToHost, cp.out)
                   : cudaSuccess;
    };

    // copies in, in the order the stages need them
    if (ev->used) STEP_CK(cudaStreamWaitEvent(cp.in, ev->e[E_DONE], 0));
    STEP_CK(in(l.K, K, l.kv_bytes));
    STEP_CK(in(l.mask, punct_mask, l.mask_bytes));
    STEP_CK(cudaEventRecord(ev->e[E_K], cp.in));
    STEP_CK(in(l.Q, Q, l.q_bytes));
    STEP_CK(cudaEventRecord(ev->e[E_Q], cp.in));
    STEP_CK(in(l.V, V, l.kv_bytes));
    STEP_CK(cudaEventRecord(ev->e[E_V], cp.in));
    STEP_CK(in(l.dO, dO, l.q_bytes));
    STEP_CK(cudaEventRecord(ev->e[E_DO], cp.in));

    // the kernels, each stage after its inputs
    int32_t* idx = reinterpret_cast<int32_t*>(w + l.idx);
    int32_t* cnt = reinterpret_cast<int32_t*>(w + l.cnt);
    float* lse_d = reinterpret_cast<float*>(w + l.lse);
    STEP_CK(cudaStreamWaitEvent(cs, ev->e[E_K], 0));
    if ((rc = phsa_build_block_repr(w + l.K, w + l.mask, s, lambda, w + l.Kr, cs)) != PHSA_OK)
        return rc;
    STEP_CK(cudaStreamWaitEvent(cs, ev->e[E_Q], 0));
    if ((rc = phsa_select_blocks(w + l.Q, w + l.Kr, s, p, idx, cnt, cs)) != PHSA_OK) return rc;
    STEP_CK(cudaStreamWaitEvent(cs, ev->e[E_V], 0));
    if ((rc = phsa_sparse_attn_fwd(w + l.Q, w + l.K, w + l.V, idx, cnt, s, p.topk, p.sm_scale,
                                   w + l.O, lse_d, cs)) != PHSA_OK)
        return rc;
    STEP_CK(cudaEventRecord(ev->e[E_FWD], cs));
    STEP_CK(cudaStreamWaitEvent(cs, ev->e[E_DO], 0));
    STEP_CK(phsa::launch_attn_bwd(w + l.Q, w + l.K, w + l.V, w + l.O, w + l.dO, lse_d, idx, cnt, s,
                                  p.topk, p.sm_scale, w + l.bwd, w + l.dQ, w + l.dK, w + l.dV,
                                  status, cs, ev->e[E_DQ]));
    STEP_CK(cudaEventRecord(ev->e[E_BWD], cs));

    // copies out, each result once it is final
    STEP_CK(cudaStreamWaitEvent(cp.out, ev->e[E_FWD], 0));
    STEP_CK(out(O, l.O, l.q_bytes));
    STEP_CK(out(lse, l.lse, l.lse_bytes));
    STEP_CK(out(block_idx, l.idx, l.idx_bytes));
    STEP_CK(out(block_cnt, l.cnt, l.cnt_bytes));
    STEP_CK(cudaStreamWaitEvent(cp.out, ev->e[E_DQ], 0));
    STEP_CK(out(dQ, l.dQ, l.q_bytes));
    STEP_CK(cudaStreamWaitEvent(cp.out, ev->e[E_BWD], 0));
    STEP_CK(out(dK, l.dK, l.kv_bytes));
    STEP_CK(out(dV, l.dV, l.kv_bytes));
    STEP_CK(cudaEventRecord(ev->e[E_DONE], cp.out));
    ev->used = true;
    if (done_ev)
        STEP_CK(cudaEventRecord(done_ev, cp.out));
    else
        STEP_CK(cudaStreamWaitEvent(cs, ev->e[E_DONE], 0));
    return PHSA_OK;
}

int phsa_step_host_release(void* workspace) {
    std::lock_guard<std::mutex> lk(g_mu);
    auto it = g_ws.find(workspace);
    if (it == g_ws.end()) return PHSA_OK;
    int rc = PHSA_OK;
    if (it->second.used && cudaEventSynchronize(it->second.e[E_DONE]) != cudaSuccess)
        rc = PHSA_ERR_CUDA;
    for (int i = 0; i < kWsEvents; ++i) cudaEventDestroy(it->second.e[i]);
    g_ws.erase(it);
    return rc;
}

}  // extern "C"
