// Optional per-kernel timing. When enabled, every kernel launch of the library
// is bracketed by two CUDA events recorded on its own stream; reading the
// records waits for those events and returns the accumulated time and launch
// count per kernel. Disabled (the default), the hooks cost one relaxed load.
#include <atomic>
#include <mutex>
#include <vector>

#include "phsa_internal.h"

namespace phsa {

namespace {

const char* const kNames[K_COUNT] = {
    "block_repr", "select_blocks", "attn_fwd", "bwd_delta", "bwd_idx_mark",
    "bwd_idx_build", "bwd_dkdv", "bwd_dkdv_sum", "bwd_dq", "decode_repr", "decode_select",
    "decode_attn", "prefill_append",
};

struct Record {
    int kid;
    cudaEvent_t start, stop;
};

std::atomic<bool> g_on{false};
std::mutex g_mu;
std::vector<Record> g_records;
std::vector<cudaEvent_t> g_pool;
thread_local cudaEvent_t t_start = nullptr;

cudaEvent_t take_event() {
    cudaEvent_t e = nullptr;
    {
        std::lock_guard<std::mutex> lk(g_mu);
        if (!g_pool.empty()) {
            e = g_pool.back();
            g_pool.pop_back();
        }
    }
    if (!e && cudaEventCreate(&e) != cudaSuccess) return nullptr;
    return e;
}

}  // namespace

void prof_begin(int kid, cudaStream_t st) {
    (void)kid;
    if (!g_on.load(std::memory_order_relaxed)) return;
    t_start = take_event();
    if (t_start) cudaEventRecord(t_start, st);
}

void prof_end(int kid, cudaStream_t st) {
    if (!g_on.load(std::memory_order_relaxed) || !t_start) return;
    cudaEvent_t stop = take_event();
    if (!stop) return;
    cudaEventRecord(stop, st);
    std::lock_guard<std::mutex> lk(g_mu);
    g_records.push_back({kid, t_start, stop});
    t_start = nullptr;
}

}  // namespace phsa

extern "C" {

int phsa_profile_enable(int on) {
    return phsa::g_on.exchange(on != 0) ? 1 : 0;
}

int phsa_profile_read(int max_kinds, const char** names, double* total_ms, int* launches) {
    using namespace phsa;
    std::vector<Record> recs;
    {
        std::lock_guard<std::mutex> lk(g_mu);
        recs.swap(g_records);
    }
    double ms_acc[K_COUNT] = {0};
    int n_acc[K_COUNT] = {0};
    int rc = K_COUNT;
    for (const Record& r : recs) {
        float ms = 0.f;
        if (cudaEventSynchronize(r.stop) != cudaSuccess ||
            cudaEventElapsedTime(&ms, r.start, r.stop) != cudaSuccess)
            rc = PHSA_ERR_CUDA;
        ms_acc[r.kid] += ms;
        n_acc[r.kid] += 1;
    }
    {
        std::lock_guard<std::mutex> lk(g_mu);
        for (const Record& r : recs) {
            g_pool.push_back(r.start);
            g_pool.push_back(r.stop);
        }
    }
    const int n = max_kinds < K_COUNT ? max_kinds : K_COUNT;
    for (int k = 0; k < n; ++k) {
        if (names) names[k] = kNames[k];
        if (total_ms) total_ms[k] = ms_acc[k];
        if (launches) launches[k] = n_acc[k];
    }
    return rc;
}

}  // extern "C"
