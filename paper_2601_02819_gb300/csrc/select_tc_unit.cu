// Stage (b) on the tensor cores for GQA pairs at block size 64 on sequences of
// up to 1024 query blocks: query-to-block relevance and Top-K selection (Eq. 8;
// Algorithm 1 step 3), one (query block qb, KV head g) unit at a time.
// Persistent: a CTA (352 threads, 2 per SM) walks the units u = blockIdx.x,
// blockIdx.x + gridDim.x, ... Two CTAs per SM keep two units' loads, MMAs and
// elementwise work in flight, which hides the short units' latencies better
// than the span-pair kernel of select_tc.cu (kept for longer sequences, whose
// candidate chunks that kernel loads once for two spans).
//
// The candidate representative keys C = [n_init, qb - n_local] stream through
// a two-slot shared-memory ring in chunks of 128 rows (TMA). Each chunk is
// used twice, and the scores never leave the SM:
//   pass 1  S = Q Kr^T   (M = 128 query rows, N = 128 candidates) in TMEM;
//           two threads per row (TMEM lane r, one per half of the columns)
//           keep a running max and sum of 2^(S*scale - max) (online
//           softmax); the halves are merged once, after the last chunk;
//   pass 2  S^T = Kr Q^T (M = 128 candidates, N = 128 rows) in TMEM;
//           two threads per candidate j (lane j, one per half of the rows)
//           sum p = 2^(S*scale - m_r - log2 Z_r) over their 64 rows in row order;
//           A[t] = half 0 + half 1. Every candidate follows the same order,
//           so equal candidates get bit-identical sums.
//   top-k   a dedicated warp, on a double-buffered copy of A, while the
//           elementwise warps already score the next unit: larger A first,
//           lower t on exact ties (topk.cuh).
// The max-logit rule (PHSA_AGG_MAX_LOGIT) needs no softmax statistics: it runs
// pass 2 alone, each thread taking the largest score of its candidate over its
// 64 rows (rows past L excluded), A[t] = max(half 0, half 1) * scale.
// Warps 0-7 do the elementwise work, warp 8 issues TMA, warp 9 the MMAs,
// warps 10 and 11 the top-k of alternate units (one warp's top-k of a long
// unit took longer than the elementwise warps' scoring of the next one). The
// ring, the TMEM buffers and every barrier run on counters that continue
// across units. Every wait is bounded in time.
#include "phsa_common.cuh"
#include "phsa_internal.h"
#include "tc_common.cuh"
#include "topk.cuh"

namespace phsa {

namespace {

using namespace tc;

constexpr int kCand = 128;                 // candidates per chunk
constexpr int kHalf = 128 * 64 * 2;        // 128 rows x 64 columns bf16 (16 KB)
constexpr int kTile = 2 * kHalf;           // 128 x 128 (32 KB)
constexpr int kOffQ = 0;
constexpr int kOffKr = kOffQ + kTile;      // 2 slots
constexpr int kOffStats = kOffKr + 2 * kTile;  // m + log2 Z [128], half partials m[2][128], z[2][128]
constexpr int kOffBar = kOffStats + 5 * 128 * 4;
constexpr int B_Q = 0, B_QFREE = 1, B_KFULL = 2, B_KEMPTY = 4, B_SFULL = 6, B_SFREE = 8,
              B_AFULL = 10, B_AFREE = 12, B_DRAIN = 14, kNumBars = 15;
constexpr int kOffMisc = kOffBar + kNumBars * 8;  // tmem base, abort flag
constexpr int kOffA = kOffMisc + 16;  // 2 buffers x (A0[NQB], A1[NQB]), then sel[2][topk]
constexpr int kThreads = 384;
constexpr uint32_t kTmemCols = 256;
constexpr int kRegKeys = 16;  // candidate keys per lane kept in registers by the top-k warps

// kSub query blocks of m = 64 / kSub tokens share a unit (the 64-token span):
// A holds two buffers of two halves (kSub = 1) or one buffer of kSub x two
// halves (kSub > 1, where the elementwise warps run the top-k themselves).
size_t select_tc_smem(int nqb, int topk, int kSub) {
    const size_t na = kSub == 1 ? 4 : (size_t)2 * kSub;
    return 1024 + (size_t)kOffA + na * nqb * 4 + (size_t)2 * topk * 4 + 16;
}

struct SelArgs {
    int32_t* idx_out;
    int32_t* cnt_out;
    int* status;
    int Hq, Hkv, L, T, NQB, topk, n_init, n_local, units, agg;
    float scale_log2, scale;
    int nsb;  // units per (b, g): query blocks (kSub = 1) or 64-token spans
};

// Everything about a unit that every role derives the same way.
struct SelUnit {
    int qb, bg, hq0, n_init_q, loc_lo, c_lo, c_hi, nC, nF, ksel, nch;
    long long lu;
    bool scored;  // false: the budget covers every candidate, nothing to score
};

__device__ __forceinline__ SelUnit sel_unit(const SelArgs& a, int u) {
    SelUnit d;
    d.qb = a.NQB - 1 - (u % a.NQB);  // heaviest query blocks first
    d.bg = u / a.NQB;
    d.hq0 = (d.bg / a.Hkv) * a.Hq + (d.bg % a.Hkv) * 2;
    d.lu = (long long)d.bg * a.NQB + d.qb;
    d.n_init_q = min(a.n_init, d.qb + 1);                // forced initial [0, n_init_q)
    d.loc_lo = max(d.n_init_q, d.qb - a.n_local + 1);    // forced local [loc_lo, qb]
    d.c_lo = a.n_init;                                   // candidates [c_lo, c_hi]
    d.c_hi = d.qb - a.n_local;
    d.nC = max(0, d.c_hi - d.c_lo + 1);
    d.nF = d.n_init_q + (d.qb - d.loc_lo + 1);
    d.ksel = a.topk - d.nF;
    d.scored = d.ksel < d.nC;
    d.nch = d.scored ? (d.nC + kCand - 1) / kCand : 0;  // chunks per pass
    return d;
}

// The chunk that step s of a unit with nch chunks per pass works on. Pass 2
// takes the last two chunks of pass 1 first: they are still in the ring's two
// slots (same slot parity, the ring alternates), so they are not loaded again;
// then chunks 0 .. nch - 3. Each chunk holds its own candidates, so the order
// of the chunks changes no sum.
__device__ __forceinline__ int step_chunk(int s, int nch, bool pass2_only) {
    if (pass2_only || s < nch) return s;
    const int j = s - nch;
    if (nch < 2) return 0;
    return j < 2 ? nch - 2 + j : j - 2;
}
// Step s reuses the chunk already in its slot (pass 2's first two steps).
__device__ __forceinline__ bool step_resident(int s, int nch, bool pass2_only) {
    return !pass2_only && nch >= 2 && s >= nch && s < nch + 2;
}

// Query block qb's forced sets and candidate range (Algorithm 1), any block size.
struct QbSel {
    int n_init_q, loc_lo, c_hi, nC, nF, ksel;
    bool scored;
};
__device__ __forceinline__ QbSel qb_sel(const SelArgs& a, int qb) {
    QbSel q;
    q.n_init_q = min(a.n_init, qb + 1);
    q.loc_lo = max(q.n_init_q, qb - a.n_local + 1);
    q.c_hi = qb - a.n_local;
    q.nC = max(0, q.c_hi - a.n_init + 1);
    q.nF = q.n_init_q + (qb - q.loc_lo + 1);
    q.ksel = a.topk - q.nF;
    q.scored = q.ksel < q.nC;
    return q;
}

// A unit of kSub > 1 query blocks: the span's union of candidate ranges is
// scored (that of its last query block); scored if any of them needs scoring.
template <int kSub>
__device__ __forceinline__ SelUnit sel_unit_k(const SelArgs& a, int u) {
    if constexpr (kSub == 1) {
        return sel_unit(a, u);
    } else {
        SelUnit d;
        d.qb = a.nsb - 1 - (u % a.nsb);  // the span; heaviest first
        d.bg = u / a.nsb;
        d.hq0 = (d.bg / a.Hkv) * a.Hq + (d.bg % a.Hkv) * 2;
        d.lu = (long long)d.bg * a.NQB + (long long)d.qb * kSub;
        const int last = min(a.NQB - 1, d.qb * kSub + kSub - 1);
        d.scored = false;
        for (int qb = d.qb * kSub; qb <= last; ++qb) d.scored |= qb_sel(a, qb).scored;
        d.c_lo = a.n_init;
        d.c_hi = last - a.n_local;
        d.nC = max(0, d.c_hi - d.c_lo + 1);
        d.n_init_q = d.loc_lo = d.nF = d.ksel = 0;  // per query block: qb_sel
        d.nch = d.scored ? (d.nC + kCand - 1) / kCand : 0;
        return d;
    }
}

// Writes query block qb's selection when its budget covers every candidate
// (threads t0, t0 + step, ...).
__device__ __forceinline__ void write_unscored(const SelArgs& a, int bg, int qb, const QbSel& q,
                                               int t0, int step) {
    int32_t* out = a.idx_out + ((long long)bg * a.NQB + qb) * a.topk;
    const int n = q.nF + q.nC;
    for (int j = t0; j < a.topk; j += step) {
        int v = -1;
        if (j < q.n_init_q) v = j;
        else if (j < q.n_init_q + q.nC) v = a.n_init + (j - q.n_init_q);
        else if (j < n) v = q.loc_lo + (j - q.n_init_q - q.nC);
        out[j] = v;
    }
    if (t0 == 0) a.cnt_out[(long long)bg * a.NQB + qb] = n;
}

template <bool kMaxLogit, int kSub>
__global__ void __launch_bounds__(kThreads, 2)
select_tc_unit_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmKr,
                 const SelArgs a) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~uintptr_t(1023));
    const uint32_t sb = smem_u32(smem);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    auto bar = [&](int i) { return sb + kOffBar + 8u * (uint32_t)i; };
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + kOffMisc + 4);
    float* m2s = reinterpret_cast<float*>(smem + kOffStats);  // per row: max + log2 of the sum
    float* pm = m2s + 128;  // [2][128] per-half running max (pass 1)
    float* pz = pm + 256;   // [2][128] per-half running sum
    float* Abuf = reinterpret_cast<float*>(smem + kOffA);  // [2][A0 | A1], NQB each
    int* sel0 = reinterpret_cast<int*>(smem + kOffA + (size_t)a.NQB * 4 * (kSub == 1 ? 4 : 2 * kSub));

    if (tid == 0) {
        mbar_init(bar(B_Q), 1);
        mbar_init(bar(B_QFREE), 1);
        for (int s = 0; s < 2; ++s) {
            mbar_init(bar(B_KFULL + s), 1);
            mbar_init(bar(B_KEMPTY + s), 1);
            mbar_init(bar(B_SFULL + s), 1);
            mbar_init(bar(B_SFREE + s), 256);
            mbar_init(bar(B_AFULL + s), 256);
            mbar_init(bar(B_AFREE + s), 1);
        }
        mbar_init(bar(B_DRAIN), 1);
        fence_barrier_init();
        *abort_flag = 0;
    }
    if (warp == 9) {
        tmem_alloc(sb + kOffMisc, kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(smem + kOffMisc);

    if (warp == 8) {
        // ------------------------------------------------ TMA producer
        if (lane == 0) {
            prefetch_tmap(&tmKr);
            prefetch_tmap(&tmQ);
            int gs = 0, su = 0, q_last = -1;  // chunk loads issued; scored units begun
            bool ok = true;
            for (int u = blockIdx.x; ok && u < a.units; u += gridDim.x) {
                const SelUnit d = sel_unit_k<kSub>(a, u);
                if (!d.scored) continue;
                const int steps = (kMaxLogit ? 1 : 2) * d.nch;
                for (int s = 0; ok && s < steps; ++s, ++gs) {
                    const int slot = gs & 1, c = step_chunk(s, d.nch, kMaxLogit);
                    if (gs >= 2 && !mbar_wait(bar(B_KEMPTY + slot), ((gs >> 1) - 1) & 1, abort_flag, a.status)) {
                        ok = false;
                        break;
                    }
                    if (step_resident(s, d.nch, kMaxLogit)) {
                        // the slot holds this chunk: its last reader is done (KEMPTY
                        // above), so the full phase completes without a copy
                        mbar_arrive(bar(B_KFULL + slot));
                        continue;
                    }
                    // four 8 KB boxes (64 rows x 64 columns): TMA moves them faster into one
                    // SM than two 16 KB boxes
                    mbar_expect_tx(bar(B_KFULL + slot), kTile);
                    for (int dh = 0; dh < 2; ++dh)
                        for (int rh = 0; rh < 2; ++rh)
                            tma_load_3d(sb + kOffKr + slot * kTile + dh * kHalf + rh * (kHalf / 2), &tmKr,
                                        bar(B_KFULL + slot), dh * 64, d.c_lo + c * kCand + 64 * rh, d.bg);
                    if (s == 0) {  // Q once the previous unit's last MMA has read the old one
                        if (su > 0 && !mbar_wait(bar(B_QFREE), (su - 1) & 1, abort_flag, a.status)) {
                            ok = false;
                            ++gs;
                            break;
                        }
                        mbar_expect_tx(bar(B_Q), kTile);
                        for (int hl = 0; hl < 2; ++hl)
                            for (int dh = 0; dh < 2; ++dh)
                                tma_load_3d(sb + kOffQ + dh * kHalf + hl * (kHalf / 2), &tmQ, bar(B_Q),
                                            dh * 64, d.qb * 64, d.hq0 + hl);
                        q_last = su;
                    }
                }
                ++su;
            }
            if (q_last >= 0) mbar_wait_drain(bar(B_Q), q_last & 1);
            for (int s = gs - 2; s < gs; ++s)
                if (s >= 0) mbar_wait_drain(bar(B_KFULL + (s & 1)), (s >> 1) & 1);
        }
    } else if (warp == 9) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_bf16(128, 128, false);
            const uint64_t dQ0 = sdesc_sw128(sb + kOffQ, 16, 1024);
            const uint64_t dKr0 = sdesc_sw128(sb + kOffKr, 16, 1024);
            int gs = 0, su = 0;
            bool ok = true;
            for (int u = blockIdx.x; ok && u < a.units; u += gridDim.x) {
                const SelUnit d = sel_unit_k<kSub>(a, u);
                if (!d.scored) continue;
                ok = mbar_wait(bar(B_Q), su & 1, abort_flag, a.status);
                tc_fence_after();
                const int steps = (kMaxLogit ? 1 : 2) * d.nch;
                for (int s = 0; ok && s < steps; ++s, ++gs) {
                    const int slot = gs & 1;
                    ok = mbar_wait(bar(B_KFULL + slot), (gs >> 1) & 1, abort_flag, a.status) &&
                         (gs < 2 || mbar_wait(bar(B_SFREE + slot), ((gs >> 1) - 1) & 1, abort_flag, a.status));
                    if (!ok) break;
                    tc_fence_after();
                    const uint64_t kr = sdesc_at(dKr0, slot * kTile);
                    const bool pass1 = !kMaxLogit && s < d.nch;
#pragma unroll
                    for (int ks = 0; ks < 8; ++ks) {
                        const uint32_t off = (uint32_t)((ks >> 2) * kHalf + (ks & 3) * 32);
                        const uint64_t dq = sdesc_at(dQ0, off);
                        const uint64_t dk = sdesc_at(kr, off);
                        // pass 1: rows x candidates; pass 2: candidates x rows
                        mma_ss(tmem + 128u * slot, pass1 ? dq : dk, pass1 ? dk : dq, idesc,
                               ks > 0 ? 1u : 0u);
                    }
                    mma_commit(bar(B_SFULL + slot));
                    mma_commit(bar(B_KEMPTY + slot));
                }
                if (ok) mma_commit(bar(B_QFREE));  // this unit's MMAs are all issued
                ++su;
            }
            mma_commit(bar(B_DRAIN));
            mbar_wait_drain(bar(B_DRAIN), 0);
        }
    } else if (warp >= 10) {
        // ------------------------------------------------ top-k (kSub = 1): warp 10 takes
        // the even scored units (A buffer 0), warp 11 the odd ones (buffer 1)
        const int tw = warp - 10;
        int* sel = sel0 + tw * a.topk;
        int su = 0;
        bool ok = kSub == 1;
        for (int u = blockIdx.x; ok && u < a.units; u += gridDim.x) {
            const SelUnit d = sel_unit_k<kSub>(a, u);
            int32_t* out = a.idx_out + d.lu * a.topk;
            if (!d.scored) {  // the budget covers every candidate
                if (tw != 0) continue;
                const int n = d.nF + d.nC;
                for (int j = lane; j < a.topk; j += 32) {
                    int v = -1;
                    if (j < d.n_init_q) v = j;
                    else if (j < d.n_init_q + d.nC) v = d.c_lo + (j - d.n_init_q);
                    else if (j < n) v = d.loc_lo + (j - d.n_init_q - d.nC);
                    out[j] = v;
                }
                if (lane == 0) a.cnt_out[d.lu] = n;
                continue;
            }
            const int buf = su & 1;
            if (buf != tw) {
                ++su;
                continue;
            }
            ok = mbar_wait(bar(B_AFULL + buf), (su >> 1) & 1, abort_flag, a.status);
            ok = __all_sync(0xffffffffu, ok);
            if (!ok) break;
            float* A0 = Abuf + (size_t)buf * 2 * a.NQB;
            float* A1 = A0 + a.NQB;
            // key = bits(A) << 32 | ~t, A = half 0 + half 1 (the same order for every
            // candidate) or, for max logits, the larger half; each lane holds its
            // candidates' keys in registers
            const int nC = d.nC, ksel = d.ksel, c_lo = d.c_lo;
            constexpr bool mx = kMaxLogit;
            auto key_of = [&](int cj) {
                return topk::make_key_agg(mx ? fmaxf(A0[cj], A1[cj]) : A0[cj] + A1[cj], c_lo + cj, mx);
            };
            if (nC <= 32 * kRegKeys) {
                unsigned long long key[kRegKeys];
#pragma unroll
                for (int r = 0; r < kRegKeys; ++r) {
                    const int cj = lane + 32 * r;
                    key[r] = cj < nC ? key_of(cj) : 0ull;
                }
                for (int k = 0; k < ksel; ++k) {
                    // the lane's largest key: a tree of depth 4 instead of a chain of 15
                    unsigned long long tr[kRegKeys / 2];
#pragma unroll
                    for (int r = 0; r < kRegKeys / 2; ++r) tr[r] = topk::umax64(key[r], key[r + kRegKeys / 2]);
#pragma unroll
                    for (int w = kRegKeys / 4; w >= 1; w >>= 1)
#pragma unroll
                        for (int r = 0; r < w; ++r) tr[r] = topk::umax64(tr[r], tr[r + w]);
                    const unsigned long long best = tr[0];
                    const unsigned mh = (unsigned)(best >> 32), ml = (unsigned)best;
                    const unsigned bh = __reduce_max_sync(0xffffffffu, mh);
                    const unsigned bl = __reduce_max_sync(0xffffffffu, mh == bh ? ml : 0u);
                    const unsigned long long win = ((unsigned long long)bh << 32) | bl;
                    if (lane == 0) sel[k] = topk::key_block(win);
#pragma unroll
                    for (int r = 0; r < kRegKeys; ++r)
                        if (key[r] == win) key[r] = 0ull;
                }
            } else {
                // a pick is marked by a NaN bit pattern that arithmetic never produces
                topk::rounds_one_warp(
                    nC, ksel, key_of, [&](int cj) { return __float_as_uint(A1[cj]) == 0xffffffffu; },
                    [&](int t) { A1[t - c_lo] = __uint_as_float(0xffffffffu); }, sel, lane);
            }
            __syncwarp();
            // A is no longer needed: the elementwise warps may refill this buffer
            if (lane == 0) mbar_arrive(bar(B_AFREE + buf));
            for (int j = lane; j < a.topk; j += 32) {
                if (j < d.n_init_q) out[j] = j;
                else if (j >= d.n_init_q + ksel && j < d.nF + ksel) out[j] = d.loc_lo + (j - d.n_init_q - ksel);
                else if (j >= d.nF + ksel) out[j] = -1;
            }
            for (int j = lane; j < ksel; j += 32) {
                const int v = sel[j];
                int rank = 0;
                for (int i = 0; i < ksel; ++i) rank += sel[i] < v;
                out[d.n_init_q + rank] = v;
            }
            if (lane == 0) a.cnt_out[d.lu] = d.nF + ksel;
            __syncwarp();  // sel is reused by the next unit
            ++su;
        }
    } else {
        // ------------------------------------------------ elementwise (8 warps)
        const uint32_t lane_base = tmem + ((uint32_t)((warp & 3) * 32) << 16);
        const int r = (warp & 3) * 32 + lane;  // pass 1: query row; pass 2: candidate
        const int hh = warp >> 2;              // half of the TMEM columns this thread reads
        bool ok = true;
        int gs = 0, su = 0;
        // After a failed wait the loops keep running without work, so that all eight
        // warps reach the named barriers after pass 1 the same number of times.
        const int et = threadIdx.x;  // 0..255 over the elementwise warps
        for (int u = blockIdx.x; u < a.units; u += gridDim.x) {
            const SelUnit d = sel_unit_k<kSub>(a, u);
            if constexpr (kSub > 1) {
                if (!d.scored) {  // every query block of the span is covered by its budget
                    for (int j = 0; j < kSub && d.qb * kSub + j < a.NQB; ++j)
                        write_unscored(a, d.bg, d.qb * kSub + j, qb_sel(a, d.qb * kSub + j), et, 256);
                    continue;
                }
            }
            if (!d.scored) continue;
            const int nch = d.nch, steps = (kMaxLogit ? 1 : 2) * nch, c_lo = d.c_lo, c_hi = d.c_hi, nC = d.nC;
            const bool row_ok = d.qb * 64 + (r & 63) < a.L;
            // pass 1: this row's own candidate bound (its query block's, at kSub > 1)
            const int c_hi_r = kSub == 1 ? c_hi : min(c_hi, d.qb * kSub + (r & 63) / (64 / kSub) - a.n_local);
            const int buf = kSub == 1 ? (su & 1) : 0;
            float* A0 = Abuf + (size_t)buf * 2 * a.NQB;
            float* A1 = A0 + a.NQB;
            if (kSub == 1 && ok && su >= 2) {  // the top-k warp is done with this buffer's previous unit
                ok = mbar_wait(bar(B_AFREE + buf), ((su >> 1) - 1) & 1, abort_flag, a.status);
                ok = __all_sync(0xffffffffu, ok);
            }
            float m = -INFINITY, z = 0.f;
            for (int s = 0; s < steps; ++s, ++gs) {
                const int slot = gs & 1, c = step_chunk(s, nch, kMaxLogit);
                if (ok) {
                    ok = mbar_wait(bar(B_SFULL + slot), (gs >> 1) & 1, abort_flag, a.status);
                    ok = __all_sync(0xffffffffu, ok);
                }
                if (ok) tc_fence_after();
                if (ok && !kMaxLogit && s < nch) {
                    // pass 1: row r against 64 candidates of the chunk, two loads of 32
                    const int t0 = c_lo + c * kCand + 64 * hh;
                    const bool full = t0 + 63 <= c_hi_r;
#pragma unroll 1
                    for (int q = 0; q < 2; ++q) {
                        if (t0 + 32 * q > c_hi) break;  // no candidate left in this group (warp-uniform)
                        uint32_t v[32];
                        tmem_ld32(lane_base + 128u * slot + 64 * hh + 32 * q, v);
                        // max of the raw scores (three-input maxima), then the scale (positive) once
                        float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
                        if (!full) {
#pragma unroll
                            for (int j = 0; j < 32; ++j)
                                if (t0 + 32 * q + j > c_hi_r) v[j] = __float_as_uint(-INFINITY);
                        }
#pragma unroll
                        for (int j = 0; j < 32; j += 2)
                            m4[(j >> 1) & 3] = fmax3(m4[(j >> 1) & 3], __uint_as_float(v[j]), __uint_as_float(v[j + 1]));
                        const float mn = fmaxf(m, fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3])) * a.scale_log2);
                        if (mn != -INFINITY) {
                            // packed: two scores per FFMA2 and FADD2, one SFU op each
                            const float2 cc = make_float2(a.scale_log2, a.scale_log2), nn = make_float2(-mn, -mn);
                            float2 s2[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
                            for (int j = 0; j < 32; j += 2) {
                                float2 e = __ffma2_rn(make_float2(__uint_as_float(v[j]), __uint_as_float(v[j + 1])), cc, nn);
                                e.x = ex2_approx(e.x);
                                e.y = ex2_approx(e.y);
                                s2[(j >> 1) & 1] = __fadd2_rn(s2[(j >> 1) & 1], e);
                            }
                            if (mn > m) z *= ex2_approx(m - mn);  // the running max moved
                            const float2 st = __fadd2_rn(s2[0], s2[1]);
                            z += st.x + st.y;
                            m = mn;
                        }
                    }
                    tc_fence_before();
                    mbar_arrive(bar(B_SFREE + slot));
                } else if (ok && kMaxLogit && kSub > 1) {
                    // max logit, per query block of the span: candidate r against the
                    // rows of half hh (head hh), kSub groups of 64 / kSub tokens
                    float mxs[kSub];
#pragma unroll
                    for (int sb = 0; sb < kSub; ++sb) mxs[sb] = -INFINITY;
                    if (c * kCand + (warp & 3) * 32 < nC) {
#pragma unroll
                        for (int q = 0; q < 2; ++q) {
                            uint32_t v[32];
                            tmem_ld32(lane_base + 128u * slot + 64 * hh + 32 * q, v);
                            const int tok0 = d.qb * 64 + 32 * q;
#pragma unroll
                            for (int j = 0; j < 32; ++j) {
                                constexpr int kTok = 64 / kSub;
                                const float x = tok0 + j < a.L ? __uint_as_float(v[j]) : -INFINITY;
                                mxs[(32 * q + j) / kTok] = fmaxf(mxs[(32 * q + j) / kTok], x);
                            }
                        }
                    }
                    tc_fence_before();
                    mbar_arrive(bar(B_SFREE + slot));
                    const int cj = c * kCand + r;
                    if (cj < nC) {
#pragma unroll
                        for (int sb = 0; sb < kSub; ++sb)
                            Abuf[(size_t)(2 * sb + hh) * a.NQB + cj] = mxs[sb] * a.scale;
                    }
                } else if (ok && !kMaxLogit && kSub > 1 && s >= nch) {
                    // pass 2, per query block of the span: the sums over its rows of
                    // head hh, in row order. Query block sb of the span has candidates
                    // up to qb*kSub + sb - n_local; this thread's candidate t past that
                    // bound takes no part in sb's sum (its 2^x is not evaluated).
                    const float* mrow = m2s + 64 * hh;
                    const int t_c = c_lo + c * kCand + r;
                    const int sb_bound = d.qb * kSub - a.n_local;  // + sb: query block sb's c_hi
                    float accs[kSub][2];
#pragma unroll
                    for (int sb = 0; sb < kSub; ++sb) accs[sb][0] = accs[sb][1] = 0.f;
                    if (c * kCand + (warp & 3) * 32 < nC) {
#pragma unroll
                        for (int q = 0; q < 2; ++q) {
                            uint32_t v[32];
                            tmem_ld32(lane_base + 128u * slot + 64 * hh + 32 * q, v);
#pragma unroll
                            for (int j = 0; j < 32; ++j) {
                                constexpr int kTok = 64 / kSub;
                                const int sb = (32 * q + j) / kTok;
                                if (t_c <= sb_bound + sb)
                                    accs[sb][j & 1] += ex2_approx(
                                        fmaf(__uint_as_float(v[j]), a.scale_log2, -mrow[32 * q + j]));
                            }
                        }
                    }
                    tc_fence_before();
                    mbar_arrive(bar(B_SFREE + slot));
                    const int cj = c * kCand + r;
                    if (cj < nC) {
#pragma unroll
                        for (int sb = 0; sb < kSub; ++sb)
                            Abuf[(size_t)(2 * sb + hh) * a.NQB + cj] = accs[sb][0] + accs[sb][1];
                    }
                } else if (ok && kMaxLogit) {
                    // max logit: candidate r against the 64 rows of half hh (head hh)
                    float mx4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
                    const bool live = c * kCand + (warp & 3) * 32 < nC;
#pragma unroll 1
                    for (int q = 0; q < (live ? 2 : 0); ++q) {
                        uint32_t v[32];
                        tmem_ld32(lane_base + 128u * slot + 64 * hh + 32 * q, v);
                        const int tok0 = d.qb * 64 + 32 * q;  // rows of head hh: tokens tok0 + j
                        const bool all_rows = tok0 + 31 < a.L;
#pragma unroll
                        for (int j = 0; j < 32; ++j) {
                            const float x = (all_rows || tok0 + j < a.L) ? __uint_as_float(v[j]) : -INFINITY;
                            mx4[j & 3] = fmaxf(mx4[j & 3], x);
                        }
                    }
                    tc_fence_before();
                    mbar_arrive(bar(B_SFREE + slot));
                    const int cj = c * kCand + r;
                    if (cj < nC)
                        (hh ? A1 : A0)[cj] = fmaxf(fmaxf(mx4[0], mx4[1]), fmaxf(mx4[2], mx4[3])) * a.scale;
                } else if (ok) {
                    // pass 2: candidate r against the 64 rows of half hh, in row order;
                    // a warp whose 32 candidates all lie past the last one skips the work
                    // p = 2^(S*scale - m_r - log2 Z_r): the row's max and sum in one offset
                    const float* mrow = m2s + 64 * hh;
                    float2 acc[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
                    const bool live = c * kCand + (warp & 3) * 32 < nC;
                    const float2 cc = make_float2(a.scale_log2, a.scale_log2);
#pragma unroll 1
                    for (int q = 0; q < (live ? 2 : 0); ++q) {
                        uint32_t vq[32];
                        tmem_ld32(lane_base + 128u * slot + 64 * hh + 32 * q, vq);
#pragma unroll
                        for (int j = 0; j < 32; j += 4) {
                            // -(m_r + log2 Z_r) of four rows, two per packed FFMA2
                            const float4 mm = *reinterpret_cast<const float4*>(mrow + 32 * q + j);
                            float2 e0 = __ffma2_rn(make_float2(__uint_as_float(vq[j]), __uint_as_float(vq[j + 1])), cc,
                                                   make_float2(-mm.x, -mm.y));
                            float2 e1 = __ffma2_rn(make_float2(__uint_as_float(vq[j + 2]), __uint_as_float(vq[j + 3])), cc,
                                                   make_float2(-mm.z, -mm.w));
                            e0.x = ex2_approx(e0.x);
                            e0.y = ex2_approx(e0.y);
                            e1.x = ex2_approx(e1.x);
                            e1.y = ex2_approx(e1.y);
                            acc[0] = __fadd2_rn(acc[0], e0);
                            acc[1] = __fadd2_rn(acc[1], e1);
                        }
                    }
                    tc_fence_before();
                    mbar_arrive(bar(B_SFREE + slot));
                    const int cj = c * kCand + r;
                    const float2 sacc = __fadd2_rn(acc[0], acc[1]);
                    if (cj < nC) (hh ? A1 : A0)[cj] = sacc.x + sacc.y;
                }
                if (!kMaxLogit && s == nch - 1) {
                    // merge the two column halves of every row: (m, z) -> max and 1/sum
                    pm[hh * 128 + r] = m;
                    pz[hh * 128 + r] = z;
                    named_barrier(1, 256);
                    if (hh == 0) {
                        const float ma = pm[r], mb = pm[128 + r];
                        const float mx = fmaxf(ma, mb);
                        const float za = ma == -INFINITY ? 0.f : pz[r] * ex2_approx(ma - mx);
                        const float zb = mb == -INFINITY ? 0.f : pz[128 + r] * ex2_approx(mb - mx);
                        const float zz = za + zb;
                        // a row past L (or without candidates) contributes 2^-inf = 0
                        m2s[r] = (row_ok && zz > 0.f) ? mx + log2f(zz) : INFINITY;
                    }
                    named_barrier(1, 256);
                }
            }
            if constexpr (kSub == 1) {
                if (ok) mbar_arrive(bar(B_AFULL + buf));  // this thread's A entries are written
            } else {
                // Top-k of each query block of the span, by the eight elementwise
                // warps: the two-level selection (topk.cuh) when it applies, else
                // one warp's rounds; every warp passes the same barriers.
                named_barrier(1, 256);  // every A entry of the span is written
                unsigned long long* fin = reinterpret_cast<unsigned long long*>(pm);  // 2 KB
                for (int j = 0; j < kSub; ++j) {
                    const int qb = d.qb * kSub + j;
                    if (qb >= a.NQB) break;
                    const QbSel q = qb_sel(a, qb);
                    if (!q.scored) {
                        write_unscored(a, d.bg, qb, q, et, 256);
                        continue;
                    }
                    float* Aj0 = Abuf + (size_t)(2 * j) * a.NQB;
                    float* Aj1 = Aj0 + a.NQB;
                    auto key_of = [&](int cj) {
                        return topk::make_key_agg(kMaxLogit ? fmaxf(Aj0[cj], Aj1[cj]) : Aj0[cj] + Aj1[cj],
                                                  c_lo + cj, kMaxLogit);
                    };
                    if (topk::two_level(q.nC, q.ksel)) {
                        topk::level1(q.nC, q.ksel, key_of, fin, warp, lane);
                        named_barrier(1, 256);
                        topk::level2(fin, q.ksel, sel0, et);
                    } else if (warp == 0) {
                        // a pick is marked by a NaN bit pattern that arithmetic never produces
                        topk::rounds_one_warp(
                            q.nC, q.ksel, key_of,
                            [&](int cj) { return __float_as_uint(Aj1[cj]) == 0xffffffffu; },
                            [&](int t) { Aj1[t - c_lo] = __uint_as_float(0xffffffffu); }, sel0, lane);
                    }
                    named_barrier(1, 256);
                    int32_t* out = a.idx_out + ((long long)d.bg * a.NQB + qb) * a.topk;
                    for (int x = et; x < a.topk; x += 256) {
                        if (x < q.n_init_q) out[x] = x;
                        else if (x >= q.n_init_q + q.ksel && x < q.nF + q.ksel) out[x] = q.loc_lo + (x - q.n_init_q - q.ksel);
                        else if (x >= q.nF + q.ksel) out[x] = -1;
                    }
                    for (int x = et; x < q.ksel; x += 256) {
                        const int v = sel0[x];
                        int rank = 0;
                        for (int i = 0; i < q.ksel; ++i) rank += sel0[i] < v;
                        out[q.n_init_q + rank] = v;
                    }
                    if (et == 0) a.cnt_out[(long long)d.bg * a.NQB + qb] = q.nF + q.ksel;
                    named_barrier(1, 256);  // sel and fin are reused
                }
            }
            ++su;
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 9) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

}  // namespace

size_t select_tc_unit_smem_bytes(const phsa_shape& s, int topk) {
    return select_tc_smem((s.L + 63) / 64, topk, 1);
}

cudaError_t launch_select_tc_unit(const void* Q, const void* Krepr, const phsa_shape& s,
                             const phsa_select_params& p, int32_t* idx, int32_t* cnt, int* status,
                             cudaStream_t st) {
    const int bm = s.block_size, kSub = 64 / bm;
    const int T = s.L / bm, NQB = (s.L + bm - 1) / bm;
    CUtensorMap tq, tkr;
    if (!make_tmap_bf16_rows128(&tq, Q, s.L, (uint64_t)s.B * s.Hq, 64)) return cudaErrorInvalidValue;
    // Krepr may be absent when no query block has a candidate (T < 2): the map is
    // then built over Q, which is never read through it.
    if (!make_tmap_bf16_rows128(&tkr, T > 0 ? Krepr : Q, T > 0 ? T : 1,
                                (uint64_t)s.B * s.Hkv, 64))
        return cudaErrorInvalidValue;
    const size_t smem = select_tc_smem(NQB, p.topk, kSub);
    const bool mx = p.aggregation == PHSA_AGG_MAX_LOGIT;
    if (kSub != 1) return cudaErrorInvalidValue;  // block size 64 only
    auto kern = mx ? select_tc_unit_kernel<true, 1> : select_tc_unit_kernel<false, 1>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    int dev = 0, nsm = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
        return e;
    const int nsb = kSub == 1 ? NQB : (NQB + kSub - 1) / kSub;
    const int units = s.B * s.Hkv * nsb;
    const int per_sm = smem * 2 + 2048 <= kMaxDynSmem + 1024 ? 2 : 1;  // two CTAs when shared memory allows
    SelArgs args{idx, cnt, status, s.Hq, s.Hkv, s.L, T, NQB, p.topk, p.n_init, p.n_local, units,
                 p.aggregation, p.sm_scale * kLog2e, p.sm_scale, nsb};
    ProfScope prof(K_SELECT, st);
    kern<<<(unsigned)min(units, per_sm * nsm), kThreads, smem, st>>>(tq, tkr, args);
    return cudaGetLastError();
}

}  // namespace phsa
