// Stage (c) forward on the 5th-generation tensor cores (tcgen05 + TMEM + TMA),
// for GQA groups of two query heads (G*64 = 128 query rows per tile), at block
// sizes m = 64, 32 and 16.
//
// A unit is a 64-token span of one KV head: its 128 query rows (two heads x 64
// tokens) are the kSub = 64/m query blocks of the span. At m = 64 that is one
// query block and its selected blocks are the unit's key sequence. At m < 64
// the key sequence is the union of the span's kSub block lists (ascending), and
// each union entry carries an owner mask: which of the span's query blocks
// selected it. A 64-key tile holds kSub consecutive union entries (m rows of K
// and V each, gathered by TMA), and row r of query block j = (r mod 64) / m
// attends a tile slot only if bit j of its owner mask is set (and, in j's own
// block, only keys at or before its token). Padding slots past the union
// repeat its last block and are masked for every row.
//
// Persistent: two CTAs per SM, each walking the units (query block qb, KV
// head g) u = blockIdx.x, blockIdx.x + gridDim.x, ... with 256 threads in
// five roles; rings, TMEM buffers and barriers run on counters that continue
// across units, so one unit's loads and first MMAs overlap the previous
// unit's last blocks and epilogue:
//   warp 4             stages each unit's block list (at m < 64: the union and
//                      its owner masks, built by the whole warp through one
//                      bitmap per query block) into one of four list slots, a
//                      unit ahead; its lane 0 gathers the K tiles (64 x 128, by
//                      block index) into a two-slot ring; a slot is refilled as
//                      soon as the QK MMA that read it is done.
//   warp 6 (one lane)  loads each unit's Q tile (128 x 128) once the previous
//                      unit's last QK MMA is done, and the selected V tiles
//                      into their own two-slot ring, refilled when the PV MMA
//                      is done.
//   warp 5 (one lane)  MMA issuer: S_j = Q K_j^T (M=128, N=64, K=128) into one
//                      of two TMEM score buffers, and O += P_j V_j (M=128,
//                      N=128, K=64) with P_j read from TMEM. It polls and issues
//                      whichever is ready first, QK of block j+1 (once PV of
//                      block j-1 is issued) or PV of block j, so the tensor
//                      core works while the softmax of block j runs.
//   warps 0-3          softmax: thread r owns query row r (TMEM lane r). It
//                      loads its 64 scores, applies the causal mask inside the
//                      query's own block, keeps a running max and sum in the
//                      log2 domain, and writes P (bf16) over its scores in
//                      TMEM. O is rescaled in TMEM only when the block max
//                      exceeds the running max by more than 2^8 (exact: the
//                      final normalisation uses the same running max).
//                      Epilogue: O / l -> bf16 rows stored from registers;
//                      LSE = (max + log2 l) ln 2. O's TMEM columns are handed
//                      back to the next unit's first PV once read.
//   warp 7             idle (keeps the softmax warps on TMEM lane groups 0-3).
// TMEM: O in columns [0,128), score buffers in [128,192) and [192,256).
// Every wait is bounded in time (tc_common.cuh); on expiry the kernel records
// PHSA_ERR_TIMEOUT, drains its own copies and MMAs, frees TMEM and returns.
#include "phsa_common.cuh"
#include "phsa_internal.h"
#include "tc_common.cuh"
#include "union.cuh"

namespace phsa {

namespace {

using namespace tc;

constexpr int kSlots = 2;                   // K ring and V ring
constexpr int kHalfQ = 128 * 64 * 2;        // one 64-column half of the Q tile (16 KB)
constexpr int kQBytes = 2 * kHalfQ;         // 32 KB
constexpr int kKVHalf = 64 * 64 * 2;        // one 64-column half of a K or V block (8 KB)
constexpr int kKBytes = 2 * kKVHalf;        // 16 KB
constexpr int kOffQ = 0;
constexpr int kOffK = kQBytes;                        // K slots
constexpr int kOffV = kOffK + kSlots * kKBytes;       // V slots
constexpr int kOffBar = kOffV + kSlots * kKBytes;
// barriers
constexpr int B_Q = 0;                      // this unit's Q tile landed
constexpr int B_QFREE = 1;                  // the unit's last QK MMA is done
constexpr int B_KFULL = 2;                  // + slot
constexpr int B_KEMPTY = B_KFULL + kSlots;
constexpr int B_VFULL = B_KEMPTY + kSlots;
constexpr int B_VEMPTY = B_VFULL + kSlots;
constexpr int B_SFULL = B_VEMPTY + kSlots;  // + buffer
constexpr int B_PFULL = B_SFULL + 2;
constexpr int B_PVDONE = B_PFULL + 2;
constexpr int B_OFINAL = B_PVDONE + 1;      // the unit's last PV MMA is done
constexpr int B_OFREE = B_OFINAL + 1;       // the softmax warps have read O out
constexpr int kListSlots = 4;
constexpr int B_UFULL = B_OFREE + 1;        // + list slot
constexpr int B_UFREE = B_UFULL + kListSlots;
constexpr int B_DRAIN = B_UFREE + kListSlots;
constexpr int kNumBars = B_DRAIN + 1;
constexpr int kOffMisc = kOffBar + ((kNumBars * 8 + 15) & ~15);  // tmem base, abort flag
constexpr int kOffList = kOffMisc + 16;     // list slots: count, then the compacted list
constexpr int kThreads = 256;
constexpr int kUFreeCount = 3 + 128;        // K producer, V producer, MMA thread, softmax threads
constexpr uint32_t kTmemCols = 256;
constexpr uint32_t kColO = 0;
constexpr float kRescaleLog2 = 8.0f;
static_assert(kOffBar + kNumBars * 8 <= kOffMisc, "barrier region");

// A list slot: [0] the count n, then n block indices (capacity kSub * topk),
// then (kSub > 1) one owner-mask byte per entry.
__host__ __device__ constexpr int list_cap(int topk, int kSub) { return kSub * topk; }
__host__ __device__ constexpr int list_slot_ints(int topk, int kSub) {
    return (1 + list_cap(topk, kSub) + (kSub > 1 ? (list_cap(topk, kSub) + 3) / 4 : 0) + 3) & ~3;
}
// words of one query block's bitmap over the blocks [0, nqb)
__host__ __device__ constexpr int bitmap_words(int nqb) { return (nqb + 31) / 32; }
__host__ __device__ constexpr size_t fwd_tc_smem(int topk, int kSub, int nqb) {
    return 1024 + (size_t)kOffList + kListSlots * (size_t)list_slot_ints(topk, kSub) * 4 +
           (kSub > 1 ? (size_t)kSub * bitmap_words(nqb) * 4 : 0);
}

struct FwdTcArgs {
    const int32_t* idx;
    const int32_t* cnt;
    __nv_bfloat16* O;
    float* lse;
    int* status;
    int Hq, Hkv, L, NQB, topk, units;  // NQB: query blocks of m tokens
    int nsb;                           // 64-token spans per (b, g)
    float scale_log2;
};

struct FwdUnit {
    int qb, bg, hq0;
    long long lu;
};

// d.qb is the 64-token span (the query block itself at m = 64); d.lu the flat
// index of its first query block.
template <int kSub>
__device__ __forceinline__ FwdUnit fwd_unit(const FwdTcArgs& a, int u) {
    FwdUnit d;
    d.qb = a.nsb - 1 - (u % a.nsb);  // heaviest spans first
    d.bg = u / a.nsb;
    d.hq0 = (d.bg / a.Hkv) * a.Hq + (d.bg % a.Hkv) * 2;
    d.lu = (long long)d.bg * a.NQB + (long long)d.qb * kSub;
    return d;
}

// Warp-collective (all 32 lanes): the union of the block lists of the span's
// query blocks with owner masks (union.cuh) into a list slot; the
// per-query-block bitmaps over [0, NQB) are left cleared.
template <int kSub>
__device__ __forceinline__ void stage_union(const FwdTcArgs& a, const FwdUnit& d, int* sl,
                                            uint32_t* bm, int lane) {
    const int cap = list_cap(a.topk, kSub);
    build_block_union<kSub>(a.idx, a.cnt, d.lu, d.qb * kSub, min(kSub, a.NQB - d.qb * kSub), a.topk,
                            bm, bitmap_words(a.NQB), sl + 1, reinterpret_cast<uint8_t*>(sl + 1 + cap),
                            sl, a.status, lane);
    __threadfence_block();
    __syncwarp();
}

__device__ __forceinline__ uint32_t col_s(int buf) { return 128u + 64u * (uint32_t)buf; }

__device__ __forceinline__ uint4 shfl_xor4(const uint4& v, int m) {
    return make_uint4(__shfl_xor_sync(0xffffffffu, v.x, m), __shfl_xor_sync(0xffffffffu, v.y, m),
                      __shfl_xor_sync(0xffffffffu, v.z, m), __shfl_xor_sync(0xffffffffu, v.w, m));
}

// One round of a 4 x 4 transpose among lanes r and r ^ m: a lane with sel = 0
// keeps (a0, a1) and replaces (b0, b1) with its partner's (a0, a1); a lane
// with sel = 1 keeps (b0, b1) and replaces (a0, a1) with its partner's (b0, b1).
__device__ __forceinline__ void xchg_pieces(uint4& a0, uint4& a1, uint4& b0, uint4& b1, int sel,
                                            int m) {
    const uint4 r0 = shfl_xor4(sel ? a0 : b0, m);
    const uint4 r1 = shfl_xor4(sel ? a1 : b1, m);
    if (sel) {
        a0 = r0;
        a1 = r1;
    } else {
        b0 = r0;
        b1 = r1;
    }
}

template <int kSub>
__global__ void __launch_bounds__(kThreads, 2)
attn_fwd_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                   const __grid_constant__ CUtensorMap tmV, const FwdTcArgs a) {
    constexpr int kBm = 64 / kSub;  // block size m: rows of one gathered block
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~uintptr_t(1023));
    const uint32_t sb = smem_u32(smem);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    auto bar = [&](int i) { return sb + kOffBar + 8u * (uint32_t)i; };
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + kOffMisc + 4);
    const int lsi = list_slot_ints(a.topk, kSub);
    const int cap = list_cap(a.topk, kSub);
    // the K/V block of slot q of tile j of a list slot (padding repeats the last)
    auto tile_block = [&](const int* sl, int j, int q) {
        const int n = sl[0], ui = j * kSub + q;
        return sl[1 + (ui < n ? ui : n - 1)];
    };
    auto slot_ptr = [&](int k) {
        return reinterpret_cast<int*>(smem + kOffList) + (k % kListSlots) * lsi;
    };
    auto unit_of = [&](int k) { return (int)blockIdx.x + k * (int)gridDim.x; };

    if (threadIdx.x == 0) {
        mbar_init(bar(B_Q), 1);
        mbar_init(bar(B_QFREE), 1);
        for (int s = 0; s < kSlots; ++s) {
            mbar_init(bar(B_KFULL + s), 1);
            mbar_init(bar(B_KEMPTY + s), 1);
            mbar_init(bar(B_VFULL + s), 1);
            mbar_init(bar(B_VEMPTY + s), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar(B_SFULL + i), 1);
            mbar_init(bar(B_PFULL + i), 128);
        }
        for (int i = 0; i < kListSlots; ++i) {
            mbar_init(bar(B_UFULL + i), 1);
            mbar_init(bar(B_UFREE + i), kUFreeCount);
        }
        mbar_init(bar(B_PVDONE), 1);
        mbar_init(bar(B_OFINAL), 1);
        mbar_init(bar(B_OFREE), 128);
        mbar_init(bar(B_DRAIN), 1);
        fence_barrier_init();
        *abort_flag = 0;
    }
    if constexpr (kSub > 1) {  // the union bitmaps start cleared (stage_union leaves them so)
        uint32_t* bm = reinterpret_cast<uint32_t*>(smem + kOffList + (size_t)kListSlots * lsi * 4);
        for (int i = threadIdx.x; i < kSub * bitmap_words(a.NQB); i += kThreads) bm[i] = 0u;
    }
    if (warp == 5) {
        tmem_alloc(sb + kOffMisc, kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(smem + kOffMisc);

    if (warp == 4) {
        // ------------------------------------------------ lists and K tiles
        // At m = 64 lane 0 alone compacts each list; at m < 64 the whole warp builds
        // the union, so every lane runs this loop and lane 0 issues the copies.
        if (kSub > 1 || lane == 0) {
            if (lane == 0) prefetch_tmap(&tmK);
            uint32_t* bm = reinterpret_cast<uint32_t*>(smem + kOffList + (size_t)kListSlots * lsi * 4);
            // unit k's list into its slot, once every role is done with the slot's
            // previous unit (k - kListSlots)
            auto stage = [&](int k) {
                const int ls = k % kListSlots;
                bool ok1 = k < kListSlots ||
                           mbar_wait(bar(B_UFREE + ls), ((k / kListSlots) - 1) & 1, abort_flag, a.status);
                if constexpr (kSub > 1) ok1 = __all_sync(0xffffffffu, ok1);
                if (!ok1) return false;
                const FwdUnit d = fwd_unit<kSub>(a, unit_of(k));
                int* sl = slot_ptr(k);
                if constexpr (kSub == 1) {
                    sl[0] = compact_block_list(a.idx + d.lu * a.topk, a.cnt[d.lu], a.topk, d.qb,
                                               sl + 1, a.status);
                } else {
                    stage_union<kSub>(a, d, sl, bm, lane);
                }
                if (lane == 0) mbar_arrive(bar(B_UFULL + ls));
                return true;
            };
            bool ok = unit_of(0) >= a.units || stage(0);
            int gk = 0;  // K loads issued, over all units
            for (int k = 0; ok && unit_of(k) < a.units; ++k) {
                const FwdUnit d = fwd_unit<kSub>(a, unit_of(k));
                const int* sl = slot_ptr(k);
                const int nt = (sl[0] + kSub - 1) / kSub;  // 64-key tiles
                bool staged = false;  // the next unit's list, once this unit's ring is full
                for (int j = 0; j < nt; ++j, ++gk) {
                    if (j == kSlots && unit_of(k + 1) < a.units) {
                        if (!(ok = stage(k + 1))) break;
                        staged = true;
                    }
                    const int s = gk % kSlots;
                    bool okw = gk < kSlots ||
                               mbar_wait(bar(B_KEMPTY + s), ((gk / kSlots) - 1) & 1, abort_flag, a.status);
                    if constexpr (kSub > 1) okw = __all_sync(0xffffffffu, okw);
                    if (!okw) {
                        ok = false;
                        break;
                    }
                    if (lane == 0) {
                        mbar_expect_tx(bar(B_KFULL + s), kKBytes);
#pragma unroll
                        for (int q = 0; q < kSub; ++q) {
                            const int blk = tile_block(sl, j, q);
                            for (int dh = 0; dh < 2; ++dh)
                                tma_load_3d(sb + kOffK + s * kKBytes + dh * kKVHalf + q * kBm * 128, &tmK,
                                            bar(B_KFULL + s), dh * 64, blk * kBm, d.bg);
                        }
                    }
                }
                if (!ok) break;
                if (!staged && unit_of(k + 1) < a.units) ok = stage(k + 1);
                if (lane == 0) mbar_arrive(bar(B_UFREE + k % kListSlots));
            }
            // Own copies must have landed before the CTA may exit.
            if (lane == 0)
                for (int g = gk - kSlots; g < gk; ++g)
                    if (g >= 0) mbar_wait_drain(bar(B_KFULL + g % kSlots), (g / kSlots) & 1);
        }
    } else if (warp == 6) {
        // ------------------------------------------------ Q and V tiles
        if (lane == 0) {
            prefetch_tmap(&tmQ);
            prefetch_tmap(&tmV);
            int gv = 0, q_last = -1;  // V loads issued; last unit whose Q was loaded
            bool ok = true;
            for (int k = 0; ok && unit_of(k) < a.units; ++k) {
                const FwdUnit d = fwd_unit<kSub>(a, unit_of(k));
                ok = mbar_wait(bar(B_UFULL + k % kListSlots), (k / kListSlots) & 1, abort_flag, a.status);
                if (!ok) break;
                const int* sl = slot_ptr(k);
                const int n = (sl[0] + kSub - 1) / kSub;  // 64-key tiles
                // Q once the previous unit's last QK MMA has read the old tile
                if (k >= 1 && !mbar_wait(bar(B_QFREE), (k - 1) & 1, abort_flag, a.status)) {
                    ok = false;
                    break;
                }
                mbar_expect_tx(bar(B_Q), kQBytes);
                for (int hl = 0; hl < 2; ++hl)
                    for (int dh = 0; dh < 2; ++dh)
                        tma_load_3d(sb + kOffQ + dh * kHalfQ + hl * (kHalfQ / 2), &tmQ, bar(B_Q),
                                    dh * 64, d.qb * 64, d.hq0 + hl);
                q_last = k;
                for (int j = 0; j < n; ++j, ++gv) {
                    const int s = gv % kSlots;
                    if (gv >= kSlots &&
                        !mbar_wait(bar(B_VEMPTY + s), ((gv / kSlots) - 1) & 1, abort_flag, a.status)) {
                        ok = false;
                        break;
                    }
                    mbar_expect_tx(bar(B_VFULL + s), kKBytes);
#pragma unroll
                    for (int q = 0; q < kSub; ++q) {
                        const int blk = tile_block(sl, j, q);
                        for (int dh = 0; dh < 2; ++dh)
                            tma_load_3d(sb + kOffV + s * kKBytes + dh * kKVHalf + q * kBm * 128, &tmV,
                                        bar(B_VFULL + s), dh * 64, blk * kBm, d.bg);
                    }
                }
                if (!ok) break;
                mbar_arrive(bar(B_UFREE + k % kListSlots));
            }
            if (q_last >= 0) mbar_wait_drain(bar(B_Q), q_last & 1);
            for (int g = gv - kSlots; g < gv; ++g)
                if (g >= 0) mbar_wait_drain(bar(B_VFULL + g % kSlots), (g / kSlots) & 1);
        }
    } else if (warp == 5) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc_qk = idesc_bf16(128, 64, false);
            constexpr uint32_t idesc_pv = idesc_bf16(128, 128, true);
            const uint64_t dQ0 = sdesc_sw128(sb + kOffQ, 16, 1024);
            const uint64_t dK0 = sdesc_sw128(sb + kOffK, 16, 1024);
            const uint64_t dV0 = sdesc_sw128(sb + kOffV, kKVHalf, 1024);
            int g0 = 0;  // blocks of the previous units (QK and PV MMAs issued so far)
            bool ok = true;
            for (int k = 0; ok && unit_of(k) < a.units; ++k) {
                ok = mbar_wait(bar(B_UFULL + k % kListSlots), (k / kListSlots) & 1, abort_flag, a.status);
                if (!ok) break;
                const int n = (slot_ptr(k)[0] + kSub - 1) / kSub;  // 64-key tiles
                mbar_arrive(bar(B_UFREE + k % kListSlots));  // only the count is needed here
                ok = mbar_wait(bar(B_Q), k & 1, abort_flag, a.status);
                if (!ok) break;
                tc_fence_after();
                if (n == 0) {  // nothing to attend: keep the per-unit phases
                    mma_commit(bar(B_QFREE));
                    mma_commit(bar(B_OFINAL));
                    continue;
                }
                int nq = 0, np = 0;  // next QK and next PV of this unit
                Deadline dl;
                while (ok && np < n) {
                    bool progressed = false;
                    const int gq = g0 + nq, gv = g0 + np;
                    // QK_nq reuses score buffer gq&1, free once the PV two blocks back is issued.
                    if (nq < n && nq <= np + 1 &&
                        mbar_test_wait(bar(B_KFULL + gq % kSlots), (gq / kSlots) & 1)) {
                        tc_fence_after();
                        const uint64_t kd = sdesc_at(dK0, (gq % kSlots) * kKBytes);
                        const uint32_t d = tmem + col_s(gq & 1);
#pragma unroll
                        for (int ks = 0; ks < 8; ++ks)
                            mma_ss(d, sdesc_at(dQ0, (ks >> 2) * kHalfQ + (ks & 3) * 32),
                                   sdesc_at(kd, (ks >> 2) * kKVHalf + (ks & 3) * 32), idesc_qk,
                                   ks > 0 ? 1u : 0u);
                        mma_commit(bar(B_SFULL + (gq & 1)));
                        mma_commit(bar(B_KEMPTY + gq % kSlots));
                        ++nq;
                        if (nq == n) mma_commit(bar(B_QFREE));  // the Q tile may be replaced
                        progressed = true;
                    }
                    if (np < nq && mbar_test_wait(bar(B_PFULL + (gv & 1)), (gv >> 1) & 1)) {
                        // the first PV overwrites O: the previous unit's O must be read out
                        if ((np == 0 && k >= 1 &&
                             !mbar_wait(bar(B_OFREE), (k - 1) & 1, abort_flag, a.status)) ||
                            !mbar_wait(bar(B_VFULL + gv % kSlots), (gv / kSlots) & 1, abort_flag, a.status)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint64_t vd = sdesc_at(dV0, (gv % kSlots) * kKBytes);
                        const uint32_t pt = tmem + col_s(gv & 1);
#pragma unroll
                        for (int ks = 0; ks < 4; ++ks)
                            mma_ts(tmem + kColO, pt + ks * 8, sdesc_at(vd, ks * 2048), idesc_pv,
                                   (np > 0 || ks > 0) ? 1u : 0u);
                        mma_commit(bar(B_VEMPTY + gv % kSlots));
                        mma_commit(bar(B_PVDONE));
                        if (np == n - 1) mma_commit(bar(B_OFINAL));
                        ++np;
                        progressed = true;
                    }
                    if (progressed) {
                        dl.reset();
                    } else if (*abort_flag) {
                        ok = false;
                    } else if (dl.expired()) {
                        *abort_flag = 1;
                        atomicCAS(a.status, 0, PHSA_ERR_TIMEOUT);
                        ok = false;
                    }
                }
                g0 += n;
            }
            // Every MMA issued above must be complete before TMEM is freed.
            mma_commit(bar(B_DRAIN));
            mbar_wait_drain(bar(B_DRAIN), 0);
        }
    } else if (warp < 4) {
        // ------------------------------------------------ softmax + epilogue
        const int row = threadIdx.x;  // TMEM lane
        const int tok = row & 63, hl = row >> 6;
        const uint32_t lane_base = tmem + ((uint32_t)(warp * 32) << 16);
        int g0 = 0;
        bool ok = true;
        const int jr = tok / kBm, tb = tok % kBm;  // the row's query block in the span, position in it
        for (int k = 0; unit_of(k) < a.units; ++k) {
            const FwdUnit d = fwd_unit<kSub>(a, unit_of(k));
            ok = ok && mbar_wait(bar(B_UFULL + k % kListSlots), (k / kListSlots) & 1, abort_flag, a.status);
            ok = __all_sync(0xffffffffu, ok);
            if (!ok) break;
            const int* sl = slot_ptr(k);
            const int nu = sl[0];
            const int n = (nu + kSub - 1) / kSub;  // 64-key tiles
            const int* list = sl + 1;
            const uint8_t* own = reinterpret_cast<const uint8_t*>(sl + 1 + cap);
            const int qb_r = d.qb * kSub + jr;  // the row's query block
            float m_used = -INFINITY, l = 0.f;
            for (int j = 0; j < n; ++j) {
                const int g = g0 + j, buf = g & 1;
                ok = mbar_wait(bar(B_SFULL + buf), (g >> 1) & 1, abort_flag, a.status);
                ok = __all_sync(0xffffffffu, ok);
                if (!ok) break;
                tc_fence_after();
                uint32_t sr[64];
                tmem_ld64(lane_base + col_s(buf), sr);
                if constexpr (kSub == 1) {
                    if (list[j] == d.qb) {  // the query's own block: token-level causal mask
#pragma unroll
                        for (int c = 0; c < 64; ++c)
                            if (c > tok) sr[c] = __float_as_uint(-INFINITY);
                    }
                } else {
                    // slot q: attended if the row's query block selected its block; in
                    // the row's own block, only keys at or before its token
                    uint32_t full = 0u, part = 0u;
#pragma unroll
                    for (int q = 0; q < kSub; ++q) {
                        const int ui = j * kSub + q;
                        const bool sel = ui < nu && ((own[ui] >> jr) & 1u);
                        if (sel && list[ui] != qb_r) full |= 1u << q;
                        if (sel && list[ui] == qb_r) part |= 1u << q;
                    }
                    if (full != (1u << kSub) - 1u) {
#pragma unroll
                        for (int c = 0; c < 64; ++c) {
                            const int q = c / kBm;
                            const bool keep = ((full >> q) & 1u) || (((part >> q) & 1u) && c % kBm <= tb);
                            if (!keep) sr[c] = __float_as_uint(-INFINITY);
                        }
                    }
                }
                // row max of the raw scores (the scale is positive), three-input maxima
                float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
                for (int c = 0; c < 64; c += 2)
                    m4[(c >> 1) & 3] = fmax3(m4[(c >> 1) & 3], __uint_as_float(sr[c]), __uint_as_float(sr[c + 1]));
                const float mx = fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3])) * a.scale_log2;
                if (j == 0) {
                    m_used = mx;
                } else {
                    const bool need = mx > m_used + kRescaleLog2;
                    if (__any_sync(0xffffffffu, need)) {
                        // PV of the previous block must be complete before O is touched.
                        ok = mbar_wait(bar(B_PVDONE), (g - 1) & 1, abort_flag, a.status);
                        ok = __all_sync(0xffffffffu, ok);
                        if (!ok) break;
                        tc_fence_after();
                        const float f = need ? ex2_approx(m_used - mx) : 1.0f;
#pragma unroll 1
                        for (int c8 = 0; c8 < 8; ++c8) {
                            uint32_t o[16];
                            tmem_ld16(lane_base + kColO + 16 * c8, o);
#pragma unroll
                            for (int c = 0; c < 16; ++c) o[c] = __float_as_uint(__uint_as_float(o[c]) * f);
                            tmem_st16(lane_base + kColO + 16 * c8, o);
                        }
                        if (need) {
                            l *= f;
                            m_used = mx;
                        }
                    }
                }
                // p = 2^(s * scale_log2 - m): one packed FFMA per two scores and one SFU
                // op per score. P is packed in place: entry c (c < 32) takes the pair
                // (2c, 2c+1), both read before entry c is overwritten.
                float2 r2[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
                const float2 sc2 = make_float2(a.scale_log2, a.scale_log2);
                // a row with no attended key so far (m_used = -inf) has only masked
                // scores here: 2^(-inf) = 0 with a zero offset
                const float nm = m_used == -INFINITY ? 0.f : -m_used;
                const float2 nm2 = make_float2(nm, nm);
#pragma unroll
                for (int c = 0; c < 32; ++c) {
                    float2 p2 = __ffma2_rn(make_float2(__uint_as_float(sr[2 * c]), __uint_as_float(sr[2 * c + 1])), sc2, nm2);
                    p2.x = ex2_approx(p2.x);
                    p2.y = ex2_approx(p2.y);
                    r2[c & 1] = __fadd2_rn(r2[c & 1], p2);
                    sr[c] = pack2_bf16(p2.x, p2.y);
                }
                const float2 rr = __fadd2_rn(r2[0], r2[1]);
                const float rs = rr.x + rr.y;
                l += rs;
                tmem_st32(lane_base + col_s(buf), sr);
                tc_fence_before();
                mbar_arrive(bar(B_PFULL + buf));
            }
            if (!ok) break;
            mbar_arrive(bar(B_UFREE + k % kListSlots));  // the list is no longer read
            // Epilogue: the unit's O accumulation must be complete.
            ok = mbar_wait(bar(B_OFINAL), k & 1, abort_flag, a.status);
            ok = __all_sync(0xffffffffu, ok);
            if (!ok) break;
            tc_fence_after();
            const float inv = l > 0.f ? 1.0f / l : 0.f;
            const int i = d.qb * 64 + tok;
            // Rows go out through a 4 x 4 transpose of 16-byte pieces among each four
            // lanes (two rounds of xor shuffles): afterwards lane 4j + c holds piece c
            // of rows 4j .. 4j + 3, so a store instruction writes eight 64-byte row
            // segments instead of thirty-two 16-byte pieces.
            const int sel1 = (lane >> 1) & 1, sel0 = lane & 1;
#pragma unroll 1
            for (int c4 = 0; c4 < 4; ++c4) {
                uint32_t o[32];
                if (n > 0) {
                    tmem_ld32(lane_base + kColO + 32 * c4, o);
                } else {
#pragma unroll
                    for (int c = 0; c < 32; ++c) o[c] = 0u;
                }
                if (c4 == 3) {  // O is in registers: the next unit's first PV may overwrite it
                    tc_fence_before();
                    mbar_arrive(bar(B_OFREE));
                }
                uint4 x[4];
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    x[q].x = pack2_bf16(__uint_as_float(o[8 * q + 0]) * inv, __uint_as_float(o[8 * q + 1]) * inv);
                    x[q].y = pack2_bf16(__uint_as_float(o[8 * q + 2]) * inv, __uint_as_float(o[8 * q + 3]) * inv);
                    x[q].z = pack2_bf16(__uint_as_float(o[8 * q + 4]) * inv, __uint_as_float(o[8 * q + 5]) * inv);
                    x[q].w = pack2_bf16(__uint_as_float(o[8 * q + 6]) * inv, __uint_as_float(o[8 * q + 7]) * inv);
                }
                xchg_pieces(x[0], x[1], x[2], x[3], sel1, 2);  // rows r, r^2: halves of the pieces
                xchg_pieces(x[0], x[2], x[1], x[3], sel0, 1);  // rows r, r^1: single pieces
#pragma unroll
                for (int s4 = 0; s4 < 4; ++s4) {
                    const int r = warp * 32 + (lane & ~3) + s4;  // the row this piece belongs to
                    const int ri = d.qb * 64 + (r & 63);
                    if (ri < a.L)
                        reinterpret_cast<uint4*>(a.O + ((size_t)(d.hq0 + (r >> 6)) * a.L + ri) * 128)
                            [4 * c4 + (lane & 3)] = x[s4];
                }
            }
            if (i < a.L)
                a.lse[(size_t)(d.hq0 + hl) * a.L + i] = l > 0.f ? (m_used + log2f(l)) * kLn2 : -INFINITY;
            g0 += n;
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 5) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

}  // namespace

size_t attn_fwd_tc_smem_bytes(const phsa_shape& s, int topk) {
    const int bm = s.block_size;
    return fwd_tc_smem(topk, 64 / bm, (s.L + bm - 1) / bm);
}

cudaError_t launch_attn_fwd_tc(const void* Q, const void* K, const void* V, const int32_t* idx,
                               const int32_t* cnt, const phsa_shape& s, int topk, float sm_scale,
                               void* O, float* lse, int* status, cudaStream_t st) {
    const int bm = s.block_size, kSub = 64 / bm;
    const int NQB = (s.L + bm - 1) / bm, nsb = (s.L + 63) / 64;
    CUtensorMap tq, tk, tv;
    if (!make_tmap_bf16_rows128(&tq, Q, s.L, (uint64_t)s.B * s.Hq, 64) ||
        !make_tmap_bf16_rows128(&tk, K, s.L, (uint64_t)s.B * s.Hkv, (uint32_t)bm) ||
        !make_tmap_bf16_rows128(&tv, V, s.L, (uint64_t)s.B * s.Hkv, (uint32_t)bm))
        return cudaErrorInvalidValue;
    const size_t smem = fwd_tc_smem(topk, kSub, NQB);
    auto kern = kSub == 1 ? attn_fwd_tc_kernel<1> : kSub == 2 ? attn_fwd_tc_kernel<2> : attn_fwd_tc_kernel<4>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    if ((e = cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout, 100)) !=
        cudaSuccess)
        return e;
    int dev = 0, nsm = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
        return e;
    // Two CTAs per SM (shared memory and registers are sized for it); CTAs never
    // wait on one another, so the grid is correct whatever number is resident.
    const long long units = (long long)s.B * s.Hkv * nsb;
    const long long cap = 2LL * nsm;
    const unsigned grid = (unsigned)(units < cap ? units : cap);
    FwdTcArgs args{idx, cnt, static_cast<__nv_bfloat16*>(O), lse, status, s.Hq, s.Hkv, s.L, NQB,
                   topk, (int)units, nsb, sm_scale * kLog2e};
    ProfScope prof(K_FWD, st);
    kern<<<grid, kThreads, smem, st>>>(tq, tk, tv, args);
    return cudaGetLastError();
}

// ---------------------------------------------------------------- self-test
// One CTA runs the two MMA shapes of the kernel above on fixed operands:
//   S = A B^T (A: 128 x 128, B: 64 x 128, both K-major from TMA tiles),
//   O = bf16(S) V (bf16(S) written to TMEM, V: 64 x 128 as an MN-major B).
namespace {

__global__ void __launch_bounds__(128)
tc_selftest_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ CUtensorMap tmV, float* S, float* O, int* status) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~uintptr_t(1023));
    const uint32_t sb = smem_u32(smem);
    const int warp = threadIdx.x >> 5;
    const uint32_t sA = sb, sB = sb + kQBytes, sV = sB + kKBytes;
    const uint32_t bars = sV + kKBytes;  // 0: loads, 1: S done, 2: P stored, 3: O done
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + (bars - sb) + 64);
    if (threadIdx.x == 0) {
        for (int i = 0; i < 4; ++i) mbar_init(bars + 8 * i, i == 2 ? 128 : 1);
        fence_barrier_init();
        *abort_flag = 0;
    }
    if (warp == 0) {
        tmem_alloc(bars + 48, kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(smem + (bars - sb) + 48);
    bool ok = true;
    if (threadIdx.x == 0) {
        mbar_expect_tx(bars, kQBytes + 2 * kKBytes);
        for (int dh = 0; dh < 2; ++dh) {
            for (int hl = 0; hl < 2; ++hl)
                tma_load_3d(sA + dh * kHalfQ + hl * (kHalfQ / 2), &tmA, bars, dh * 64, hl * 64, 0);
            tma_load_3d(sB + dh * kKVHalf, &tmB, bars, dh * 64, 0, 0);
            tma_load_3d(sV + dh * kKVHalf, &tmV, bars, dh * 64, 0, 0);
        }
        ok = mbar_wait(bars, 0, abort_flag, status);
        if (!ok) mbar_wait_drain(bars, 0);  // the copies must land before exit
        tc_fence_after();
        if (ok) {
#pragma unroll
            for (int ks = 0; ks < 8; ++ks) {
                const uint32_t off = (uint32_t)((ks & 3) * 32);
                mma_ss(tmem + 128, sdesc_sw128(sA + (ks >> 2) * kHalfQ + off, 16, 1024),
                       sdesc_sw128(sB + (ks >> 2) * kKVHalf + off, 16, 1024),
                       idesc_bf16(128, 64, false), ks > 0 ? 1u : 0u);
            }
        }
        mma_commit(bars + 8);
    }
    ok = mbar_wait(bars + 8, 0, abort_flag, status);
    ok = __all_sync(0xffffffffu, ok);
    const int row = threadIdx.x;
    const uint32_t lane_base = tmem + ((uint32_t)(warp * 32) << 16);
    if (ok) {
        tc_fence_after();
        uint32_t sr[64];
        tmem_ld32(lane_base + 128, sr);
        tmem_ld32(lane_base + 160, sr + 32);
        for (int c = 0; c < 64; ++c) S[row * 64 + c] = __uint_as_float(sr[c]);
        uint32_t pk[32];
        for (int c = 0; c < 32; ++c)
            pk[c] = pack2_bf16(__uint_as_float(sr[2 * c]), __uint_as_float(sr[2 * c + 1]));
        tmem_st32(lane_base + 128, pk);
        tc_fence_before();
        mbar_arrive(bars + 16);
    }
    if (threadIdx.x == 0 && ok) {
        ok = mbar_wait(bars + 16, 0, abort_flag, status);
        tc_fence_after();
        if (ok) {
#pragma unroll
            for (int ks = 0; ks < 4; ++ks)
                mma_ts(tmem, tmem + 128 + ks * 8, sdesc_sw128(sV + ks * 2048, kKVHalf, 1024),
                       idesc_bf16(128, 128, true), ks > 0 ? 1u : 0u);
        }
        mma_commit(bars + 24);
    }
    ok = mbar_wait(bars + 24, 0, abort_flag, status);
    ok = __all_sync(0xffffffffu, ok);
    if (ok) {
        tc_fence_after();
        for (int c4 = 0; c4 < 4; ++c4) {
            uint32_t o[32];
            tmem_ld32(lane_base + 32 * c4, o);
            for (int c = 0; c < 32; ++c) O[row * 128 + 32 * c4 + c] = __uint_as_float(o[c]);
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

}  // namespace

cudaError_t launch_tc_selftest(const void* A, const void* B, const void* V, float* S, float* O,
                               int* status, cudaStream_t st) {
    CUtensorMap ta, tb, tv;
    if (!make_tmap_bf16_rows128(&ta, A, 128, 1, 64) || !make_tmap_bf16_rows128(&tb, B, 64, 1, 64) ||
        !make_tmap_bf16_rows128(&tv, V, 64, 1, 64))
        return cudaErrorInvalidValue;
    const size_t smem = 1024 + kQBytes + 2 * kKBytes + 256;
    cudaError_t e = cudaFuncSetAttribute(tc_selftest_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    tc_selftest_kernel<<<1, 128, smem, st>>>(ta, tb, tv, S, O, status);
    return cudaGetLastError();
}

}  // namespace phsa
