// Stage (c) backward on the tensor cores (tcgen05 + TMEM + TMA), for GQA
// groups of two query heads, so that every MMA has M = 128.
//
// dq_tc_kernel: persistent, one CTA per SM over the units (query block qb,
//   KV head g), 384 threads; rings and barriers continue across units. The
//   selected blocks are taken in pairs (an odd count pairs the last block with
//   a masked copy of itself); each pair's K and V tiles (128 keys) are gathered
//   by TMA into 3- and 2-slot rings. At the start of a unit its Q and dO tiles
//   are copied from their staging buffers into TMEM (tcgen05.cp), where they
//   are the A operands of S and dP; the staging buffers then load the next
//   unit's tiles, a whole unit ahead. Per pair p:
//     S_p  = Q Kp^T       (M128 N128 K128, A = Q in TMEM)
//     dP_p = dO Vp^T      (M128 N128 K128, A = dO in TMEM)
//     dS_p = P_p (dP_p - Delta), P_p = exp(S_p * scale - lse)   (8 warps, TMEM)
//     dQ  += dS_p Kp      (M128 N128 K128, A = dS_p in TMEM, B = Kp MN-major)
//   S and dP have one TMEM buffer each: S_{p+1} is computed as soon as the
//   elementwise warps hold S_p in registers, dP_{p+1} once dQ_p has read the
//   dS_p written over dP_p. dQ * scale is stored from registers. Before the
//   first pair the elementwise warps compute Delta_i = dO_i . O_i (O read from
//   global memory, dO from its staging tile) and write it for the dK/dV
//   kernel, which runs after this one. A fourth producer warp loads each
//   unit's Q and dO and stages the elementwise warps' copy of the unit's block
//   list before it arrives on the barrier that the Q tile completes.
//
// dkdv_tc_kernel: persistent, one CTA per SM over the work items (KV block t,
//   chunk of <= 32 query blocks that selected t), 352 threads; K_t and V_t are
//   reloaded per item as soon as its predecessor's S/dP MMAs are done, and the
//   dV^T/dK^T accumulators are double-buffered in TMEM. K_t and V_t stay in shared memory;
//   the Q and dO tiles (both heads stacked: 128 rows) of every listed query
//   block stream through a two-stage ring:
//     S  = Q K_t^T, dP = dO V_t^T            (M128 N64 K128; one MMA thread)
//     P, then dS (8 warps) -> shared memory  (bf16, 128 rows x 64 keys, two buffers)
//     dV^T += dO^T P, dK^T += Q^T dS          (M128 N64 K128; A = dO / Q read
//                                             MN-major, B = P / dS MN-major; a
//                                             second MMA thread)
//   Each product has its own barrier: P is formed while dP is still being
//   computed, and dV^T runs while dS is being formed. One issuing thread per
//   stream keeps either stream from waiting behind the other's 16 MMAs.
//   dK^T and dV^T live in TMEM with the head dimension on the lanes. A KV
//   block with a single chunk writes bf16 dK, dV straight from registers; a longer
//   list writes fp32 partials, and the chunk that finishes last (an atomic
//   counter per KV block) adds them in chunk order and stores the bf16 tile, so
//   the sum does not depend on which CTA finishes last.
//
// Every wait is bounded in time; on expiry the kernel records
// PHSA_ERR_TIMEOUT, drains its own copies and MMAs, frees TMEM and returns.
#include "phsa_common.cuh"
#include "phsa_internal.h"
#include "tc_common.cuh"

namespace phsa {

namespace {

using namespace tc;

constexpr int kHalf128 = 128 * 64 * 2;  // 128 rows x 64 columns, bf16 (16 KB)
constexpr int kHalf64 = 64 * 64 * 2;    // 64 rows x 64 columns (8 KB)
constexpr int kTile128 = 2 * kHalf128;  // 128 x 128 (32 KB)
constexpr int kTile64 = 2 * kHalf64;    // 64 x 128 (16 KB)
constexpr uint32_t kTmemCols = 512;

__device__ __forceinline__ uint32_t sw_off(int row, int chunk) {
    return (uint32_t)(row * 128 + ((chunk ^ (row & 7)) << 4));
}

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

// ============================================================== dQ
// Persistent: one CTA per SM walks the units (query block, KV head) u =
// blockIdx.x, blockIdx.x + gridDim.x, ...; the K/V rings, the S/dP buffers and
// every barrier run on counters that continue across units, so the next
// unit's Q/dO and first K/V pairs load while the current one finishes.
// Blocks are processed in pairs, so the S and dP MMAs have N = 128 keys.
namespace dq {
// Ring depths and shared-memory layout per block size: at m < 64 the K ring
// has two slots instead of three, so that the longer lists (the unions of a
// span's query-block lists, with owner masks) fit beside the tiles.
template <int kSub>
struct Cfg {
    static constexpr int kKSlots = kSub == 1 ? 3 : 2, kVSlots = 2;  // ring slots, one tile pair each
    static constexpr int kPair = 2 * kTile64;                        // two 64 x 128 tiles (32 KB)
    static constexpr int kOffQ = 0;
    static constexpr int kOffDO = kOffQ + kTile128;
    static constexpr int kOffK = kOffDO + kTile128;
    static constexpr int kOffV = kOffK + kKSlots * kPair;
    static constexpr int kOffBar = kOffV + kVSlots * kPair;
    // B_Q/B_DO: a unit's Q / dO tile is in its staging buffer; B_QFREE/B_DOFREE:
    // the staging buffer may be refilled (copied into TMEM, and seen by the
    // elementwise warps / read for Delta); B_O/B_OFREE: the unit's O tile is in
    // the Q staging buffer / has been read for Delta; B_SFULL/B_SFREE, B_DPFULL: the single
    // S and dP buffers in TMEM; B_DSFULL: dS is in TMEM (two barriers by pair parity)
    static constexpr int B_Q = 0, B_QFREE = 1, B_DO = 2, B_DOFREE = 3, B_O = 4, B_OFREE = 5, B_KFULL = 6,
                         B_KEMPTY = B_KFULL + kKSlots, B_VFULL = B_KEMPTY + kKSlots,
                         B_VEMPTY = B_VFULL + kVSlots, B_SFULL = B_VEMPTY + kVSlots,
                         B_SFREE = B_SFULL + 1, B_DPFULL = B_SFREE + 1, B_DSFULL = B_DPFULL + 1,
                         B_FINAL = B_DSFULL + 2, B_DQFREE = B_FINAL + 1, B_DRAIN = B_DQFREE + 1,
                         kNumBars = B_DRAIN + 1;
    static constexpr int kOffMisc = kOffBar + kNumBars * 8;
    static constexpr int kOffDPart = kOffMisc + 16;  // Delta of the 128 rows, fp32
    static constexpr int kOffList = kOffDPart + 128 * 4;  // block lists: 6 slots
};
constexpr int kListK = 0, kListV = 2, kListE = 4, kListSlots = 6;
constexpr int kThreads = 384;  // 8 elementwise warps, K producer, MMA, V producer, Q/dO producer
// TMEM: dQ [0,128), S [128,256), dP [256,384), the unit's Q [384,448) and dO
// [448,512) as bf16 A operands (copied from their staging tiles). dS of key
// half h overwrites dP columns [64h, 64h + 32) (read by the same thread).
constexpr uint32_t kColDQ = 0, kColS = 128, kColDP = 256, kColQ = 384, kColDO = 448;
// A list slot: the entries (capacity kSub * topk, one padding entry, the count
// in the last int of the entry region), then at m < 64 the owner masks (bytes).
__host__ __device__ constexpr int list_ints(int topk, int kSub) { return (kSub * topk + 2 + 15) & ~15; }
__host__ __device__ constexpr int slot_ints(int topk, int kSub) {
    return list_ints(topk, kSub) + (kSub > 1 ? (kSub * topk + 15) / 16 * 4 : 0);
}
template <int kSub>
constexpr size_t smem_bytes(int topk) {
    return 1024 + (size_t)Cfg<kSub>::kOffList + (size_t)kListSlots * slot_ints(topk, kSub) * 4;
}
}  // namespace dq

struct DqArgs {
    const int32_t* idx;
    const int32_t* cnt;
    const int32_t* ulist;   // m < 64: per span, the union of its query blocks' lists
    const int32_t* ucnt;
    const uint8_t* umask;   //         and the owner masks of its entries
    const float* lse;
    const __nv_bfloat16* O;
    float* delta;  // written: Delta_i = dO_i . O_i for every valid row
    __nv_bfloat16* dQ;
    int* status;
    int Hq, Hkv, L, NQB, topk, units;  // NQB: query blocks of m tokens
    int nsb, ucap;                     // 64-token spans per (b, g); union capacity
    float scale_log2, sm_scale;
};

// Copies one unit's block list row to shared memory with independent loads
// (one memory latency per 16 entries, the count fetched alongside) and
// compacts it there: -1 entries are skipped, and so is an entry outside
// [0, qb] or not above its predecessor (the rule of compact_block_list).
// Returns the number of valid blocks; out holds list_stride() ints.
__device__ __forceinline__ int stage_list(const int32_t* __restrict__ row,
                                          const int32_t* __restrict__ cntp, int topk, int qb,
                                          int* out) {
    const int cnt = __ldg(cntp);
    for (int j0 = 0; j0 < topk; j0 += 16) {
        int v[16];
#pragma unroll
        for (int k = 0; k < 16; ++k) v[k] = j0 + k < topk ? __ldg(row + j0 + k) : -1;
#pragma unroll
        for (int k = 0; k < 16; ++k)
            if (j0 + k < topk) out[j0 + k] = v[k];
    }
    const int n_raw = cnt < 0 ? 0 : min(cnt, topk);
    int k = 0, prev = -1;
    for (int j = 0; j < n_raw; ++j) {
        const int t = out[j];
        if (t == -1 || t < 0 || t > qb || t <= prev) continue;
        out[k++] = t;
        prev = t;
    }
    out[k] = k > 0 ? out[k - 1] : 0;  // an odd count pairs the last block with itself
    return k;
}

// A unit is a 64-token span of one (b, g) (the query block itself at m = 64);
// lu indexes its list row: idx/cnt at m = 64, the union rows at m < 64.
struct DqUnit {
    int qb, bg, hq0;
    long long lu;
};

template <int kSub>
__device__ __forceinline__ DqUnit dq_unit(const DqArgs& a, int u) {
    DqUnit d;
    d.qb = a.nsb - 1 - (u % a.nsb);  // heaviest spans first
    d.bg = u / a.nsb;
    d.hq0 = (d.bg / a.Hkv) * a.Hq + (d.bg % a.Hkv) * 2;
    d.lu = kSub == 1 ? (long long)d.bg * a.NQB + d.qb : (long long)d.bg * a.nsb + d.qb;
    return d;
}

// Copies a span's union list (already validated, ascending) to shared memory
// with independent loads, and its owner masks when mout is given. Returns the
// count; out[n] repeats the last entry.
__device__ __forceinline__ int stage_union_list(const DqArgs& a, long long row, int* out,
                                                uint8_t* mout) {
    const int n = min(__ldg(a.ucnt + row), a.ucap);
    const int32_t* src = a.ulist + row * a.ucap;
    for (int j0 = 0; j0 < n; j0 += 16) {
        int v[16];
#pragma unroll
        for (int k = 0; k < 16; ++k) v[k] = j0 + k < n ? __ldg(src + j0 + k) : 0;
#pragma unroll
        for (int k = 0; k < 16; ++k)
            if (j0 + k < n) out[j0 + k] = v[k];
    }
    if (mout)
        for (int j = 0; j < n; ++j) mout[j] = __ldg(a.umask + row * a.ucap + j);
    out[n] = n > 0 ? out[n - 1] : 0;
    return n;
}

// The unit's list into a slot (entries; masks too when mout is given).
template <int kSub>
__device__ __forceinline__ int stage_unit(const DqArgs& a, const DqUnit& d, int* out, uint8_t* mout) {
    if constexpr (kSub == 1)
        return stage_list(a.idx + d.lu * a.topk, a.cnt + d.lu, a.topk, d.qb, out);
    else
        return stage_union_list(a, d.lu, out, mout);
}

template <int kSub>
__global__ void __launch_bounds__(dq::kThreads, 1)
dq_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
             const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmdO,
             const __grid_constant__ CUtensorMap tmO, const DqArgs a) {
    using namespace dq;
    using C = Cfg<kSub>;
    constexpr int kMq = 64 / kSub;  // tokens of a query block (and keys of a KV block)
    const int li = list_ints(a.topk, kSub);  // entry ints of a list slot
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~uintptr_t(1023));
    const uint32_t sb = smem_u32(smem);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    auto bar = [&](int i) { return sb + C::kOffBar + 8u * (uint32_t)i; };
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::kOffMisc + 4);

    if (threadIdx.x == 0) {
        // Q's staging buffer is free once its copy into TMEM is done and the
        // elementwise warps have seen this unit's Q barrier (so that it cannot
        // complete twice before they wait on it); dO's once its copy is done and
        // the elementwise warps have read it for Delta
        mbar_init(bar(C::B_Q), 1);
        mbar_init(bar(C::B_QFREE), 257);
        mbar_init(bar(C::B_DO), 1);
        mbar_init(bar(C::B_DOFREE), 257);
        mbar_init(bar(C::B_O), 1);
        mbar_init(bar(C::B_OFREE), 256);
        for (int s = 0; s < C::kKSlots; ++s) {
            mbar_init(bar(C::B_KFULL + s), 1);
            mbar_init(bar(C::B_KEMPTY + s), 1);
        }
        for (int s = 0; s < C::kVSlots; ++s) {
            mbar_init(bar(C::B_VFULL + s), 1);
            mbar_init(bar(C::B_VEMPTY + s), 1);
        }
        mbar_init(bar(C::B_SFULL), 1);
        mbar_init(bar(C::B_SFREE), 256);
        mbar_init(bar(C::B_DPFULL), 1);
        mbar_init(bar(C::B_DSFULL), 256);
        mbar_init(bar(C::B_DSFULL + 1), 256);
        mbar_init(bar(C::B_FINAL), 1);
        mbar_init(bar(C::B_DQFREE), 256);
        mbar_init(bar(C::B_DRAIN), 1);
        fence_barrier_init();
        *abort_flag = 0;
    }
    if (warp == 9) {
        tmem_alloc(sb + C::kOffMisc, kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(smem + C::kOffMisc);

    if (warp == 8 || warp == 10) {
        // ------------------------------------------------ K and V producers (block pairs)
        if (lane == 0) {
            const bool is_k = warp == 8;
            const CUtensorMap* map = is_k ? &tmK : &tmV;
            const int slots = is_k ? C::kKSlots : C::kVSlots;
            const int full = is_k ? C::B_KFULL : C::B_VFULL, empty = is_k ? C::B_KEMPTY : C::B_VEMPTY;
            const uint32_t ring = sb + (is_k ? C::kOffK : C::kOffV);
            prefetch_tmap(map);
            const int ls = slot_ints(a.topk, kSub);
            int* lists = reinterpret_cast<int*>(smem + C::kOffList) + (is_k ? kListK : kListV) * ls;
            // Two list slots by unit parity. The next unit's list is staged once the
            // current unit's pairs are all issued, while the ring is still full, so
            // its memory latency stays off the load path.
            auto stage = [&](int u, int slot) {
                return stage_unit<kSub>(a, dq_unit<kSub>(a, u), lists + slot * ls, nullptr);
            };
            int n_cur = blockIdx.x < a.units ? stage(blockIdx.x, 0) : 0;
            int gp = 0;  // pairs issued so far, over all units
            bool ok = true;
            int ul = 0;
            for (int u = blockIdx.x; ok && u < a.units; u += gridDim.x, ++ul) {
                const DqUnit d = dq_unit<kSub>(a, u);
                const int* list = lists + (ul & 1) * ls;
                const int n = n_cur;
                const int np = ((n + kSub - 1) / kSub + 1) >> 1;  // pairs of 64-key tiles
                for (int p = 0; p < np; ++p, ++gp) {
                    const int s = gp % slots;
                    if (gp >= slots &&
                        !mbar_wait(bar(empty + s), ((gp / slots) - 1) & 1, abort_flag, a.status)) {
                        ok = false;
                        break;
                    }
                    mbar_expect_tx(bar(full + s), C::kPair);
                    // slot layout: [d half][tile of the pair][64 rows][64 columns]; a tile
                    // holds kSub blocks of kMq rows; entries past the list repeat its
                    // last block (masked by the consumer)
                    for (int h = 0; h < 2; ++h)
#pragma unroll
                        for (int q = 0; q < kSub; ++q) {
                            const int e = (2 * p + h) * kSub + q;
                            const int blk = list[e < n ? e : n - 1];
                            for (int dh = 0; dh < 2; ++dh)
                                tma_load_3d(ring + s * C::kPair + dh * kHalf128 + h * kHalf64 + q * kMq * 128,
                                            map, bar(full + s), dh * 64, blk * kMq, d.bg);
                        }
                }
                const int u2 = u + (int)gridDim.x;
                n_cur = ok && u2 < a.units ? stage(u2, (ul + 1) & 1) : 0;
            }
            for (int q = gp - slots; q < gp; ++q)
                if (q >= 0) mbar_wait_drain(bar(full + q % slots), (q / slots) & 1);
        }
    } else if (warp == 11) {
        // ------------------------------------------------ Q / dO / O producer
        // Per unit j, in this order: O_j into the Q staging buffer (once Q_{j-1}
        // has been copied into TMEM), dO_j into the dO staging buffer (once
        // dO_{j-1} has been copied and read for Delta), then Q_j over O_j once the
        // elementwise warps have taken Delta_j from both (during unit j - 1).
        if (lane == 0) {
            prefetch_tmap(&tmQ);
            prefetch_tmap(&tmdO);
            prefetch_tmap(&tmO);
            const int ls = slot_ints(a.topk, kSub);
            int* elists = reinterpret_cast<int*>(smem + C::kOffList) + kListE * ls;
            int ul = 0, last_q = -1, last_o = -1, last_do = -1;
            auto load_tile = [&](uint32_t dst, const CUtensorMap* map, uint32_t b, const DqUnit& d) {
                for (int hl = 0; hl < 2; ++hl)
                    for (int dh = 0; dh < 2; ++dh)
                        tma_load_3d(dst + dh * kHalf128 + hl * kHalf64, map, b, dh * 64, d.qb * 64, d.hq0 + hl);
            };
            for (int u = blockIdx.x; u < a.units; u += gridDim.x, ++ul) {
                const DqUnit d = dq_unit<kSub>(a, u);
                if (ul > 0 && !mbar_wait(bar(C::B_QFREE), (ul - 1) & 1, abort_flag, a.status)) break;
                mbar_expect_tx(bar(C::B_O), kTile128);
                load_tile(sb + C::kOffQ, &tmO, bar(C::B_O), d);
                last_o = ul;
                if (ul > 0 && !mbar_wait(bar(C::B_DOFREE), (ul - 1) & 1, abort_flag, a.status)) break;
                mbar_expect_tx(bar(C::B_DO), kTile128);
                load_tile(sb + C::kOffDO, &tmdO, bar(C::B_DO), d);
                last_do = ul;
                // this unit's and the next unit's tiles come from HBM: bring the next
                // unit's into L2 now
                const int u2 = u + (int)gridDim.x;
                if (u2 < a.units) {
                    const DqUnit d2 = dq_unit<kSub>(a, u2);
                    for (int hl = 0; hl < 2; ++hl)
                        for (int dh = 0; dh < 2; ++dh) {
                            tma_prefetch_3d(&tmO, dh * 64, d2.qb * 64, d2.hq0 + hl);
                            tma_prefetch_3d(&tmdO, dh * 64, d2.qb * 64, d2.hq0 + hl);
                            tma_prefetch_3d(&tmQ, dh * 64, d2.qb * 64, d2.hq0 + hl);
                        }
                }
                if (!mbar_wait(bar(C::B_OFREE), ul & 1, abort_flag, a.status)) break;
                // The tile first; then the elementwise warps' copy of the block list
                // (its slot's unit two back is done: they have passed the previous
                // unit's Q barrier), published by this thread's arrival on C::B_Q.
                mbar_expect_tx_only(bar(C::B_Q), kTile128);
                load_tile(sb + C::kOffQ, &tmQ, bar(C::B_Q), d);
                int* el = elists + (ul & 1) * ls;
                el[li - 1] = stage_unit<kSub>(a, d, el, reinterpret_cast<uint8_t*>(el + li));
                mbar_arrive(bar(C::B_Q));
                last_q = ul;
            }
            if (last_o >= 0) mbar_wait_drain(bar(C::B_O), last_o & 1);
            if (last_do >= 0) mbar_wait_drain(bar(C::B_DO), last_do & 1);
            if (last_q >= 0) mbar_wait_drain(bar(C::B_Q), last_q & 1);
        }
    } else if (warp == 9) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t id_s = idesc_bf16(128, 128, false);
            constexpr uint32_t id_dq = idesc_bf16(128, 128, true);
            const uint64_t dQ0 = sdesc_sw128(sb + C::kOffQ, 16, 1024);
            const uint64_t dDO0 = sdesc_sw128(sb + C::kOffDO, 16, 1024);
            const uint64_t dK0 = sdesc_sw128(sb + C::kOffK, 16, 1024);
            const uint64_t dKmn0 = sdesc_sw128(sb + C::kOffK, kHalf128, 1024);  // K read MN-major
            const uint64_t dV0 = sdesc_sw128(sb + C::kOffV, 16, 1024);
            // K step ks of a [d half][128 rows][64] tile: 16 columns of the head dimension
            auto koff = [](int ks) { return (uint32_t)((ks >> 2) * kHalf128 + (ks & 3) * 32); };
            auto issue_s = [&](int gp) {  // S = Q Kpair^T (A = Q in TMEM)
                const uint64_t kd = sdesc_at(dK0, (gp % C::kKSlots) * C::kPair);
#pragma unroll
                for (int ks = 0; ks < 8; ++ks)
                    mma_ts(tmem + kColS, tmem + kColQ + ks * 8, sdesc_at(kd, koff(ks)), id_s, ks > 0 ? 1u : 0u);
                mma_commit(bar(C::B_SFULL));
            };
            auto issue_dp = [&](int gp) {  // dP = dO Vpair^T (A = dO in TMEM); releases the V slot
                const uint64_t vd = sdesc_at(dV0, (gp % C::kVSlots) * C::kPair);
#pragma unroll
                for (int ks = 0; ks < 8; ++ks)
                    mma_ts(tmem + kColDP, tmem + kColDO + ks * 8, sdesc_at(vd, koff(ks)), id_s, ks > 0 ? 1u : 0u);
                mma_commit(bar(C::B_DPFULL));
                mma_commit(bar(C::B_VEMPTY + gp % C::kVSlots));
            };
            auto wait_k = [&](int gp) {
                return mbar_wait(bar(C::B_KFULL + gp % C::kKSlots), (gp / C::kKSlots) & 1, abort_flag, a.status);
            };
            auto wait_v = [&](int gp) {
                return mbar_wait(bar(C::B_VFULL + gp % C::kVSlots), (gp / C::kVSlots) & 1, abort_flag, a.status);
            };
            // S_gp reuses the S buffer once the elementwise warps hold S_{gp-1}
            auto wait_sfree = [&](int gp) {
                return gp == 0 || mbar_wait(bar(C::B_SFREE), (gp - 1) & 1, abort_flag, a.status);
            };
            // dP_gp reuses the dP buffer once dQ_{gp-1} has read the dS written over it
            // (its commit is the K slot's release)
            auto wait_dq_done = [&](int gp) {
                return gp == 0 || mbar_wait(bar(C::B_KEMPTY + (gp - 1) % C::kKSlots), ((gp - 1) / C::kKSlots) & 1,
                                            abort_flag, a.status);
            };
            bool ok = true;
            int gp0 = 0, ul = 0;
            // Per unit: Q and dO copied into TMEM, then S_0 dP_0 | S_1 | dS_0 -> dQ_0 |
            // dP_1 | S_2 | dS_1 -> dQ_1 | dP_2 ...
            // the unit's entry count, staged with its list by the Q/dO producer before
            // it arrives on C::B_Q (no global load on this thread's path)
            const int ls = slot_ints(a.topk, kSub);
            const int* elists = reinterpret_cast<const int*>(smem + C::kOffList) + kListE * ls;
            for (int u = blockIdx.x; ok && u < a.units; u += gridDim.x, ++ul) {
                // Q into TMEM once it has landed and the previous unit's last S has read
                // the previous Q; its staging buffer is then free for the next unit's
                ok = mbar_wait(bar(C::B_Q), ul & 1, abort_flag, a.status) &&
                     (gp0 == 0 || mbar_wait(bar(C::B_SFULL), (gp0 - 1) & 1, abort_flag, a.status));
                if (!ok) break;
                const int nu = elists[(ul & 1) * ls + li - 1];
                const int np = ((nu + kSub - 1) / kSub + 1) >> 1;
                tc_fence_after();
#pragma unroll
                for (int ks = 0; ks < 8; ++ks) tmem_cp_128x256b(tmem + kColQ + ks * 8, sdesc_at(dQ0, koff(ks)));
                mma_commit(bar(C::B_QFREE));
                // dO likewise, after the previous unit's last dP
                ok = mbar_wait(bar(C::B_DO), ul & 1, abort_flag, a.status) &&
                     (gp0 == 0 || mbar_wait(bar(C::B_DPFULL), (gp0 - 1) & 1, abort_flag, a.status));
                if (!ok) break;
                tc_fence_after();
#pragma unroll
                for (int ks = 0; ks < 8; ++ks) tmem_cp_128x256b(tmem + kColDO + ks * 8, sdesc_at(dDO0, koff(ks)));
                mma_commit(bar(C::B_DOFREE));
                if (np >= 1) {
                    ok = wait_k(gp0) && wait_sfree(gp0);
                    if (!ok) break;
                    tc_fence_after();
                    issue_s(gp0);
                    ok = wait_v(gp0) && wait_dq_done(gp0);
                    if (!ok) break;
                    tc_fence_after();
                    issue_dp(gp0);
                } else {
                    // the previous unit's dQ must be read out before FINAL completes again
                    ok = ul == 0 || mbar_wait(bar(C::B_DQFREE), (ul - 1) & 1, abort_flag, a.status);
                    if (!ok) break;
                    mma_commit(bar(C::B_FINAL));
                }
                for (int p = 0; ok && p < np; ++p) {
                    const int gp = gp0 + p;
                    if (p + 1 < np) {
                        ok = wait_k(gp + 1) && wait_sfree(gp + 1);
                        if (!ok) break;
                        tc_fence_after();
                        issue_s(gp + 1);
                    }
                    ok = mbar_wait(bar(C::B_DSFULL + (gp & 1)), (gp >> 1) & 1, abort_flag, a.status);
                    if (ok && p == 0 && ul > 0)  // dQ's accumulator: the previous unit is read out
                        ok = mbar_wait(bar(C::B_DQFREE), (ul - 1) & 1, abort_flag, a.status);
                    if (!ok) break;
                    tc_fence_after();
                    // dQ += dS Kpair: A = dS (TMEM, over dP), B = the K pair read MN-major
                    const uint64_t kmn = sdesc_at(dKmn0, (gp % C::kKSlots) * C::kPair);
#pragma unroll
                    for (int ks = 0; ks < 8; ++ks)
                        mma_ts(tmem + kColDQ, tmem + kColDP + (ks >> 2) * 64 + (ks & 3) * 8,
                               sdesc_at(kmn, ks * 2048), id_dq, (p > 0 || ks > 0) ? 1u : 0u);
                    mma_commit(bar(C::B_KEMPTY + gp % C::kKSlots));
                    if (p == np - 1) mma_commit(bar(C::B_FINAL));
                    if (p + 1 < np) {
                        ok = wait_v(gp + 1) && wait_dq_done(gp + 1);
                        if (!ok) break;
                        tc_fence_after();
                        issue_dp(gp + 1);
                    }
                }
                gp0 += np;
            }
            mma_commit(bar(C::B_DRAIN));
            mbar_wait_drain(bar(C::B_DRAIN), 0);
        }
    } else {
        // ------------------------------------------------ elementwise (8 warps)
        const int row = (warp & 3) * 32 + lane;  // TMEM lane
        const int half = warp >> 2;              // block of the pair (64 keys); d half for dQ
        const int tok = row & 63, hl = row >> 6;
        const uint32_t lane_base = tmem + ((uint32_t)((warp & 3) * 32) << 16);
        const int et = threadIdx.x;  // 0..255 over the elementwise warps
        const int pc = et & 15;      // 16-byte piece of a row in the Delta pass
        float* dpart = reinterpret_cast<float*>(smem + C::kOffDPart);
        bool ok = true;
        int gp0 = 0, ul = 0;
        const int ls = slot_ints(a.topk, kSub);
        int* lists = reinterpret_cast<int*>(smem + C::kOffList) + kListE * ls;
        // A unit's lse (for P) is fetched at the end of the previous unit; its block
        // list is staged by the producer before it arrives on C::B_Q.
        float neg_lse2 = 0.f;
        auto fetch_unit = [&](const DqUnit& d) {
            const int i = d.qb * 64 + tok;
            neg_lse2 = i < a.L ? -__ldg(a.lse + (size_t)(d.hq0 + hl) * a.L + i) * kLog2e : -INFINITY;
        };
        // Each unit's coordinates are worked out during the previous unit's wait for
        // its last dQ MMAs: their integer divisions (and the special-function unit
        // they use) stay off the unit boundary.
        DqUnit d_cur{};
        if (blockIdx.x < a.units) {
            d_cur = dq_unit<kSub>(a, blockIdx.x);
            fetch_unit(d_cur);
        }
        // Delta_i = dO_i . O_i of local unit ulx from its O tile (in the Q staging
        // buffer) and dO tile (in its own), both waited for here: the warps of d
        // half 0 take one row each over the whole head dimension. Returns this
        // thread's row's value. Every warp calls it once per unit, also after an
        // abort (doing no work then), so its named barrier is reached the same
        // number of times by all.
        auto delta_pass = [&](int ulx) -> float {
            if (ok) {
                ok = mbar_wait(bar(C::B_O), ulx & 1, abort_flag, a.status) &&
                     mbar_wait(bar(C::B_DO), ulx & 1, abort_flag, a.status);
                ok = __all_sync(0xffffffffu, ok);
            }
            if (ok && half == 0) {
                float acc = 0.f;
#pragma unroll
                for (int c = 0; c < 16; ++c) {
                    const uint32_t off = (uint32_t)((c >> 3) * kHalf128) + sw_off(row, c & 7);
                    const uint4 ov = *reinterpret_cast<const uint4*>(smem + C::kOffQ + off);
                    const uint4 dv = *reinterpret_cast<const uint4*>(smem + C::kOffDO + off);
                    const uint32_t ow[4] = {ov.x, ov.y, ov.z, ov.w};
                    const uint32_t dw[4] = {dv.x, dv.y, dv.z, dv.w};
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        const float2 fo = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&ow[j]));
                        const float2 fd = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&dw[j]));
                        acc = fmaf(fo.x, fd.x, acc);
                        acc = fmaf(fo.y, fd.y, acc);
                    }
                }
                dpart[row] = acc;
            }
            named_barrier(1, 256);  // Delta is visible
            const float v = dpart[row];
            // This thread is done with O, dO and Delta's exchange slots: Q may be
            // loaded over O, the next unit's dO loaded once dO has been copied, and
            // dpart rewritten once all have arrived.
            if (ok) {
                mbar_arrive(bar(C::B_OFREE));
                mbar_arrive(bar(C::B_DOFREE));
            }
            return v;
        };
        // Into L2: unit u's successor's lse (read at the end of unit u), and the
        // block list and count two units after it (staged a unit ahead).
        auto prefetch_ahead = [&](int u) {
            const int u1 = u + (int)gridDim.x, u3 = u + 2 * (int)gridDim.x;
            if (u1 < a.units) {
                const DqUnit d1 = dq_unit<kSub>(a, u1);
                const int r1 = et >> 1, i1 = d1.qb * 64 + (r1 & 63);
                if (i1 < a.L && (r1 & 31) == 0 && (et & 1) == 0)
                    prefetch_l2(a.lse + (size_t)(d1.hq0 + (r1 >> 6)) * a.L + i1);
            }
            if (u3 < a.units) {
                const DqUnit d3 = dq_unit<kSub>(a, u3);
                if constexpr (kSub == 1) {
                    if (et == 0) prefetch_l2(a.cnt + d3.lu);
                    if (et < 4 && et * 32 < a.topk) prefetch_l2(a.idx + d3.lu * a.topk + et * 32);
                    if (et == 4) prefetch_l2(a.idx + d3.lu * a.topk + a.topk - 1);
                } else {
                    if (et == 0) prefetch_l2(a.ucnt + d3.lu);
                    if (et < 8 && et * 32 < a.ucap) prefetch_l2(a.ulist + d3.lu * a.ucap + et * 32);
                }
            }
        };
        float dlt_next = 0.f;
        for (int u = blockIdx.x; u < a.units; u += gridDim.x, ++ul) {
            const int* list = lists + (ul & 1) * ls;
            const DqUnit d = d_cur;
            const int qb = d.qb;
            const int i = qb * 64 + tok;
            const bool valid = i < a.L;
            const size_t ridx = (size_t)(d.hq0 + hl) * a.L + (valid ? i : 0);
            const float nl2 = neg_lse2;
            if (ul == 0) prefetch_ahead(u);  // later units': during the previous unit's last dQ
            // Delta of the CTA's first unit here (its Q is loaded over its O only after
            // that); every later unit's was computed during the previous unit
            if (ul == 0) dlt_next = delta_pass(0);
            if (ok) {
                ok = mbar_wait(bar(C::B_Q), ul & 1, abort_flag, a.status);
                if (ok) mbar_arrive(bar(C::B_QFREE));
                ok = __all_sync(0xffffffffu, ok);
            }
            const float dlt = dlt_next;
            const int n = list[li - 1];
            const int nt = (n + kSub - 1) / kSub;  // 64-key tiles
            const int np = (nt + 1) >> 1;
            const uint8_t* own = reinterpret_cast<const uint8_t*>(list + li);
            const int jr = tok / kMq, tt = tok % kMq;  // the row's query block in the span, token in it
            const int qb_r = qb * kSub + jr;
            if (ok && half == 0 && valid) a.delta[ridx] = dlt;
            const int u2 = u + (int)gridDim.x;
            // the next unit's Delta, after pair pd of this one (its O and dO tiles
            // were loaded at the start of this unit)
            const int pd = min(2, np - 1);
            bool next_delta = u2 < a.units;
            for (int p = 0; ok && p < np; ++p) {
                const int gp = gp0 + p;
                ok = mbar_wait(bar(C::B_SFULL), gp & 1, abort_flag, a.status);
                ok = __all_sync(0xffffffffu, ok);
                if (!ok) break;
                tc_fence_after();
                const int tile = 2 * p + half;    // this half's tile of the pair
                // slot q of the tile: attended by the row if its query block selected
                // the slot's block (full), or only up to its token (part: its own block)
                uint32_t full = 0u, part = 0u;
#pragma unroll
                for (int q = 0; q < kSub; ++q) {
                    const int e = tile * kSub + q;
                    const bool sel = e < n && (kSub == 1 || ((own[e] >> jr) & 1u));
                    const bool mine = sel && list[e] == qb_r;
                    full |= (uint32_t)(sel && !mine) << q;
                    part |= (uint32_t)mine << q;
                }
                float pf[64];
                {
                    uint32_t sv[64];
                    tmem_ld64(lane_base + kColS + 64 * half, sv);
                    tc_fence_before();
                    mbar_arrive(bar(C::B_SFREE));  // S is in registers: the next S may be computed
                    // P = 2^(S scale_log2 - lse log2 e), two keys at a time (packed f32x2);
                    // the masks (the query's own block and the duplicate of an odd count)
                    // are warp-uniform branches off the main path
                    const float2 sc2 = make_float2(a.scale_log2, a.scale_log2);
                    const float2 nl2v = make_float2(nl2, nl2);
                    if (full == (1u << kSub) - 1u) {
#pragma unroll
                        for (int c = 0; c < 32; ++c) {
                            const float2 pv = __ffma2_rn(
                                make_float2(__uint_as_float(sv[2 * c]), __uint_as_float(sv[2 * c + 1])), sc2, nl2v);
                            pf[2 * c] = ex2_approx(pv.x);
                            pf[2 * c + 1] = ex2_approx(pv.y);
                        }
                    } else {
#pragma unroll
                        for (int c = 0; c < 32; ++c) {
                            const float2 pv = __ffma2_rn(
                                make_float2(__uint_as_float(sv[2 * c]), __uint_as_float(sv[2 * c + 1])), sc2, nl2v);
                            const int q0 = (2 * c) / kMq, q1 = (2 * c + 1) / kMq;
                            const bool k0 = ((full >> q0) & 1u) || (((part >> q0) & 1u) && (2 * c) % kMq <= tt);
                            const bool k1 = ((full >> q1) & 1u) || (((part >> q1) & 1u) && (2 * c + 1) % kMq <= tt);
                            pf[2 * c] = k0 ? ex2_approx(pv.x) : 0.f;
                            pf[2 * c + 1] = k1 ? ex2_approx(pv.y) : 0.f;
                        }
                    }
                }
                // dS = P (dP - Delta), written over this half's dP columns [64 half, +32)
                ok = mbar_wait(bar(C::B_DPFULL), gp & 1, abort_flag, a.status);
                ok = __all_sync(0xffffffffu, ok);
                if (!ok) break;
                tc_fence_after();
                const float2 ndl = make_float2(-dlt, -dlt);
                uint32_t dsv[32];
#pragma unroll
                for (int hh = 0; hh < 2; ++hh) {  // 32 keys at a time, for fewer live registers
                    uint32_t dp[32];
                    tmem_ld32(lane_base + kColDP + 64 * half + 32 * hh, dp);
#pragma unroll
                    for (int c = 0; c < 16; ++c) {
                        const float2 d = __fadd2_rn(make_float2(__uint_as_float(dp[2 * c]), __uint_as_float(dp[2 * c + 1])), ndl);
                        const float2 ds = __fmul2_rn(make_float2(pf[32 * hh + 2 * c], pf[32 * hh + 2 * c + 1]), d);
                        dsv[16 * hh + c] = pack2_bf16(ds.x, ds.y);
                    }
                }
                tmem_st32(lane_base + kColDP + 64 * half, dsv);
                tc_fence_before();
                mbar_arrive(bar(C::B_DSFULL + (gp & 1)));
                if (p == pd && next_delta) {
                    dlt_next = delta_pass(ul + 1);
                    next_delta = false;
                }
            }
            gp0 += np;
            if (next_delta) dlt_next = delta_pass(ul + 1);  // no pair reached pd (or an abort)
            if (u2 < a.units) {
                d_cur = dq_unit<kSub>(a, u2);
                fetch_unit(d_cur);  // the next unit's lse
            }
            if (u2 < a.units) prefetch_ahead(u2);  // while this unit's last dQ MMAs run
            if (ok) {
                ok = mbar_wait(bar(C::B_FINAL), ul & 1, abort_flag, a.status);
                ok = __all_sync(0xffffffffu, ok);
            }
            if (ok) {
                // dQ row `row`, columns [64 half, 64 half + 64): read out of TMEM in
                // one go, so that the next unit's dQ MMAs may start, then stored
                tc_fence_after();
                uint32_t o[64];
                if (n > 0) {
                    tmem_ld64(lane_base + kColDQ + 64 * half, o);
                } else {
#pragma unroll
                    for (int c = 0; c < 64; ++c) o[c] = 0u;
                }
                tc_fence_before();
                mbar_arrive(bar(C::B_DQFREE));
                // Rows go out through a 4 x 4 transpose of 16-byte pieces among each
                // four lanes (two rounds of xor shuffles): afterwards lane 4j + c holds
                // piece c of rows 4j .. 4j + 3 of a group of four pieces, so a store
                // instruction writes eight 64-byte row segments instead of thirty-two
                // 16-byte pieces of 32 different rows.
                const float s = a.sm_scale;
                const int sel1 = (lane >> 1) & 1, sel0 = lane & 1;
#pragma unroll
                for (int c4 = 0; c4 < 2; ++c4) {
                    uint4 x[4];
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        const int b = 32 * c4 + 8 * q;
                        x[q].x = pack2_bf16(__uint_as_float(o[b + 0]) * s, __uint_as_float(o[b + 1]) * s);
                        x[q].y = pack2_bf16(__uint_as_float(o[b + 2]) * s, __uint_as_float(o[b + 3]) * s);
                        x[q].z = pack2_bf16(__uint_as_float(o[b + 4]) * s, __uint_as_float(o[b + 5]) * s);
                        x[q].w = pack2_bf16(__uint_as_float(o[b + 6]) * s, __uint_as_float(o[b + 7]) * s);
                    }
                    xchg_pieces(x[0], x[1], x[2], x[3], sel1, 2);  // rows r, r^2: halves of the pieces
                    xchg_pieces(x[0], x[2], x[1], x[3], sel0, 1);  // rows r, r^1: single pieces
#pragma unroll
                    for (int s4 = 0; s4 < 4; ++s4) {
                        const int r = (warp & 3) * 32 + (lane & ~3) + s4;  // the row of piece x[s4]
                        const int ri = qb * 64 + (r & 63);
                        if (ri < a.L)
                            reinterpret_cast<uint4*>(a.dQ + ((size_t)(d.hq0 + (r >> 6)) * a.L + ri) * 128)
                                [8 * half + 4 * c4 + (lane & 3)] = x[s4];
                    }
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 9) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

// ============================================================== dK / dV
// Persistent: one CTA per SM takes work items (KV block t of one (b, g), chunk
// of <= 32 query blocks that selected t) from a global queue by tickets from
// one counter. The queue (built by idx_build) holds the items of >= 4
// iterations, (b, g) after (b, g) and longest first within each, then the
// short ones: the Q/dO tiles of the (b, g) in progress stay in L2 and the SMs
// end together on short items.
// The producer thread takes the tickets and hands each item to the MMA and
// elementwise roles through a ring in shared memory. K_t/V_t are reloaded as
// soon as the previous item's last S/dP MMAs are done, the Q/dO ring, the S/dP
// and P/dS buffers run on counters that continue across items, and the
// dV^T/dK^T accumulators are double-buffered in TMEM, so an item's epilogue
// overlaps the next item's work.
namespace kv {
constexpr int kOffK = 0;
constexpr int kOffV = kOffK + kTile64;
// Q and dO tiles (128 rows x 128 columns, 32 KB each) stream through a ring of
// kSlots half-slots in the order Q_0, dO_0, Q_1, dO_1, ...: load l of the CTA
// goes to slot l % kSlots. dO_i is released by the dV^T MMAs of iteration i,
// Q_i by its dK^T MMAs, so the next iterations' tiles load while one finishes.
constexpr int kSlots = 5;
constexpr int kOffSlot = kOffV + kTile64;
// P and dS [128 rows][64 keys] bf16, one buffer each
constexpr int kOffP = kOffSlot + kSlots * kTile128;
constexpr int kOffDS = kOffP + kHalf128;
constexpr int kOffBar = kOffDS + kHalf128;
constexpr int kRing = 8;  // item descriptors in flight
// Barriers (pairs are indexed by iteration parity or accumulator buffer):
//   KV/KVFREE     K_t, V_t landed / the item's last dP has read them
//   HFULL/HEMPTY  a half-slot has landed / its last MMA is done (kSlots each)
//   SFULL/DPFULL  S / dP of the iteration are in TMEM
//   PFULL/DSFULL  the elementwise warps have read S / dP and stored P / dS
//   PFREE/DSFREE  the dV^T / dK^T MMAs that read P / dS are done
//   FINAL/DKVFREE an item's accumulators are complete / have been read
constexpr int B_KV = 0, B_KVFREE = 1, B_HFULL = 2, B_HEMPTY = B_HFULL + kSlots,
              B_SFULL = B_HEMPTY + kSlots, B_DPFULL = B_SFULL + 2, B_PFULL = B_DPFULL + 2,
              B_DSFULL = B_PFULL + 2, B_PFREE = B_DSFULL + 2, B_DSFREE = B_PFREE + 2,
              B_FINAL = B_DSFREE + 2, B_DKVFREE = B_FINAL + 2, B_DRAIN = B_DKVFREE + 2,
              B_IFULL = B_DRAIN + 2, B_IFREE = B_IFULL + kRing, kNumBars = B_IFREE + kRing;
constexpr int kIFreeCount = 10;  // the two MMA threads and the 8 elementwise warps
constexpr int kOffMisc = kOffBar + kNumBars * 8;  // tmem base, abort flag, last-arriver flag
constexpr int kOffQL = kOffMisc + 16;  // the producer's copy of an item's query blocks
constexpr int kMaxItemQ = kBwdChunk * 4;      // query blocks per item at m = 16
constexpr int kOffN = kOffQL + kMaxItemQ * 4;  // iteration counts of recent items [4]
constexpr int kOffRing = (kOffN + 16 + 15) / 16 * 16;  // item descriptors [kRing][8 ints]
constexpr int kThreads = 352;  // 8 elementwise warps, producer, S/dP MMA, dV/dK MMA
// TMEM: S of iteration buffer b at 128b, dP at 64 + 128b; dV^T and dK^T of
// accumulator buffer c at 256 + 128c and 320 + 128c.
__device__ __forceinline__ uint32_t col_s(int b) { return 128u * (uint32_t)b; }
__device__ __forceinline__ uint32_t col_dp(int b) { return 64u + 128u * (uint32_t)b; }
__device__ __forceinline__ uint32_t col_dv(int c) { return 256u + 128u * (uint32_t)c; }
__device__ __forceinline__ uint32_t col_dk(int c) { return 320u + 128u * (uint32_t)c; }
constexpr size_t kSmem = 1024 + (size_t)kOffRing + kRing * 32;
static_assert(kSmem <= kMaxDynSmem, "dK/dV shared memory");
}  // namespace kv

// Rows of the transposed selection are KV spans t of 64 keys (kSub = 64/m
// blocks of m keys; the span is the block at m = 64); an item iterates over
// kSub selecting query blocks (of m tokens) at a time: 2 heads x kSub x m =
// 128 query rows, gathered by TMA. At m < 64, masks holds per (span, query
// block) which of the span's blocks the query block selected (kSub bits).
struct KvArgs {
    const float* lse;
    const float* delta;
    const BwdTInfo* tinfo;
    const int32_t* qlist;
    const uint8_t* masks;  // m < 64: per span row, a byte per query block
    const int2* queue;    // [kQueueClasses][qcap] {bg * nrows + t, chunk}
    const int* qcount;    // items per class
    int* ticket;          // next queue position to take
    float* partial;
    int* arrive;  // per (b, g, t): chunks of t finished so far
    __nv_bfloat16* dK;
    __nv_bfloat16* dV;
    int* status;
    long long qcap;
    long long nnzq;  // query-list entries per (b, g)
    int Hq, Hkv, L, nrows, topk, slot_max, mrow, chunkq;
    float scale_log2, sm_scale;
};

// One work item as the ring carries it (8 ints); n_it < 0 ends the stream.
struct KvItem {
    int bg, t, chunk, n_it;
    BwdTInfo info;
};

// Query blocks of an item (chunk c of span t's list): its iterations take kSub at a time.
__device__ __forceinline__ int item_nq(const KvArgs& a, const KvItem& it) {
    const int q_begin = it.chunk * a.chunkq;
    return max(0, min(it.info.n, q_begin + a.chunkq) - q_begin);
}

// Queue position j -> its entry {bg * nrows + t, chunk}; valid = false past the end.
__device__ __forceinline__ int2 queue_entry(const KvArgs& a, const int* qn, int j, bool& valid) {
    int c = 0;
#pragma unroll
    for (int k = 0; k < kQueueClasses; ++k)
        if (c == k && j >= qn[k]) {
            j -= qn[k];
            ++c;
        }
    valid = c < kQueueClasses;
    return valid ? a.queue[(size_t)c * a.qcap + j] : make_int2(0, 0);
}

template <int kSub>
__device__ __forceinline__ KvItem item_of(const KvArgs& a, int2 e, const BwdTInfo& info) {
    KvItem it;
    it.bg = e.x / a.nrows;
    it.t = e.x - it.bg * a.nrows;
    it.chunk = e.y;
    it.info = info;
    it.n_it = (item_nq(a, it) + kSub - 1) / kSub;
    return it;
}

__device__ __forceinline__ const int32_t* item_qlist(const KvArgs& a, const KvItem& it) {
    return a.qlist + (size_t)it.bg * a.nnzq + it.info.off + it.chunk * a.chunkq;
}

// The kSub-bit mask of the blocks of span t that query block qb selected.
template <int kSub>
__device__ __forceinline__ uint32_t span_mask(const KvArgs& a, int bg, int t, int qb) {
    if constexpr (kSub == 1) {
        return 1u;
    } else {
        return __ldg(a.masks + ((size_t)bg * a.nrows + t) * a.mrow + qb);
    }
}

__device__ __forceinline__ void ring_put(int* e, const KvItem& it) {
    *reinterpret_cast<int4*>(e) = make_int4(it.bg, it.t, it.chunk, it.n_it);
    *reinterpret_cast<int4*>(e + 4) = make_int4(it.info.off, it.info.n, it.info.nch, it.info.slot);
}

__device__ __forceinline__ KvItem ring_get(const int* e) {
    const int4 x = *reinterpret_cast<const int4*>(e);
    const int4 y = *reinterpret_cast<const int4*>(e + 4);
    KvItem it;
    it.bg = x.x;
    it.t = x.y;
    it.chunk = x.z;
    it.n_it = x.w;
    it.info.off = y.x;
    it.info.n = y.y;
    it.info.nch = y.z;
    it.info.slot = y.w;
    return it;
}

template <int kSub>
__global__ void __launch_bounds__(kv::kThreads, 1)
dkdv_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
               const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmdO,
               const KvArgs a) {
    using namespace kv;
    constexpr int kMq = 64 / kSub;  // tokens of a query block (and keys of a KV block)
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~uintptr_t(1023));
    const uint32_t sb = smem_u32(smem);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    auto bar = [&](int i) { return sb + kOffBar + 8u * (uint32_t)i; };
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + kOffMisc + 4);

    if (threadIdx.x == 0) {
        mbar_init(bar(B_KV), 1);
        mbar_init(bar(B_KVFREE), 1);
        for (int h = 0; h < kSlots; ++h) {
            mbar_init(bar(B_HFULL + h), 1);
            mbar_init(bar(B_HEMPTY + h), 1);
        }
        for (int s = 0; s < 2; ++s) {
            mbar_init(bar(B_SFULL + s), 1);
            mbar_init(bar(B_DPFULL + s), 1);
            mbar_init(bar(B_PFULL + s), 256);
            mbar_init(bar(B_DSFULL + s), 256);
            mbar_init(bar(B_PFREE + s), 1);
            mbar_init(bar(B_DSFREE + s), 1);
            mbar_init(bar(B_FINAL + s), 1);
            mbar_init(bar(B_DKVFREE + s), 256);
            mbar_init(bar(B_DRAIN + s), 1);
        }
        for (int r = 0; r < kRing; ++r) {
            mbar_init(bar(B_IFULL + r), 1);
            mbar_init(bar(B_IFREE + r), kIFreeCount);
        }
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
            prefetch_tmap(&tmQ);
            prefetch_tmap(&tmdO);
            prefetch_tmap(&tmK);
            prefetch_tmap(&tmV);
            int* qls = reinterpret_cast<int*>(smem + kOffQL);
            int* ring = reinterpret_cast<int*>(smem + kOffRing);
            int qn[kQueueClasses];
#pragma unroll
            for (int c = 0; c < kQueueClasses; ++c)
                qn[c] = (int)min((long long)max(a.qcount[c], 0), a.qcap);
            int gl = 0, kvc = 0, r = 0;  // Q/dO half-slot loads issued; items with K/V loaded; ring items
            bool ok = true;
            // hands item x to the other roles once its ring slot's last reader is done
            auto publish = [&](const KvItem& x) {
                const int slot = r % kRing;
                if (r >= kRing &&
                    !mbar_wait(bar(B_IFREE + slot), ((r / kRing) - 1) & 1, abort_flag, a.status))
                    return false;
                ring_put(ring + slot * 8, x);
                mbar_arrive(bar(B_IFULL + slot));
                ++r;
                return true;
            };
            auto entry_of = [&](int j, bool& valid) { return queue_entry(a, qn, j, valid); };
            bool valid;
            int2 e = entry_of(atomicAdd(a.ticket, 1), valid);
            KvItem it;
            it.n_it = -1;
            if (valid) it = item_of<kSub>(a, e, a.tinfo[e.x]);
            ok = publish(it);
            while (ok && it.n_it >= 0) {
                // the next item's ticket now, its queue entry after this item's
                // K/V loads and its block info after the Q/dO loads, so no load
                // latency lies on the producer's path
                const int j_nx = atomicAdd(a.ticket, 1);
                bool nx_valid = false;
                if (it.n_it > 0) {
                    const int32_t* ql = item_qlist(a, it);
                    const int nq = item_nq(a, it);
                    // this item's query blocks, batches of independent loads
                    for (int j0 = 0; j0 < kSub * kBwdChunk; j0 += kBwdChunk) {
                        int v[kBwdChunk];
#pragma unroll
                        for (int j = 0; j < kBwdChunk; ++j) v[j] = j0 + j < nq ? __ldg(ql + j0 + j) : 0;
#pragma unroll
                        for (int j = 0; j < kBwdChunk; ++j) qls[j0 + j] = v[j];
                    }
                    // K_t and V_t, once the previous item's S/dP MMAs have read theirs
                    if (kvc > 0 && !mbar_wait(bar(B_KVFREE), (kvc - 1) & 1, abort_flag, a.status)) {
                        ok = false;
                        break;
                    }
                    mbar_expect_tx(bar(B_KV), 2 * kTile64);
                    for (int dh = 0; dh < 2; ++dh) {
                        tma_load_3d(sb + kOffK + dh * kHalf64, &tmK, bar(B_KV), dh * 64, it.t * 64, it.bg);
                        tma_load_3d(sb + kOffV + dh * kHalf64, &tmV, bar(B_KV), dh * 64, it.t * 64, it.bg);
                    }
                    ++kvc;
                    e = entry_of(j_nx, nx_valid);
                    const int hq0 = (it.bg / a.Hkv) * a.Hq + (it.bg % a.Hkv) * 2;
                    for (int i = 0; ok && i < it.n_it; ++i) {
                        // Q_i then dO_i, each into the next half-slot of the ring
                        for (int h = 0; h < 2; ++h, ++gl) {
                            const int slot = gl % kSlots;
                            if (gl >= kSlots && !mbar_wait(bar(B_HEMPTY + slot), ((gl / kSlots) - 1) & 1,
                                                           abort_flag, a.status)) {
                                ok = false;
                                break;
                            }
                            const uint32_t st = sb + kOffSlot + slot * kTile128;
                            const CUtensorMap* tm = h == 0 ? &tmQ : &tmdO;
                            mbar_expect_tx(bar(B_HFULL + slot), kTile128);
                            // kSub query blocks of kMq tokens, both heads (a short last
                            // iteration repeats its last block; the rows are masked)
#pragma unroll
                            for (int j = 0; j < kSub; ++j) {
                                const int e = i * kSub + j;
                                const int qb = qls[e < nq ? e : nq - 1];
                                const uint32_t r0 = (uint32_t)(j * kMq * 128);
                                for (int hl = 0; hl < 2; ++hl)
                                    for (int dh = 0; dh < 2; ++dh)
                                        tma_load_3d(st + dh * kHalf128 + hl * kHalf64 + r0, tm,
                                                    bar(B_HFULL + slot), dh * 64, qb * kMq, hq0 + hl);
                            }
                        }
                    }
                    if (!ok) break;
                } else {
                    e = entry_of(j_nx, nx_valid);
                }
                it.n_it = -1;
                if (nx_valid) it = item_of<kSub>(a, e, a.tinfo[e.x]);
                ok = publish(it);
            }
            if (kvc > 0) mbar_wait_drain(bar(B_KV), (kvc - 1) & 1);
            for (int l = gl - kSlots; l < gl; ++l)
                if (l >= 0) mbar_wait_drain(bar(B_HFULL + l % kSlots), (l / kSlots) & 1);
        }
    } else if (warp == 9) {
        // ------------------------------------------------ S / dP MMA issuer
        // S = Q K_t^T and dP = dO V_t^T (M128 N64 K128) of every iteration, each
        // into its TMEM buffer as soon as the elementwise warps have read that
        // buffer two iterations back; separate commits, so P can be formed while
        // dP is still being computed.
        if (lane == 0) {
            constexpr uint32_t id_s = idesc_bf16(128, 64, false);
            const uint64_t dSl0 = sdesc_sw128(sb + kOffSlot, 16, 1024);  // Q/dO K-major
            const uint64_t dK0 = sdesc_sw128(sb + kOffK, 16, 1024);
            const uint64_t dV0 = sdesc_sw128(sb + kOffV, 16, 1024);
            const int* ring = reinterpret_cast<const int*>(smem + kOffRing);
            int ns = 0, kvi = 0;  // global iteration; items with iterations
            bool ok = true;
            for (int r = 0; ok; ++r) {
                if (!mbar_wait(bar(B_IFULL + r % kRing), (r / kRing) & 1, abort_flag, a.status)) break;
                const int n = ring_get(ring + (r % kRing) * 8).n_it;
                mbar_arrive(bar(B_IFREE + r % kRing));
                if (n < 0) break;
                if (n == 0) continue;
                if (!mbar_wait(bar(B_KV), kvi & 1, abort_flag, a.status)) break;
                for (int pos = 0; pos < n; ++pos, ++ns) {
                    const int b = ns & 1;
                    const uint32_t ph = (uint32_t)((ns >> 1) & 1), pp = ph ^ 1u;
                    const int lq = 2 * ns, ld = lq + 1;  // the iteration's Q and dO loads
                    // S: Q_i landed, and the elementwise warps have read S two iterations back
                    ok = mbar_wait(bar(B_HFULL + lq % kSlots), (lq / kSlots) & 1, abort_flag, a.status) &&
                         (ns < 2 || mbar_wait(bar(B_PFULL + b), pp, abort_flag, a.status));
                    if (!ok) break;
                    tc_fence_after();
                    const uint64_t qd = sdesc_at(dSl0, (lq % kSlots) * kTile128);
#pragma unroll
                    for (int ks = 0; ks < 8; ++ks)
                        mma_ss(tmem + col_s(b), sdesc_at(qd, (ks >> 2) * kHalf128 + (ks & 3) * 32),
                               sdesc_at(dK0, (ks >> 2) * kHalf64 + (ks & 3) * 32), id_s, ks > 0 ? 1u : 0u);
                    mma_commit(bar(B_SFULL + b));
                    // dP: dO_i landed, and dP two iterations back has been read
                    ok = mbar_wait(bar(B_HFULL + ld % kSlots), (ld / kSlots) & 1, abort_flag, a.status) &&
                         (ns < 2 || mbar_wait(bar(B_DSFULL + b), pp, abort_flag, a.status));
                    if (!ok) break;
                    tc_fence_after();
                    const uint64_t dd = sdesc_at(dSl0, (ld % kSlots) * kTile128);
#pragma unroll
                    for (int ks = 0; ks < 8; ++ks)
                        mma_ss(tmem + col_dp(b), sdesc_at(dd, (ks >> 2) * kHalf128 + (ks & 3) * 32),
                               sdesc_at(dV0, (ks >> 2) * kHalf64 + (ks & 3) * 32), id_s, ks > 0 ? 1u : 0u);
                    mma_commit(bar(B_DPFULL + b));
                }
                mma_commit(bar(B_KVFREE));  // the item's last S/dP: K_t/V_t may be replaced
                ++kvi;
            }
            mma_commit(bar(B_DRAIN));
            mbar_wait_drain(bar(B_DRAIN), 0);
        }
    } else if (warp == 10) {
        // ------------------------------------------------ dV^T / dK^T MMA issuer
        // dV^T += dO^T P as soon as P is stored, dK^T += Q^T dS as soon as dS is
        // (M128 N64 K128, both operands MN-major), into the item's accumulator pair.
        if (lane == 0) {
            constexpr uint32_t id_t = idesc_bf16(128, 64, true, true);  // A and B MN-major
            const uint64_t dSlT0 = sdesc_sw128(sb + kOffSlot, kHalf128, 1024);  // Q/dO MN-major
            const uint64_t dP0 = sdesc_sw128(sb + kOffP, kHalf128, 1024);
            const uint64_t dS0 = sdesc_sw128(sb + kOffDS, kHalf128, 1024);
            const int* ring = reinterpret_cast<const int*>(smem + kOffRing);
            int nv = 0, vi = 0;  // global iteration; items with iterations
            bool ok = true;
            for (int r = 0; ok; ++r) {
                if (!mbar_wait(bar(B_IFULL + r % kRing), (r / kRing) & 1, abort_flag, a.status)) break;
                const int n = ring_get(ring + (r % kRing) * 8).n_it;
                mbar_arrive(bar(B_IFREE + r % kRing));
                if (n < 0) break;
                if (n == 0) continue;
                const int c = vi & 1;  // accumulator buffer
                if (vi >= 2 && !mbar_wait(bar(B_DKVFREE + c), ((vi >> 1) - 1) & 1, abort_flag, a.status))
                    break;
                for (int pos = 0; pos < n; ++pos, ++nv) {
                    const int b = nv & 1;
                    const uint32_t ph = (uint32_t)((nv >> 1) & 1);
                    const int sq = (2 * nv) % kSlots, sd = (2 * nv + 1) % kSlots;  // Q_i, dO_i
                    // K dimension = the 128 stacked query rows, 16 per MMA. P being stored
                    // implies that S, hence Q_i, has landed (so dK^T below needs no wait
                    // of its own on Q_i), but not dO_i: its half-slot has its own
                    // barrier, which this thread waits on.
                    ok = mbar_wait(bar(B_PFULL + b), ph, abort_flag, a.status) &&
                         mbar_wait(bar(B_HFULL + sd), (uint32_t)(((2 * nv + 1) / kSlots) & 1), abort_flag,
                                   a.status);
                    if (!ok) break;
                    tc_fence_after();
                    const uint64_t dt = sdesc_at(dSlT0, sd * kTile128);
#pragma unroll
                    for (int ks = 0; ks < 8; ++ks)
                        mma_ss(tmem + col_dv(c), sdesc_at(dt, ks * 2048), sdesc_at(dP0, ks * 2048), id_t,
                               (pos > 0 || ks > 0) ? 1u : 0u);
                    mma_commit(bar(B_PFREE + b));
                    // dO_i is free once dV^T and the other thread's dP of the iteration are done
                    ok = mbar_wait(bar(B_DPFULL + b), ph, abort_flag, a.status);
                    if (!ok) break;
                    mma_commit(bar(B_HEMPTY + sd));
                    ok = mbar_wait(bar(B_DSFULL + b), ph, abort_flag, a.status);
                    if (!ok) break;
                    tc_fence_after();
                    const uint64_t qt = sdesc_at(dSlT0, sq * kTile128);
#pragma unroll
                    for (int ks = 0; ks < 8; ++ks)
                        mma_ss(tmem + col_dk(c), sdesc_at(qt, ks * 2048), sdesc_at(dS0, ks * 2048), id_t,
                               (pos > 0 || ks > 0) ? 1u : 0u);
                    mma_commit(bar(B_DSFREE + b));
                    mma_commit(bar(B_HEMPTY + sq));
                }
                if (!ok) break;
                mma_commit(bar(B_FINAL + c));
                ++vi;
            }
            mma_commit(bar(B_DRAIN + 1));
            mbar_wait_drain(bar(B_DRAIN + 1), 0);
        }
    } else {
        // ------------------------------------------------ elementwise (8 warps)
        const int row = (warp & 3) * 32 + lane;  // TMEM lane: query row (head hl, token tok)
        const int kh = warp >> 2;                // keys [32 kh, 32 kh + 32)
        const int tok = row & 63, hl = row >> 6;
        const uint32_t lane_base = tmem + ((uint32_t)((warp & 3) * 32) << 16);
        bool ok = true;
        int gi = 0, cu = 0;  // global iteration; items with iterations (accumulator uses)
        const int* ring = reinterpret_cast<const int*>(smem + kOffRing);
        for (int r = 0;; ++r) {
            const int slot = r % kRing;
            bool got = ok && mbar_wait(bar(B_IFULL + slot), (r / kRing) & 1, abort_flag, a.status);
            got = __all_sync(0xffffffffu, got);
            // the eight warps leave at the same item (the epilogue has barriers among them)
            if (!named_barrier_and(2, 256, got)) break;
            const KvItem it = ring_get(ring + slot * 8);
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(B_IFREE + slot));
            if (it.n_it < 0) break;
            const int32_t* ql = item_qlist(a, it);
            const int n_it = it.n_it, t = it.t, bg = it.bg, nq = item_nq(a, it);
            const size_t hoff = (size_t)((bg / a.Hkv) * a.Hq + (bg % a.Hkv) * 2 + hl) * a.L;
            const int jr = tok / kMq, tt = tok % kMq;  // the row's query block in the iteration, token in it
            // Row data (query block, its mask over the span's blocks, lse, Delta)
            // is fetched one iteration ahead so its latency overlaps the previous one.
            auto fetch = [&](int it2, int& qb2, uint32_t& mb2, float& nl2, float& dl2) {
                const int e = it2 * kSub + jr;
                const bool live = e < nq;
                qb2 = live ? __ldg(ql + e) : -1;
                mb2 = live ? span_mask<kSub>(a, bg, t, qb2) : 0u;
                const int i2 = qb2 * kMq + tt;
                const bool v2 = live && i2 < a.L;
                nl2 = v2 ? -__ldg(a.lse + hoff + i2) * kLog2e : -INFINITY;
                dl2 = v2 ? __ldg(a.delta + hoff + i2) : 0.f;
            };
            int qb_n = 0;
            uint32_t mb_n = 0u;
            float nl_n = 0.f, dl_n = 0.f;
            if (n_it > 0) fetch(0, qb_n, mb_n, nl_n, dl_n);
            for (int i = 0; ok && i < n_it; ++i, ++gi) {
                const int qb = qb_n;
                const uint32_t mbits = mb_n;
                const float neg_lse2 = nl_n;
                const float dlt = dl_n;
                if (i + 1 < n_it) fetch(i + 1, qb_n, mb_n, nl_n, dl_n);
                const int buf = gi & 1;
                const uint32_t ph = (uint32_t)((gi >> 1) & 1);
                // the single P and dS buffers were last read by iteration gi - 1
                const int bq = (gi - 1) & 1;
                const uint32_t pq = (uint32_t)(((gi - 1) >> 1) & 1);
                // ---- P = 2^(S scale_log2 - lse log2 e), published as soon as S is in
                ok = mbar_wait(bar(B_SFULL + buf), ph, abort_flag, a.status);
                ok = __all_sync(0xffffffffu, ok);
                if (!ok) break;
                tc_fence_after();
                uint32_t sv[32];
                tmem_ld32(lane_base + col_s(buf) + 32 * kh, sv);
                // the row's query block lies in this span: causal mask in its own block
                const bool diag = qb >= 0 && qb / kSub == t;
                const bool all = mbits == (1u << kSub) - 1u && !diag;  // every key of the tile
                // two keys at a time (packed f32x2); masks (blocks the row's query
                // block did not select, its own block's later keys, padding rows)
                // off the main path
                float pf[32];
                {
                    const float2 sc2 = make_float2(a.scale_log2, a.scale_log2);
                    const float2 nl2v = make_float2(neg_lse2, neg_lse2);
                    if (all) {  // warp-uniform: one loop per case, no per-key branch
#pragma unroll
                        for (int c = 0; c < 16; ++c) {
                            const float2 pv = __ffma2_rn(
                                make_float2(__uint_as_float(sv[2 * c]), __uint_as_float(sv[2 * c + 1])), sc2, nl2v);
                            pf[2 * c] = ex2_approx(pv.x);
                            pf[2 * c + 1] = ex2_approx(pv.y);
                        }
                    } else {
#pragma unroll
                        for (int c = 0; c < 16; ++c) {
                            const float2 pv = __ffma2_rn(
                                make_float2(__uint_as_float(sv[2 * c]), __uint_as_float(sv[2 * c + 1])), sc2, nl2v);
                            const int key = 32 * kh + 2 * c;
                            const int q0 = key / kMq, q1 = (key + 1) / kMq;
                            const bool k0 = ((mbits >> q0) & 1u) && !(diag && t * kSub + q0 == qb && key % kMq > tt);
                            const bool k1 = ((mbits >> q1) & 1u) &&
                                            !(diag && t * kSub + q1 == qb && (key + 1) % kMq > tt);
                            pf[2 * c] = k0 ? ex2_approx(pv.x) : 0.f;
                            pf[2 * c + 1] = k1 ? ex2_approx(pv.y) : 0.f;
                        }
                    }
#pragma unroll
                    for (int c = 0; c < 16; ++c) sv[c] = pack2_bf16(pf[2 * c], pf[2 * c + 1]);
                }
                tc_fence_before();
                if (gi >= 1) {  // the previous iteration's dV^T MMAs must have read P
                    ok = mbar_wait(bar(B_PFREE + bq), pq, abort_flag, a.status);
                    ok = __all_sync(0xffffffffu, ok);
                    if (!ok) break;
                }
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    *reinterpret_cast<uint4*>(smem + kOffP + sw_off(row, 4 * kh + q)) =
                        make_uint4(sv[4 * q], sv[4 * q + 1], sv[4 * q + 2], sv[4 * q + 3]);
                fence_proxy_async_smem();
                mbar_arrive(bar(B_PFULL + buf));
                // ---- dS = P (dP - Delta)
                ok = mbar_wait(bar(B_DPFULL + buf), ph, abort_flag, a.status);
                ok = __all_sync(0xffffffffu, ok);
                if (!ok) break;
                tc_fence_after();
                uint32_t dp[32];
                tmem_ld32(lane_base + col_dp(buf) + 32 * kh, dp);
                {
                    const float2 ndl = make_float2(-dlt, -dlt);
#pragma unroll
                    for (int c = 0; c < 16; ++c) {
                        const float2 d = __fadd2_rn(make_float2(__uint_as_float(dp[2 * c]), __uint_as_float(dp[2 * c + 1])), ndl);
                        const float2 ds = __fmul2_rn(make_float2(pf[2 * c], pf[2 * c + 1]), d);
                        dp[c] = pack2_bf16(ds.x, ds.y);
                    }
                }
                tc_fence_before();
                if (gi >= 1) {  // the previous iteration's dK^T MMAs must have read dS
                    ok = mbar_wait(bar(B_DSFREE + bq), pq, abort_flag, a.status);
                    ok = __all_sync(0xffffffffu, ok);
                    if (!ok) break;
                }
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    *reinterpret_cast<uint4*>(smem + kOffDS + sw_off(row, 4 * kh + q)) =
                        make_uint4(dp[4 * q], dp[4 * q + 1], dp[4 * q + 2], dp[4 * q + 3]);
                fence_proxy_async_smem();
                mbar_arrive(bar(B_DSFULL + buf));
            }
            // ---- epilogue: dV^T / dK^T, lane = head-dimension index d, keys [32 kh, +32)
            const int d = row;
            uint32_t v[32], k[32];
            if (ok && n_it > 0) {
                const int c = cu & 1;
                ok = mbar_wait(bar(B_FINAL + c), (cu >> 1) & 1, abort_flag, a.status);
                ok = __all_sync(0xffffffffu, ok);
                if (ok) {
                    tc_fence_after();
                    tmem_ld32(lane_base + col_dv(c) + 32 * kh, v);
                    tmem_ld32(lane_base + col_dk(c) + 32 * kh, k);
                    tc_fence_before();
                    mbar_arrive(bar(B_DKVFREE + c));  // the accumulators may be reused
                }
            }
            if (!(ok && n_it > 0)) {
#pragma unroll
                for (int c = 0; c < 32; ++c) { v[c] = 0u; k[c] = 0u; }
            }
            if (n_it > 0) ++cu;
            const BwdTInfo info = it.info;
            bool store = ok;
            float kscale = a.sm_scale;
            if (info.nch > 1) {
                // Multi-chunk list: write this chunk's fp32 partial; the chunk that
                // arrives last adds all partials in chunk order and stores the tile.
                float* base = a.partial + ((size_t)bg * a.slot_max + (info.slot < 0 ? 0 : info.slot)) *
                                              2 * 64 * 128;
                if (ok && info.slot >= 0) {
                    float* pk = base + (size_t)it.chunk * 2 * 64 * 128;
                    float* pv = pk + 64 * 128;
#pragma unroll
                    for (int c = 0; c < 32; ++c) {
                        const int key = 32 * kh + c;
                        pk[key * 128 + d] = __uint_as_float(k[c]) * a.sm_scale;
                        pv[key * 128 + d] = __uint_as_float(v[c]);
                    }
                }
                __threadfence();
                named_barrier(1, 256);
                volatile int* last_flag = reinterpret_cast<volatile int*>(smem + kOffMisc + 8);
                if (threadIdx.x == 0)
                    *last_flag = (ok && info.slot >= 0 &&
                                  atomicAdd(a.arrive + (size_t)bg * a.nrows + t, 1) == info.nch - 1);
                named_barrier(1, 256);
                store = ok && *last_flag;
                named_barrier(1, 256);  // every thread has read the flag before it is reused
                kscale = 1.f;  // partial sums already carry the softmax scale
                if (store) {
                    __threadfence();
                    float sk[32], sv2[32];
#pragma unroll
                    for (int c = 0; c < 32; ++c) { sk[c] = 0.f; sv2[c] = 0.f; }
                    for (int ch = 0; ch < info.nch; ++ch) {
                        const float* pk = base + (size_t)ch * 2 * 64 * 128;
#pragma unroll
                        for (int c = 0; c < 32; ++c) {
                            const int key = 32 * kh + c;
                            sk[c] += __ldcg(pk + key * 128 + d);
                            sv2[c] += __ldcg(pk + 64 * 128 + key * 128 + d);
                        }
                    }
#pragma unroll
                    for (int c = 0; c < 32; ++c) {
                        k[c] = __float_as_uint(sk[c]);
                        v[c] = __float_as_uint(sv2[c]);
                    }
                }
            }
            if (store) {
                // bf16 rows of dK and dV: for each key the 128 lanes of a warp group
                // write one contiguous 256-byte row
                __nv_bfloat16* dKr = a.dK + ((size_t)bg * a.L + (size_t)t * 64) * 128 + d;
                __nv_bfloat16* dVr = a.dV + ((size_t)bg * a.L + (size_t)t * 64) * 128 + d;
#pragma unroll
                for (int c = 0; c < 32; ++c) {
                    const int key = 32 * kh + c;
                    if (t * 64 + key < a.L) {
                        dVr[(size_t)key * 128] = __float2bfloat16_rn(__uint_as_float(v[c]));
                        dKr[(size_t)key * 128] = __float2bfloat16_rn(__uint_as_float(k[c]) * kscale);
                    }
                }
            }
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

bool dq_tc_fits(int topk, int block_size) {
    const size_t b = block_size == 16   ? dq::smem_bytes<4>(topk)
                     : block_size == 32 ? dq::smem_bytes<2>(topk)
                                        : dq::smem_bytes<1>(topk);
    return b <= kMaxDynSmem;
}

cudaError_t launch_dq_tc(const void* Q, const void* K, const void* V, const void* O,
                         const void* dO, const float* lse, float* delta, const int32_t* idx,
                         const int32_t* cnt, const int32_t* ulist, const int32_t* ucnt,
                         const uint8_t* umask, const phsa_shape& s, int topk, float sm_scale,
                         void* dQ, int* status, cudaStream_t st) {
    const int bm = s.block_size, kSub = 64 / bm;
    const int NQB = (s.L + bm - 1) / bm, nsb = (s.L + 63) / 64;
    CUtensorMap tq, tk, tv, tdo, to;
    const uint64_t pq = (uint64_t)s.B * s.Hq, pk = (uint64_t)s.B * s.Hkv;
    // Q, dO and O in 64-row boxes (the span's tokens); K and V gathered in boxes of one block
    if (!make_tmap_bf16_rows128(&tq, Q, s.L, pq, 64) ||
        !make_tmap_bf16_rows128(&tk, K, s.L, pk, (uint32_t)bm) ||
        !make_tmap_bf16_rows128(&tv, V, s.L, pk, (uint32_t)bm) ||
        !make_tmap_bf16_rows128(&tdo, dO, s.L, pq, 64) || !make_tmap_bf16_rows128(&to, O, s.L, pq, 64))
        return cudaErrorInvalidValue;
    const size_t smem = kSub == 1 ? dq::smem_bytes<1>(topk) : kSub == 2 ? dq::smem_bytes<2>(topk)
                                                                         : dq::smem_bytes<4>(topk);
    auto kern = kSub == 1 ? dq_tc_kernel<1> : kSub == 2 ? dq_tc_kernel<2> : dq_tc_kernel<4>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    int dev = 0, nsm = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
        return e;
    const int units = s.B * s.Hkv * nsb;
    DqArgs args{idx, cnt, ulist, ucnt, umask, lse, static_cast<const __nv_bfloat16*>(O), delta,
                static_cast<__nv_bfloat16*>(dQ), status, s.Hq, s.Hkv, s.L, NQB, topk, units, nsb,
                kSub * topk, sm_scale * kLog2e, sm_scale};
    ProfScope prof(K_BWD_DQ, st);
    kern<<<(unsigned)min(units, nsm), dq::kThreads, smem, st>>>(tq, tk, tv, tdo, to, args);
    return cudaGetLastError();
}

cudaError_t launch_dkdv_tc(const void* Q, const void* K, const void* V, const void* dO,
                           const float* lse, const float* delta, const BwdTInfo* tinfo,
                           const int32_t* qlist, const uint8_t* masks, const int2* queue,
                           int* qctl, const phsa_shape& s, int topk, const BwdLayout& l,
                           float sm_scale, void* dK, void* dV, float* partial, int* arrive,
                           int* status, cudaStream_t st) {
    const int kSub = l.kSub, bm = s.block_size;
    CUtensorMap tq, tk, tv, tdo;
    const uint64_t pq = (uint64_t)s.B * s.Hq, pk = (uint64_t)s.B * s.Hkv;
    // Q and dO in boxes of one query block (m rows); K and V in 64-key spans
    if (!make_tmap_bf16_rows128(&tq, Q, s.L, pq, (uint32_t)bm) ||
        !make_tmap_bf16_rows128(&tk, K, s.L, pk, 64) || !make_tmap_bf16_rows128(&tv, V, s.L, pk, 64) ||
        !make_tmap_bf16_rows128(&tdo, dO, s.L, pq, (uint32_t)bm))
        return cudaErrorInvalidValue;
    auto kern = kSub == 1 ? dkdv_tc_kernel<1> : kSub == 2 ? dkdv_tc_kernel<2> : dkdv_tc_kernel<4>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kv::kSmem);
    if (e != cudaSuccess) return e;
    int dev = 0, nsm = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
        return e;
    const long long qcap = (long long)s.B * s.Hkv * l.work_max;  // entries per queue class
    KvArgs args{lse, delta, tinfo, qlist, masks, queue, qctl, qctl + kQueueClasses, partial, arrive,
                static_cast<__nv_bfloat16*>(dK), static_cast<__nv_bfloat16*>(dV), status, qcap,
                (long long)l.nqb * topk, s.Hq, s.Hkv, s.L, l.nrows, topk, l.slot_max, l.mrow,
                l.chunk, sm_scale * kLog2e, sm_scale};
    ProfScope prof(K_BWD_DKDV, st);
    kern<<<(unsigned)(qcap < nsm ? qcap : nsm), kv::kThreads, kv::kSmem, st>>>(tq, tk, tv, tdo, args);
    return cudaGetLastError();
}

}  // namespace phsa
