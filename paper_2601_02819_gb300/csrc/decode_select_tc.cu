// Decode selection on the 5th-generation tensor cores: for the newest token of
// each sequence, the selection rule of Section 3.3 (Algorithm 1 step 3) over
// the blocks before its local window, for the G query heads of one KV head.
//
// The scores of a unit (sequence, KV head) are a dense contraction:
// S^T [candidates x G] = Krepr [candidates x D] . q^T [D x G]. The candidates
// are the M dimension (128 per tile, the representative keys loaded by TMA in
// the 128-byte swizzled layout) and the G query rows, padded with zero rows to
// N = 16, are the B operand, so each representative key is read once from
// shared memory by the tensor core and each candidate's scores land on one
// TMEM lane: thread = candidate when they are read back.
//
// One persistent CTA per SM walks the units u = blockIdx.x, + gridDim.x, ...
// (256 threads):
//   warp 4  producer: stages each unit (its length and the q^T tile) into one
//           of three unit slots, up to two units ahead, and streams the
//           candidate tiles through the ring with TMA;
//   warp 5  MMA issuer (one thread) and TMEM owner: S^T of a tile into one of
//           two TMEM buffers;
//   warps 0-3  read a tile's scores (lane = candidate), keep each head's
//           softmax statistics online (running max and sum), and write the
//           scores to one of two score buffers;
//   warps 6, 7  top-k of a unit from its score buffer while warps 0-3 score
//           the next units (warp 6 takes the units of buffer 0, warp 7 those of
//           buffer 1): A_t = sum over heads of the head's softmax probability,
//           the k largest by (A desc, t asc), then the forced blocks merged.
// Under the max-logit rule (PHSA_AGG_MAX_LOGIT) the scoring warps keep no
// statistics and A_t is the largest of the G heads' scores.
// Every wait is bounded in time; on expiry the kernel records PHSA_ERR_TIMEOUT,
// lets its own copies and MMAs finish, frees TMEM and returns.
#include "phsa_common.cuh"
#include "phsa_internal.h"
#include "tc_common.cuh"
#include "topk.cuh"

namespace phsa {

namespace {

using namespace tc;

constexpr int kCand = 128;                   // candidates per tile (MMA M)
constexpr int kN = 16;                       // MMA N: the G query rows, zero-padded
constexpr int kHalf = kCand * 64 * 2;        // one 64-column half of a tile (16 KB)
constexpr int kTile = 2 * kHalf;             // 32 KB
constexpr int kQHalf = kN * 64 * 2;          // one half of the q^T tile (2 KB)
constexpr int kQTile = 2 * kQHalf;           // 4 KB
constexpr int kSlotsMax = 6;                 // ring: up to 192 KB
constexpr int kUnitSlots = 3;
constexpr int kComputeThreads = 128;         // warps 0-3
constexpr int kThreads = 256;
constexpr int kRegKeys = 16;                 // candidate keys per lane in the top-k warp
constexpr uint32_t kTmemCols = 32;           // two 16-column score buffers

// barriers
constexpr int B_FULL = 0, B_EMPTY = kSlotsMax, B_UFULL = 2 * kSlotsMax,
              B_UFREE = B_UFULL + kUnitSlots, B_TFULL = B_UFREE + kUnitSlots, B_TFREE = B_TFULL + 2,
              B_AFULL = B_TFREE + 2, B_AFREE = B_AFULL + 2, B_DRAIN = B_AFREE + 2,
              kNumBars = B_DRAIN + 1;
// unit slots hold the length (header) and the q^T tile
constexpr int kUFreeCount = 1 + 4;  // the MMA thread (commit) and the four scoring warps

struct Args {
    const __nv_bfloat16* q;
    const int32_t* lens;
    int32_t* idx;
    int32_t* cnt;
    int* status;
    int Hq, Hkv, L, Tc, topk, n_init, n_local, units, slots, agg, bm;
    float scale_log2, scale;
};

// What one (sequence, KV head) unit asks of the selection. mode 0: no query
// (length 0, or a bad length); 1: the budget covers every candidate; 2: scored.
struct SelUnit {
    int qb, n_init_q, loc_lo, c_lo, nC, nF, ksel, mode;
};

__device__ __forceinline__ SelUnit sel_unit(const Args& a, int len) {
    SelUnit s{};
    if (len <= 0 || len > a.L) return s;
    s.qb = (len - 1) / a.bm;
    s.n_init_q = min(a.n_init, s.qb + 1);              // forced initial [0, n_init_q)
    s.loc_lo = max(s.n_init_q, s.qb - a.n_local + 1);  // forced local [loc_lo, qb]
    s.c_lo = a.n_init;                                 // candidates [c_lo, qb - n_local]
    s.nC = max(0, s.qb - a.n_local - s.c_lo + 1);
    s.nF = s.n_init_q + (s.qb - s.loc_lo + 1);
    s.ksel = a.topk - s.nF;
    s.mode = s.ksel >= s.nC ? 1 : 2;
    return s;
}

__device__ __forceinline__ int sel_tiles(const SelUnit& s) {
    return s.mode == 2 ? (s.nC + kCand - 1) / kCand : 0;
}

// Shared memory (from a 1024-byte aligned base):
//   ring [slots][32 KB] | q^T tiles [kUnitSlots][4 KB] | barriers, abort flag,
//   TMEM base | unit lengths [kUnitSlots] | per-warp statistics [4][G][2] |
//   score buffers [2]{header {unit, len, -, -}, max [G], 1/sum [G],
//   S [G][Tc]} | picks [2][topk]
__host__ __device__ constexpr int sbuf_floats(int G, int Tc) { return 4 + 2 * G + G * Tc; }
size_t fixed_smem(int G, int Tc, int topk) {
    return (size_t)kUnitSlots * kQTile + kNumBars * 8 + 16 + kUnitSlots * 4 + 4 * G * 2 * 4 +
           2 * (size_t)sbuf_floats(G, Tc) * 4 + 2 * (size_t)topk * 4 + 16;
}
int ring_slots(int G, int Tc, int topk) {
    const size_t fixed = fixed_smem(G, Tc, topk) + 1024, cap = kMaxDynSmem;
    size_t fit = fixed >= cap ? 0 : (cap - fixed) / kTile;
    if (fit > (size_t)kSlotsMax) fit = kSlotsMax;
    return fit >= 2 ? (int)fit : 0;
}
size_t smem_bytes(int G, int Tc, int topk, int slots) {
    return 1024 + (size_t)slots * kTile + fixed_smem(G, Tc, topk);
}

template <int G>
__global__ void __launch_bounds__(kThreads, 1)
decode_select_tc_kernel(const __grid_constant__ CUtensorMap tmKr,
                        const __grid_constant__ CUtensorMap tmq, const Args a) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~uintptr_t(1023));
    const uint32_t sb = smem_u32(smem);
    const int nslots = a.slots;
    uint8_t* qt0 = smem + (size_t)nslots * kTile;  // q^T tiles (1024-byte aligned)
    uint8_t* misc = qt0 + kUnitSlots * kQTile;
    const uint32_t sbar = smem_u32(misc);
    auto bar = [&](int i) { return sbar + 8u * (uint32_t)i; };
    volatile int* abort_flag = reinterpret_cast<volatile int*>(misc + kNumBars * 8);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(misc + kNumBars * 8 + 4);
    int* ulen = reinterpret_cast<int*>(misc + kNumBars * 8 + 16);  // [kUnitSlots]
    float* wstat = reinterpret_cast<float*>(ulen + kUnitSlots);    // [4][G][2]
    float* sbuf0 = wstat + 4 * G * 2;                              // [2][sbuf_floats]
    const int sbf = sbuf_floats(G, a.Tc);
    int* sel0 = reinterpret_cast<int*>(sbuf0 + 2 * sbf);           // [2][topk]
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    auto unit_of = [&](int k) { return (int)blockIdx.x + k * (int)gridDim.x; };

    if (tid == 0) {
        for (int i = 0; i < nslots; ++i) {
            mbar_init(bar(B_FULL + i), 1);
            mbar_init(bar(B_EMPTY + i), 1);
        }
        for (int i = 0; i < kUnitSlots; ++i) {
            mbar_init(bar(B_UFULL + i), 1);
            mbar_init(bar(B_UFREE + i), kUFreeCount);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar(B_TFULL + i), 1);
            mbar_init(bar(B_TFREE + i), 4);
            mbar_init(bar(B_AFULL + i), 1);
            mbar_init(bar(B_AFREE + i), 1);
        }
        mbar_init(bar(B_DRAIN), 1);
        fence_barrier_init();
        *abort_flag = 0;
    }
    if (warp == 5) {
        tmem_alloc(smem_u32(tmem_slot), kTmemCols);
        tmem_relinquish();
    }
    // rows G..15 of the q^T tiles stay zero; TMA fills rows 0..G-1 per unit
    for (int e = tid; e < kUnitSlots * kQTile / 16; e += kThreads)
        reinterpret_cast<uint4*>(qt0)[e] = make_uint4(0u, 0u, 0u, 0u);
    fence_proxy_async_smem();  // the tensor core reads them through the async proxy
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(tmem_slot);

    if (warp == 4) {
        // ------------------------------------------------ producer
        if (lane == 0) {
            prefetch_tmap(&tmKr);
            prefetch_tmap(&tmq);
        }
        // lengths of the CTA's units, 32 at a time in the lanes' registers
        int len_base = -32, len_reg = 0;
        auto len_of = [&](int k) {
            if (k >= len_base + 32) {
                len_base = k - (k & 31);
                const int u2 = unit_of(len_base + lane);
                len_reg = u2 < a.units ? __ldg(a.lens + u2 / a.Hkv) : 0;
            }
            return __shfl_sync(0xffffffffu, len_reg, k - len_base);
        };
        // the CTA's ks-th unit into unit slot ks % kUnitSlots: its length, and the
        // group's G query rows by TMA into rows 0..G-1 of the q^T tile (128-byte
        // swizzled, K-major: the layout the MMA reads)
        auto stage = [&](int ks) {
            const int u = unit_of(ks), b = u / a.Hkv, g = u % a.Hkv, us = ks % kUnitSlots;
            const int len = len_of(ks);
            if (lane == 0) {
                ulen[us] = len;
                mbar_expect_tx(bar(B_UFULL + us), 2 * G * 64 * 2);
                for (int hf = 0; hf < 2; ++hf)
                    tma_load_3d(smem_u32(qt0) + us * kQTile + hf * kQHalf, &tmq, bar(B_UFULL + us),
                                hf * 64, g * G, b);
            }
        };
        // Event loop: a tile copy whenever a ring slot is free and the next tile is
        // known; otherwise stage the next unit (up to two ahead of the copies).
        bool ok = true;
        int issued = 0, staged = -1, ik = 0, ic = 0;  // copies; last unit staged; cursor
        Deadline dl;
        while (ok) {
            bool progressed = false;
            const bool more = unit_of(ik) < a.units;
            if (more && ik <= staged) {
                const SelUnit su = sel_unit(a, ulen[ik % kUnitSlots]);
                if (ic >= sel_tiles(su)) {
                    ++ik;
                    ic = 0;
                    continue;
                }
                const int sl = issued % nslots;
                bool free_slot = issued < nslots;
                if (!free_slot && lane == 0)
                    free_slot = mbar_test_wait(bar(B_EMPTY + sl), ((issued / nslots) - 1) & 1);
                if (__shfl_sync(0xffffffffu, free_slot, 0)) {
                    if (lane == 0) {
                        // four 8 KB boxes (64 rows x 64 columns): TMA moves several
                        // smaller boxes faster than one large one
                        mbar_expect_tx(bar(B_FULL + sl), kTile);
                        for (int dh = 0; dh < 2; ++dh)
                            for (int rh = 0; rh < 2; ++rh)
                                tma_load_3d(sb + sl * kTile + dh * kHalf + rh * (kHalf / 2), &tmKr,
                                            bar(B_FULL + sl), dh * 64, su.c_lo + ic * kCand + rh * 64,
                                            unit_of(ik));
                    }
                    ++issued;
                    ++ic;
                    progressed = true;
                }
            }
            const int ks = staged + 1;
            if (!progressed && unit_of(ks) < a.units && ks <= ik + 2) {
                bool free_unit = ks < kUnitSlots;
                if (!free_unit && lane == 0)
                    free_unit = mbar_test_wait(bar(B_UFREE + ks % kUnitSlots), ((ks / kUnitSlots) - 1) & 1);
                if (__shfl_sync(0xffffffffu, free_unit, 0)) {
                    stage(ks);
                    __syncwarp();
                    staged = ks;
                    progressed = true;
                }
            }
            if (!more && unit_of(staged + 1) >= a.units) break;  // every copy issued
            if (progressed) {
                dl.reset();
            } else {
                if (*abort_flag) {
                    ok = false;
                } else if (dl.expired()) {
                    *abort_flag = 1;
                    if (lane == 0) atomicCAS(a.status, 0, PHSA_ERR_TIMEOUT);
                    ok = false;
                }
            }
            ok = __all_sync(0xffffffffu, ok) != 0;
        }
        if (lane == 0) {  // own copies land before the CTA may exit
            for (int j = max(0, issued - nslots); j < issued; ++j)
                mbar_wait_drain(bar(B_FULL + j % nslots), (j / nslots) & 1);
            for (int j = max(0, staged - kUnitSlots + 1); j <= staged; ++j)
                mbar_wait_drain(bar(B_UFULL + j % kUnitSlots), (j / kUnitSlots) & 1);
        }
    } else if (warp == 5) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_bf16(kCand, kN, false);
            const uint64_t dA0 = sdesc_sw128(sb, 16, 1024);
            const uint64_t dB0 = sdesc_sw128(smem_u32(qt0), 16, 1024);
            int gt = 0;
            bool ok = true;
            for (int k = 0; ok; ++k) {
                if (unit_of(k) >= a.units) break;
                const int us = k % kUnitSlots;
                ok = mbar_wait(bar(B_UFULL + us), (k / kUnitSlots) & 1, abort_flag, a.status);
                if (!ok) break;
                tc_fence_after();
                const int nt = sel_tiles(sel_unit(a, ulen[us]));
                const uint64_t dB = sdesc_at(dB0, us * kQTile);
                for (int i = 0; ok && i < nt; ++i, ++gt) {
                    const int sl = gt % nslots, tb = gt & 1;
                    ok = mbar_wait(bar(B_FULL + sl), (gt / nslots) & 1, abort_flag, a.status) &&
                         (gt < 2 || mbar_wait(bar(B_TFREE + tb), ((gt >> 1) - 1) & 1, abort_flag, a.status));
                    if (!ok) break;
                    tc_fence_after();
                    const uint64_t dA = sdesc_at(dA0, sl * kTile);
                    // S^T [candidates x 16] = Krepr tile . q^T, K = the 128 columns
#pragma unroll
                    for (int ks = 0; ks < 8; ++ks)
                        mma_ss(tmem + 16u * tb, sdesc_at(dA, (ks >> 2) * kHalf + (ks & 3) * 32),
                               sdesc_at(dB, (ks >> 2) * kQHalf + (ks & 3) * 32), idesc,
                               ks > 0 ? 1u : 0u);
                    mma_commit(bar(B_TFULL + tb));
                    mma_commit(bar(B_EMPTY + sl));
                }
                if (!ok) break;
                // the unit's q^T tile may be replaced once its MMAs are done
                if (nt > 0)
                    mma_commit(bar(B_UFREE + us));
                else
                    mbar_arrive(bar(B_UFREE + us));
            }
            mma_commit(bar(B_DRAIN));
            mbar_wait_drain(bar(B_DRAIN), 0);
        }
    } else if (warp < 4) {
        // ------------------------------------------------ scores (warps 0-3)
        const uint32_t lane_base = tmem + ((uint32_t)(warp * 32) << 16);
        const int lrow = warp * 32 + lane;  // TMEM lane: candidate of the tile
        int gt = 0, su = 0;                 // tiles consumed; units scored
        bool ok = true;
        for (int k = 0;; ++k) {
            const int u = unit_of(k);
            if (u >= a.units) break;
            const int us = k % kUnitSlots;
            ok = ok && mbar_wait(bar(B_UFULL + us), (k / kUnitSlots) & 1, abort_flag, a.status);
            ok = __all_sync(0xffffffffu, ok) != 0;
            // the four warps leave at the same unit (they meet at a barrier below)
            if (!named_barrier_and(1, kComputeThreads, ok)) break;
            const int len = ulen[us];
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(B_UFREE + us));  // the length is read
            const SelUnit sd = sel_unit(a, len);
            int32_t* out = a.idx + (size_t)u * a.topk;
            if (sd.mode != 2) {
                if (sd.mode == 0) {  // no query (or a bad length): empty selection
                    if (tid == 0 && (len < 0 || len > a.L)) set_status(a.status, PHSA_ERR_DEVICE_INDEX);
                    for (int j = tid; j < a.topk; j += kComputeThreads) out[j] = -1;
                    if (tid == 0) a.cnt[u] = 0;
                } else {  // the budget covers every candidate
                    const int n = sd.nF + sd.nC;
                    for (int j = tid; j < a.topk; j += kComputeThreads) {
                        int v = -1;
                        if (j < sd.n_init_q) v = j;
                        else if (j < sd.n_init_q + sd.nC) v = sd.c_lo + (j - sd.n_init_q);
                        else if (j < n) v = sd.loc_lo + (j - sd.n_init_q - sd.nC);
                        out[j] = v;
                    }
                    if (tid == 0) a.cnt[u] = n;
                }
                continue;
            }
            const int buf = su & 1;
            if (su >= 2)  // the top-k warp is done with this buffer's unit before last
                ok = ok && mbar_wait(bar(B_AFREE + buf), ((su >> 1) - 1) & 1, abort_flag, a.status);
            float* sbuf = sbuf0 + buf * sbf;
            float* Sb = sbuf + 4 + 2 * G;
            // each head's softmax statistics over the candidates, online
            float m_run[G], z_run[G];
#pragma unroll
            for (int h = 0; h < G; ++h) {
                m_run[h] = -INFINITY;
                z_run[h] = 0.f;
            }
            const int nt = sel_tiles(sd);
            for (int i = 0; i < nt; ++i, ++gt) {
                const int tb = gt & 1;
                ok = ok && mbar_wait(bar(B_TFULL + tb), (gt >> 1) & 1, abort_flag, a.status);
                ok = __all_sync(0xffffffffu, ok) != 0;  // the TMEM load is warp-wide
                uint32_t v[16];
                if (ok) {
                    tc_fence_after();
                    tmem_ld16(lane_base + 16u * tb, v);
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(B_TFREE + tb));  // the MMA may overwrite it
                const int cj = i * kCand + lrow;
                if (ok && cj < sd.nC && a.agg) {
#pragma unroll
                    for (int h = 0; h < G; ++h) Sb[h * a.Tc + cj] = __uint_as_float(v[h]) * a.scale;
                } else if (ok && cj < sd.nC) {
#pragma unroll
                    for (int h = 0; h < G; ++h) {
                        const float sc = __uint_as_float(v[h]) * a.scale_log2;
                        Sb[h * a.Tc + cj] = sc;
                        const float mn = fmaxf(m_run[h], sc);
                        z_run[h] = z_run[h] * ex2_approx(m_run[h] - mn) + ex2_approx(sc - mn);
                        m_run[h] = mn;
                    }
                }
            }
            // statistics of the warp's candidates, then of the four warps (thread 0)
#pragma unroll
            for (int h = 0; h < G; ++h) {
                float m = m_run[h], z = z_run[h];
#pragma unroll
                for (int off = 16; off > 0; off >>= 1) {
                    const float mo = __shfl_xor_sync(0xffffffffu, m, off);
                    const float zo = __shfl_xor_sync(0xffffffffu, z, off);
                    const float mn = fmaxf(m, mo);
                    z = mn == -INFINITY ? 0.f : z * ex2_approx(m - mn) + zo * ex2_approx(mo - mn);
                    m = mn;
                }
                if (lane == 0) {
                    wstat[(warp * G + h) * 2] = m;
                    wstat[(warp * G + h) * 2 + 1] = z;
                }
            }
            if (!named_barrier_and(1, kComputeThreads, ok)) break;  // scores and statistics complete
            if (tid == 0) {
#pragma unroll
                for (int h = 0; h < G; ++h) {
                    float m = -INFINITY, z = 0.f;
                    for (int w = 0; w < 4; ++w) {
                        const float mo = wstat[(w * G + h) * 2], zo = wstat[(w * G + h) * 2 + 1];
                        const float mn = fmaxf(m, mo);
                        z = mn == -INFINITY ? 0.f : z * ex2_approx(m - mn) + zo * ex2_approx(mo - mn);
                        m = mn;
                    }
                    sbuf[4 + h] = m;
                    sbuf[4 + G + h] = z > 0.f ? 1.0f / z : 0.f;
                }
                reinterpret_cast<int*>(sbuf)[0] = u;
                reinterpret_cast<int*>(sbuf)[1] = len;
                mbar_arrive(bar(B_AFULL + buf));  // hand the unit to the top-k warp
            }
            ++su;
        }
        if (tid == 0 && ok)  // the end of the CTA's units, for both top-k warps
            for (int e = su; e < su + 2; ++e) {
                const int buf = e & 1;
                bool free_buf = true;
                if (e >= 2)
                    free_buf = mbar_wait(bar(B_AFREE + buf), ((e >> 1) - 1) & 1, abort_flag, a.status);
                if (!free_buf) break;
                reinterpret_cast<int*>(sbuf0 + buf * sbf)[0] = -1;
                mbar_arrive(bar(B_AFULL + buf));
            }
    } else if (warp >= 6) {
        // ------------------------------------------------ top-k (warps 6, 7)
        const int buf = warp - 6;  // the units of this score buffer
        int* sel = sel0 + buf * a.topk;
        bool ok = true;
        for (int su = buf; ok; su += 2) {
            ok = mbar_wait(bar(B_AFULL + buf), (su >> 1) & 1, abort_flag, a.status);
            ok = __all_sync(0xffffffffu, ok) != 0;
            if (!ok) break;
            float* sbuf = sbuf0 + buf * sbf;
            const int u = reinterpret_cast<const int*>(sbuf)[0];
            if (u < 0) break;  // the end of the CTA's units
            const SelUnit d = sel_unit(a, reinterpret_cast<const int*>(sbuf)[1]);
            const float* mx = sbuf + 4;
            const float* iz = mx + G;
            float* Sb = sbuf + 4 + 2 * G;
            const int nC = d.nC, ksel = d.ksel, c_lo = d.c_lo;
            // A_t = sum over the heads of the head's softmax probability, head order;
            // or the largest of the heads' scores
            auto key_of = [&](int cj) {
                if (a.agg) {
                    float best = Sb[cj];
#pragma unroll
                    for (int h = 1; h < G; ++h) best = fmaxf(best, Sb[h * a.Tc + cj]);
                    return topk::make_key_signed(best, c_lo + cj);
                }
                float acc = 0.f;
#pragma unroll
                for (int h = 0; h < G; ++h) acc += ex2_approx(Sb[h * a.Tc + cj] - mx[h]) * iz[h];
                return topk::make_key(acc, c_lo + cj);
            };
            if (nC <= 32 * kRegKeys) {
                unsigned long long key[kRegKeys];
#pragma unroll
                for (int rr = 0; rr < kRegKeys; ++rr) {
                    const int cj = lane + 32 * rr;
                    key[rr] = cj < nC ? key_of(cj) : 0ull;
                }
                // each lane's best key is kept; only the lane that held a winner
                // looks at its keys again
                unsigned long long best = key[0];
#pragma unroll
                for (int rr = 1; rr < kRegKeys; ++rr) best = topk::umax64(best, key[rr]);
                for (int kk = 0; kk < ksel; ++kk) {
                    const unsigned mh = (unsigned)(best >> 32), ml = (unsigned)best;
                    const unsigned bh = __reduce_max_sync(0xffffffffu, mh);
                    const unsigned bl = __reduce_max_sync(0xffffffffu, mh == bh ? ml : 0u);
                    const unsigned long long win = ((unsigned long long)bh << 32) | bl;
                    if (lane == 0) sel[kk] = topk::key_block(win);
                    if (best == win) {  // keys are distinct: exactly one lane
#pragma unroll
                        for (int rr = 0; rr < kRegKeys; ++rr)
                            if (key[rr] == win) key[rr] = 0ull;
                        best = key[0];
#pragma unroll
                        for (int rr = 1; rr < kRegKeys; ++rr) best = topk::umax64(best, key[rr]);
                    }
                }
            } else if (ksel <= 32) {
                // long candidate lists: 512 keys at a time in registers, with the
                // best ksel so far carried in one register per lane
                const unsigned long long mine = topk::warp_topk32(nC, ksel, key_of, lane);
                if (lane < ksel) sel[lane] = topk::key_block(mine);
            } else {  // long lists, large budgets: rounds over shared memory; a pick is
                      // marked by a NaN score
                topk::rounds_one_warp(
                    nC, ksel, key_of, [&](int cj) { return Sb[cj] != Sb[cj]; },
                    [&](int t) { Sb[t - c_lo] = __int_as_float(0x7fc00000); }, sel, lane);
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(B_AFREE + buf));  // the scoring warps may refill it
            int32_t* out = a.idx + (size_t)u * a.topk;
            for (int j = lane; j < a.topk; j += 32) {
                if (j < d.n_init_q) out[j] = j;
                else if (j >= d.n_init_q + ksel && j < d.nF + ksel)
                    out[j] = d.loc_lo + (j - d.n_init_q - ksel);
                else if (j >= d.nF + ksel) out[j] = -1;
            }
            for (int j = lane; j < ksel; j += 32) {
                const int v = sel[j];
                int rank = 0;
                for (int i = 0; i < ksel; ++i) rank += sel[i] < v;
                out[d.n_init_q + rank] = v;
            }
            if (lane == 0) a.cnt[u] = d.nF + ksel;
            __syncwarp();  // sel is reused by the next unit
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

size_t decode_select_smem_bytes(const phsa_shape& s, int topk) {
    const int G = s.Hq / s.Hkv, Tc = s.L / s.block_size;
    const int n = ring_slots(G, Tc, topk);
    return n > 0 ? smem_bytes(G, Tc, topk, n) : (size_t)-1;
}

cudaError_t launch_decode_select(const void* q, const void* Krepr, const int32_t* lens,
                                 const phsa_shape& s, const phsa_select_params& p, int32_t* idx,
                                 int32_t* cnt, int* status, cudaStream_t st) {
    const int G = s.Hq / s.Hkv, Tc = s.L / s.block_size;
    const long long units = (long long)s.B * s.Hkv;
    const int slots = ring_slots(G, Tc, p.topk);
    if (slots == 0) return cudaErrorInvalidValue;
    CUtensorMap tm;
    // with fewer than two blocks no unit has a candidate and Krepr is never read:
    // the map then describes q (valid, unused)
    const bool have_kr = Krepr != nullptr && Tc > 0;
    if (!make_tmap_bf16_rows128(&tm, have_kr ? Krepr : q, have_kr ? (uint64_t)Tc : (uint64_t)s.Hq,
                                have_kr ? (uint64_t)units : (uint64_t)s.B, have_kr ? 64 : 1))
        return cudaErrorInvalidValue;
    CUtensorMap tq;  // q [B][Hq][128]: the G rows of one group per box
    if (!make_tmap_bf16_rows128(&tq, q, (uint64_t)s.Hq, (uint64_t)s.B, G))
        return cudaErrorInvalidValue;
    const size_t smem = smem_bytes(G, Tc, p.topk, slots);
    Args args{static_cast<const __nv_bfloat16*>(q), lens, idx, cnt, status, s.Hq, s.Hkv, s.L, Tc,
              p.topk, p.n_init, p.n_local, (int)units, slots, p.aggregation, s.block_size,
              p.sm_scale * kLog2e, p.sm_scale};
    auto kern = G == 2 ? decode_select_tc_kernel<2> : decode_select_tc_kernel<1>;
    cudaError_t e;
    if ((e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)) !=
        cudaSuccess)
        return e;
    int dev = 0, nsm = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
        return e;
    const unsigned grid = (unsigned)(units < nsm ? units : nsm);
    ProfScope prof(K_DEC_SELECT, st);
    kern<<<grid, kThreads, smem, st>>>(tm, tq, args);
    return cudaGetLastError();
}

}  // namespace phsa
