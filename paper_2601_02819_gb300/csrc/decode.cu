// Decode attention: one new token per sequence. The newest token of sequence b
// (position p = len_b - 1) attends, in each of the GQA group's G query heads,
// the blocks the selection chose for it (Eq. 10-11 for one row); the
// selection itself is in decode_select_tc.cu.
//
// The kernel reads little per unit (sequence, KV head) and is bound by HBM
// bandwidth, so it runs on the CUDA cores. Every selected K or V block is m
// consecutive rows (m = 16, 32 or 64), so a producer warp streams them into a
// shared-memory ring with 1-D bulk copies (cp.async.bulk, completion counted
// on an mbarrier per slot) and the compute warps work from shared memory: a
// half-warp per 256-byte key row (lane c holds columns 8c..8c+7). A ring slot
// holds 64 rows: 64 / m consecutive entries of the block list, each at row
// offset j m of the slot. The kernel is persistent:
// a CTA walks the units u = blockIdx.x, blockIdx.x + gridDim.x, ..., and its
// ring runs across unit boundaries, so the next unit's blocks are in flight
// while a unit finishes.
//
// Each half-warp runs an online softmax over 4 keys of every slot;
// the 16 partial states are merged (two per warp with shuffles, then the 8
// warps in shared memory). Keys after p (the unfilled part of the local block)
// are neither copied nor attended. Optionally the kernel also refreshes the
// representative key of the block the new token has just filled: that block
// is the query's own (local) block, which the kernel copies anyway, and it is
// never a candidate of the same step.
#include "phsa_common.cuh"
#include "phsa_internal.h"
#include "tc_common.cuh"

namespace phsa {

namespace {

using namespace tc;

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kRowBytes = kD * 2;                  // one bf16 key row
constexpr int kSlotRows = 64;                      // rows per ring slot (64 / m blocks)
constexpr int kSlotBytes = kSlotRows * kRowBytes;  // 16 KB
constexpr int kAttnSlots = 3;                      // attention ring: 3 x (K, V) = 96 KB

// Dot product of a 16-byte piece of a bf16 row with 8 fp32 values, added over
// the 16 lanes of a half-warp (a fixed xor tree: all 16 lanes get the sum).
// The shuffles name the whole warp: all 32 lanes must call it together.
__device__ __forceinline__ float dot8_half(const float* q, const uint4& k) {
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&k);
    float acc = 0.f;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const float2 f = __bfloat1622float2(h[j]);
        acc = fmaf(q[2 * j], f.x, acc);
        acc = fmaf(q[2 * j + 1], f.y, acc);
    }
#pragma unroll
    for (int off = 8; off > 0; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
    return acc;
}

// ============================================================== attention
struct DecAttnArgs {
    const __nv_bfloat16* q;
    const __nv_bfloat16* K;
    const __nv_bfloat16* V;
    const int32_t* idx;
    const int32_t* cnt;
    const int32_t* lens;
    __nv_bfloat16* O;
    float* lse;
    int* status;
    const uint8_t* mask;   // with Krepr: refresh the block the new token has just filled
    __nv_bfloat16* Krepr;  // null: no refresh
    float lambda;
    int Hq, Hkv, L, T, topk, units;
    float scale_log2;
};

// Warp-wide copy of one unit's block list to shared memory (out holds topk
// ints), with the rule of compact_block_list: -1 entries are skipped, and so
// is an entry outside [0, qb] or not above the last kept one (reported). A
// list whose first cnt entries are all valid and ascending -- every list the
// selection writes -- takes one load per lane; anything else goes through
// compact_block_list on lane 0. Returns the count on every lane.
__device__ __forceinline__ int stage_list_warp(const int32_t* row, const int32_t* cntp, int topk,
                                               int qb, int* out, int* status, int lane) {
    const int cnt = __ldg(cntp);
    bool good = cnt >= 0 && cnt <= topk;
    for (int j0 = 0; j0 < topk; j0 += 32) {
        const int j = j0 + lane;
        const int t = j < topk ? __ldg(row + j) : 0;
        int prev = __shfl_up_sync(0xffffffffu, t, 1);
        if (lane == 0) prev = j0 > 0 ? out[j0 - 1] : -1;
        good &= __all_sync(0xffffffffu, j >= cnt || (t >= 0 && t <= qb && t > prev)) != 0;
        if (j < topk) out[j] = t;
        __syncwarp();
    }
    if (good) return cnt;
    int n = 0;
    if (lane == 0) n = compact_block_list(row, cnt, topk, qb, out, status);
    return __shfl_sync(0xffffffffu, n, 0);
}

// Roles: warps 0-7 compute; warp 8 is the producer. The producer stages each
// unit (length, block list, the G query rows, the punctuation bits of a
// just-filled block) into one of kUnitSlots unit slots, up to two units ahead,
// and streams the selected K/V blocks through the ring. Barriers: full / empty per
// ring slot (empty counts the 8 compute warps), ufull / ufree per unit slot.
// The compute warps meet only once per unit (the merge).
constexpr int kAttnThreads = 288;
constexpr int kUnitSlots = 3;
constexpr int kAB_FULL = 0, kAB_EMPTY = kAttnSlots, kAB_UFULL = 2 * kAttnSlots,
              kAB_UFREE = kAB_UFULL + kUnitSlots, kAttnBars = kAB_UFREE + kUnitSlots;
constexpr int kAttnOffBar = kAttnSlots * 2 * kSlotBytes;
constexpr int kAttnOffUnit = kAttnOffBar + (8 * kAttnBars + 4 + 127) / 128 * 128;  // + abort flag
static_assert(kAttnOffUnit - kAttnOffBar >= 8 * kAttnBars + 4, "barriers and abort flag fit");
// unit slot: {len, n, plo, phi} | q bf16 [G][128] | block list [topk rounded up to 4]
__host__ __device__ constexpr int unit_slot_bytes(int G, int topk) {
    return 16 + G * kD * 2 + ((topk + 3) & ~3) * 4;
}
size_t dec_attn_smem(int G, int topk) {
    return (size_t)kAttnOffUnit + (size_t)kUnitSlots * unit_slot_bytes(G, topk) +
           (size_t)kWarps * G * 130 * 4 + 4 * 2 * kD * 4;
}

template <int G, int kBm>
__global__ void __launch_bounds__(kAttnThreads, 2)
decode_attn_kernel(const DecAttnArgs a) {
    constexpr int kSub = kSlotRows / kBm;  // blocks per ring slot
    extern __shared__ __align__(128) uint8_t smem[];
    const uint32_t sb = smem_u32(smem);
    auto bar = [&](int i) { return sb + kAttnOffBar + 8u * (uint32_t)i; };
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + kAttnOffBar + 8 * kAttnBars);
    const int ubytes = unit_slot_bytes(G, a.topk);
    uint8_t* units0 = smem + kAttnOffUnit;
    float* part = reinterpret_cast<float*>(units0 + kUnitSlots * ubytes);  // [8][G][130]
    float* rpart = part + kWarps * G * 130;                               // [4][2][128]
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    auto unit_of = [&](int k) { return (int)blockIdx.x + k * (int)gridDim.x; };
    const bool refresh = a.Krepr != nullptr;

    if (tid == 0) {
        for (int i = 0; i < kAttnSlots; ++i) {
            mbar_init(bar(kAB_FULL + i), 1);
            mbar_init(bar(kAB_EMPTY + i), kWarps);
        }
        for (int i = 0; i < kUnitSlots; ++i) {
            mbar_init(bar(kAB_UFULL + i), 1);
            mbar_init(bar(kAB_UFREE + i), kWarps);
        }
        fence_barrier_init();
        *abort_flag = 0;
    }
    __syncthreads();

    if (warp == kWarps) {
        // ------------------------------------------------ producer
        bool ok = true;
        int issued = 0;  // blocks copied
        // stage the CTA's k-th unit into unit slot k % kUnitSlots
        auto stage = [&](int k) {
            const int us = k % kUnitSlots;  // free: the loop has seen its ufree phase
            const int u = unit_of(k), b = u / a.Hkv, g = u % a.Hkv;
            uint8_t* slot = units0 + us * ubytes;
            int* hdr = reinterpret_cast<int*>(slot);
            int* list = hdr + 4 + G * kD / 2;
            const int len = __ldg(a.lens + b);
            const bool valid = len > 0 && len <= a.L;
            if (lane < G * 16)  // the group's query rows, 16 bytes per lane
                reinterpret_cast<uint4*>(slot + 16)[lane] = __ldg(
                    reinterpret_cast<const uint4*>(a.q + ((size_t)b * a.Hq + g * G) * kD) + lane);
            int n = 0;
            if (valid)
                n = stage_list_warp(a.idx + (size_t)u * a.topk, a.cnt + u, a.topk,
                                    (len - 1) / kBm, list, a.status, lane);
            unsigned plo = 0, phi = 0;
            if (refresh && valid && len % kBm == 0) {  // the m flags of the just-filled block
                const uint8_t* mb = a.mask + (size_t)b * a.L + (size_t)(len - kBm);
                plo = __ballot_sync(0xffffffffu, lane < kBm && mb[lane] != 0);
                phi = __ballot_sync(0xffffffffu, kBm > 32 && mb[kBm > 32 ? 32 + lane : 0] != 0);
            }
            if (lane == 0) {
                hdr[0] = len;
                hdr[1] = n;
                hdr[2] = (int)plo;
                hdr[3] = (int)phi;
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(kAB_UFULL + us));
        };
        // Event loop: a copy whenever a ring slot is free and the next block is
        // known; otherwise stage the next unit (up to two ahead of the copies),
        // so that the loads of staging never hold back a copy.
        int staged = -1, ik = 0, ii = 0;  // last unit staged; copy cursor (unit, ring slot)
        Deadline dl;
        while (ok) {
            bool progressed = false;
            const bool more = unit_of(ik) < a.units;
            if (more && ik <= staged) {
                const int* hdr = reinterpret_cast<const int*>(units0 + (ik % kUnitSlots) * ubytes);
                const int n = hdr[1];
                if (ii * kSub >= n) {
                    ++ik;
                    ii = 0;
                    continue;
                }
                const int sl = issued % kAttnSlots;
                bool free_slot = issued < kAttnSlots;
                if (!free_slot && lane == 0)
                    free_slot = mbar_test_wait(bar(kAB_EMPTY + sl), ((issued / kAttnSlots) - 1) & 1);
                free_slot = __shfl_sync(0xffffffffu, free_slot, 0) != 0;
                if (free_slot) {
                    if (lane == 0) {
                        // entries e0 .. e1 - 1 of the list, entry e0 + j at slot row j m
                        const int* lst = hdr + 4 + G * kD / 2;
                        const int len = hdr[0], p = len - 1, qb = p / kBm;
                        const int e0 = ii * kSub, e1 = min(n, e0 + kSub);
                        uint32_t total = 0;
                        for (int e = e0; e < e1; ++e) {
                            const int t = lst[e];
                            total += (uint32_t)(t == qb ? p - t * kBm + 1 : kBm) * kRowBytes;
                        }
                        mbar_expect_tx(bar(kAB_FULL + sl), 2 * total);
                        for (int e = e0; e < e1; ++e) {
                            const int t = lst[e];
                            const int rows = t == qb ? p - t * kBm + 1 : kBm;  // keys up to p
                            const size_t off = ((size_t)unit_of(ik) * a.L + (size_t)t * kBm) * kD;
                            const uint32_t bytes = (uint32_t)rows * kRowBytes;
                            const uint32_t dst = sb + sl * 2 * kSlotBytes +
                                                 (uint32_t)((e - e0) * kBm) * kRowBytes;
                            bulk_load(dst, a.K + off, bytes, bar(kAB_FULL + sl));
                            bulk_load(dst + kSlotBytes, a.V + off, bytes, bar(kAB_FULL + sl));
                        }
                    }
                    ++issued;
                    ++ii;
                    progressed = true;
                }
            }
            const int ks = staged + 1;
            if (!progressed && unit_of(ks) < a.units && ks <= ik + 2) {
                bool free_unit = ks < kUnitSlots;
                if (!free_unit && lane == 0)
                    free_unit = mbar_test_wait(bar(kAB_UFREE + ks % kUnitSlots),
                                               ((ks / kUnitSlots) - 1) & 1);
                if (__shfl_sync(0xffffffffu, free_unit, 0)) {
                    stage(ks);
                    staged = ks;
                    progressed = true;
                }
            }
            if (!more && unit_of(staged + 1) >= a.units) break;  // every copy issued
            if (progressed) {
                dl.reset();
            } else {
                __nanosleep(64);  // nothing to do yet: leave the issue slots to the other warps
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
        if (lane == 0)  // own copies land before the CTA may exit
            for (int j = max(0, issued - kAttnSlots); j < issued; ++j)
                mbar_wait_drain(bar(kAB_FULL + j % kAttnSlots), (j / kAttnSlots) & 1);
        return;
    }

    // ---------------------------------------------------- compute (warps 0-7)
    const int hw = tid >> 4, c16 = tid & 15;
    int gc = 0;  // blocks consumed
    bool ok = true;
    for (int k = 0;; ++k) {
        const int u = unit_of(k);
        if (u >= a.units) break;
        const int us = k % kUnitSlots;
        ok = ok && mbar_wait(bar(kAB_UFULL + us), (k / kUnitSlots) & 1, abort_flag, a.status);
        ok = __all_sync(0xffffffffu, ok) != 0;
        // the eight warps leave at the same unit (the merge has a barrier among them)
        if (!named_barrier_and(1, kThreads, ok)) break;
        const uint8_t* slot = units0 + us * ubytes;
        const int* hdr = reinterpret_cast<const int*>(slot);
        const int* list = hdr + 4 + G * kD / 2;
        const int len = hdr[0], nb = hdr[1];
        const unsigned plo = (unsigned)hdr[2], phi = (unsigned)hdr[3];
        const int b = u / a.Hkv, g = u % a.Hkv;
        const size_t orow = (size_t)b * a.Hq + g * G;  // first query head of the group
        if (len <= 0 || len > a.L) {  // no query: zero output, lse = -inf
            if (tid == 0 && (len < 0 || len > a.L)) set_status(a.status, PHSA_ERR_DEVICE_INDEX);
            for (int e = tid; e < G * kD; e += kThreads) a.O[orow * kD + e] = __float2bfloat16_rn(0.f);
            if (tid < G) a.lse[orow + tid] = -INFINITY;
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(kAB_UFREE + us));
            continue;
        }
        const int p = len - 1, qb = p / kBm;
        const bool fill = refresh && len % kBm == 0;  // refresh block qb's representative key
        float qv[G][8];
#pragma unroll
        for (int h = 0; h < G; ++h) {
            const uint4 v = *reinterpret_cast<const uint4*>(slot + 16 + h * kRowBytes + c16 * 16);
            const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const float2 f = __bfloat1622float2(h2[j]);
                qv[h][2 * j] = f.x * a.scale_log2;
                qv[h][2 * j + 1] = f.y * a.scale_log2;
            }
        }
        float m[G], l[G], o[G][8];
#pragma unroll
        for (int h = 0; h < G; ++h) {
            m[h] = -INFINITY;
            l[h] = 0.f;
#pragma unroll
            for (int e = 0; e < 8; ++e) o[h][e] = 0.f;
        }
        bool filled = false;
        // Half-warp hw takes slot rows [4 hw, 4 hw + 4): four consecutive keys of
        // one block (list entry i sub + jh), from its row rh on.
        const int jh = (4 * hw) / kBm, rh = 4 * hw - jh * kBm;
        const int ng = (nb + kSub - 1) / kSub;
        for (int i = 0; i < ng; ++i, ++gc) {
            const int sl = gc % kAttnSlots;
            ok = ok && mbar_wait(bar(kAB_FULL + sl), (gc / kAttnSlots) & 1, abort_flag, a.status);
            const int e = i * kSub + jh;
            const int t = e < nb ? list[e] : -1;
            const int rows = t < 0 ? 0 : t == qb ? p - t * kBm + 1 : kBm;
            const uint8_t* ks = smem + sl * 2 * kSlotBytes;
            const uint8_t* vs = ks + kSlotBytes;
            // scores first, then the values: K and V fragments are not live together
            bool vis[4];
            float sc4[G][4];
#pragma unroll
            for (int r = 0; r < 4; ++r) {
                const int key = 4 * hw + r;
                vis[r] = ok && rh + r < rows;
                const uint4 kr = vis[r] ? *reinterpret_cast<const uint4*>(ks + key * kRowBytes + c16 * 16)
                                        : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
                for (int h = 0; h < G; ++h) {
                    // dot8_half shuffles across the whole warp: call it on every lane
                    // (a masked key holds zeros), then mask the score
                    const float d = dot8_half(qv[h], kr);
                    sc4[h][r] = vis[r] ? d : -INFINITY;
                }
            }
            uint4 vr[4];
#pragma unroll
            for (int r = 0; r < 4; ++r)
                vr[r] = vis[r] ? *reinterpret_cast<const uint4*>(vs + (4 * hw + r) * kRowBytes + c16 * 16)
                               : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
            for (int h = 0; h < G; ++h) {
                const float* s = sc4[h];
                float mn = m[h];
#pragma unroll
                for (int r = 0; r < 4; ++r) mn = fmaxf(mn, s[r]);
                if (mn == -INFINITY) continue;  // no key of this step is visible
                const float sc = ex2_approx(m[h] - mn);
                l[h] *= sc;
#pragma unroll
                for (int e = 0; e < 8; ++e) o[h][e] *= sc;
#pragma unroll
                for (int r = 0; r < 4; ++r) {
                    const float pr = ex2_approx(s[r] - mn);
                    l[h] += pr;
                    const __nv_bfloat162* v2 = reinterpret_cast<const __nv_bfloat162*>(&vr[r]);
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        const float2 f = __bfloat1622float2(v2[j]);
                        o[h][2 * j] = fmaf(pr, f.x, o[h][2 * j]);
                        o[h][2 * j + 1] = fmaf(pr, f.y, o[h][2 * j + 1]);
                    }
                }
                m[h] = mn;
            }
            // the slot's entry for block qb (the list's last, when present)
            const int eq = min(nb, i * kSub + kSub) - 1;
            if (fill && ok && eq >= i * kSub && list[eq] == qb && warp < kBm / 16) {
                // Eq. 6-8 over the block's m rows in the slot, in the summation order
                // of decode_repr_kernel: warp w rows [16w, 16w + 16), even and odd
                // rows per lane half, halves added, then the warps in order
                const int half = lane >> 4, col = lane & 15;
                const uint8_t* kq = ks + (size_t)((eq - i * kSub) * kBm) * kRowBytes;
                float s0[8], sp[8];
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    s0[j] = 0.f;
                    sp[j] = 0.f;
                }
#pragma unroll
                for (int uu = 0; uu < 8; ++uu) {
                    const int r = 16 * warp + 2 * uu + half;
                    const uint4 kv = *reinterpret_cast<const uint4*>(kq + r * kRowBytes + col * 16);
                    const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&kv);
                    const bool pu = ((r < 32 ? plo >> r : phi >> (r - 32)) & 1u) != 0;
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        const float2 f = __bfloat1622float2(h2[j]);
                        s0[2 * j] += f.x;
                        s0[2 * j + 1] += f.y;
                        if (pu) {
                            sp[2 * j] += f.x;
                            sp[2 * j + 1] += f.y;
                        }
                    }
                }
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    s0[j] += __shfl_xor_sync(0xffffffffu, s0[j], 16);
                    sp[j] += __shfl_xor_sync(0xffffffffu, sp[j], 16);
                }
                if (half == 0) {
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        rpart[(warp * 2 + 0) * kD + col * 8 + j] = s0[j];
                        rpart[(warp * 2 + 1) * kD + col * 8 + j] = sp[j];
                    }
                }
                filled = true;
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(kAB_EMPTY + sl));  // this warp is done with the slot
        }

        // ---- merge: the two half-warps of a warp with shuffles, then the 8 warps
#pragma unroll
        for (int h = 0; h < G; ++h) {
            const float mo = __shfl_xor_sync(0xffffffffu, m[h], 16);
            const float lo2 = __shfl_xor_sync(0xffffffffu, l[h], 16);
            const float M2 = fmaxf(m[h], mo);
            const float fa = M2 == -INFINITY ? 0.f : ex2_approx(m[h] - M2);
            const float fb = M2 == -INFINITY ? 0.f : ex2_approx(mo - M2);
            l[h] = l[h] * fa + lo2 * fb;
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                const float oo = __shfl_xor_sync(0xffffffffu, o[h][e], 16);
                o[h][e] = o[h][e] * fa + oo * fb;
            }
            float* st = part + ((size_t)warp * G + h) * 130;
            if (lane == 0) {
                st[0] = M2;
                st[1] = l[h];
            }
            if (lane < 16) {
#pragma unroll
                for (int e = 0; e < 8; ++e) st[2 + c16 * 8 + e] = o[h][e];
            }
        }
        filled = named_barrier_and(1, kThreads, !filled) == false;  // part and rpart complete
        if (ok && tid < G * kD) {
            const int h = tid / kD, d = tid % kD;
            float M = -INFINITY;
            for (int w = 0; w < kWarps; ++w) M = fmaxf(M, part[((size_t)w * G + h) * 130]);
            float Ls = 0.f, acc = 0.f;
            if (M != -INFINITY) {
                for (int w = 0; w < kWarps; ++w) {
                    const float* st = part + ((size_t)w * G + h) * 130;
                    const float f = ex2_approx(st[0] - M);  // 0 for a warp that saw no key
                    Ls += st[1] * f;
                    acc += st[2 + d] * f;
                }
            }
            a.O[(orow + h) * kD + d] = __float2bfloat16_rn(Ls > 0.f ? acc / Ls : 0.f);
            if (d == 0) a.lse[orow + h] = Ls > 0.f ? (M + log2f(Ls)) * kLn2 : -INFINITY;
        }
        if (ok && filled && tid < kD) {
            float a0 = 0.f, ap = 0.f;
            for (int w = 0; w < kBm / 16; ++w) {
                a0 += rpart[(w * 2 + 0) * kD + tid];
                ap += rpart[(w * 2 + 1) * kD + tid];
            }
            const int c = __popc(plo) + __popc(phi);
            const float m0 = a0 * (1.0f / (float)kBm);  // Eq. 6
            const float ov = c > 0 ? a.lambda * m0 + (1.0f - a.lambda) * (ap * (1.0f / (float)c))
                                   : m0;  // Eq. 7-8; no punctuation: the mean
            a.Krepr[((size_t)u * a.T + qb) * kD + tid] = __float2bfloat16_rn(ov);
        }
        // the unit slot is no longer read; part and rpart are written again only
        // after the next unit's barrier
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(kAB_UFREE + us));
    }
}

// Persistent grid: one CTA per unit if they all fit at once, else as many
// CTAs as the device holds.
template <class Kern>
cudaError_t persistent_grid(Kern kern, int threads, size_t smem, long long units, unsigned& grid) {
    int dev = 0, nsm = 0, per_sm = 0;
    cudaError_t e;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
        return e;
    // as much shared memory as the SM has, so that several CTAs fit
    if ((e = cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout, 100)) !=
        cudaSuccess)
        return e;
    if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, threads, smem)) !=
        cudaSuccess)
        return e;
    const long long cap = (long long)nsm * (per_sm > 0 ? per_sm : 1);
    grid = (unsigned)(units < cap ? units : cap);
    return cudaSuccess;
}

cudaError_t launch_decode_attn_any(const void* q, const void* K, const void* V, const int32_t* idx,
                                   const int32_t* cnt, const int32_t* lens, const phsa_shape& s,
                                   int topk, float sm_scale, void* O, float* lse,
                                   const uint8_t* mask, float lambda, void* Krepr, int* status,
                                   cudaStream_t st) {
    const int G = s.Hq / s.Hkv;
    const size_t smem = dec_attn_smem(G, topk);
    const long long units = (long long)s.B * s.Hkv;
    DecAttnArgs args{static_cast<const __nv_bfloat16*>(q), static_cast<const __nv_bfloat16*>(K),
                     static_cast<const __nv_bfloat16*>(V), idx, cnt, lens,
                     static_cast<__nv_bfloat16*>(O), lse, status, mask,
                     static_cast<__nv_bfloat16*>(Krepr), lambda, s.Hq, s.Hkv, s.L,
                     s.L / s.block_size, topk, (int)units, sm_scale * kLog2e};
    const int bm = s.block_size;
    auto kern = G == 2 ? (bm == 16   ? decode_attn_kernel<2, 16>
                          : bm == 32 ? decode_attn_kernel<2, 32>
                                     : decode_attn_kernel<2, 64>)
                       : (bm == 16   ? decode_attn_kernel<1, 16>
                          : bm == 32 ? decode_attn_kernel<1, 32>
                                     : decode_attn_kernel<1, 64>);
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    unsigned grid = 0;
    if ((e = persistent_grid(kern, kAttnThreads, smem, units, grid)) != cudaSuccess) return e;
    ProfScope prof(K_DEC_ATTN, st);
    kern<<<grid, kAttnThreads, smem, st>>>(args);
    return cudaGetLastError();
}

}  // namespace

size_t decode_attn_smem_bytes(const phsa_shape& s, int topk) {
    return dec_attn_smem(s.Hq / s.Hkv, topk);
}

cudaError_t launch_decode_attn(const void* q, const void* K, const void* V, const int32_t* idx,
                               const int32_t* cnt, const int32_t* lens, const phsa_shape& s,
                               int topk, float sm_scale, void* O, float* lse, int* status,
                               cudaStream_t st) {
    return launch_decode_attn_any(q, K, V, idx, cnt, lens, s, topk, sm_scale, O, lse, nullptr, 0.f,
                                  nullptr, status, st);
}

cudaError_t launch_decode_attn_repr(const void* q, const void* K, const void* V,
                                    const int32_t* idx, const int32_t* cnt, const int32_t* lens,
                                    const phsa_shape& s, int topk, float sm_scale, void* O,
                                    float* lse, const uint8_t* mask, float lambda, void* Krepr,
                                    int* status, cudaStream_t st) {
    return launch_decode_attn_any(q, K, V, idx, cnt, lens, s, topk, sm_scale, O, lse, mask, lambda,
                                  Krepr, status, st);
}


// Appends the new token's key and value (and punctuation flag) at row
// len - 1 of each sequence: one warp per (b, g), lanes 0-15 copy the 256-byte
// key row and lanes 16-31 the value row, 16 bytes each.
constexpr int kAppendWarps = 8;

__global__ void __launch_bounds__(kAppendWarps * 32)
decode_append_kernel(const int4* __restrict__ knew, const int4* __restrict__ vnew,
                     const uint8_t* __restrict__ flag, const int32_t* __restrict__ lens, int B,
                     int Hkv, int L, int4* __restrict__ K, int4* __restrict__ V,
                     uint8_t* __restrict__ mask, int* status) {
    const int lane = threadIdx.x & 31;
    const long long u = (long long)blockIdx.x * kAppendWarps + (threadIdx.x >> 5);
    if (u >= (long long)B * Hkv) return;
    const int b = (int)(u / Hkv), g = (int)(u % Hkv);
    const int len = lens[b];
    if (len > L) {
        if (g == 0 && lane == 0) set_status(status, PHSA_ERR_DEVICE_INDEX);
        return;
    }
    if (len <= 0) return;
    constexpr int kRow = kD * 2 / 16;  // int4 per row
    const long long dst = (u * L + (len - 1)) * kRow;
    const int c = lane & 15;
    if (lane < 16) K[dst + c] = knew[u * kRow + c];
    else V[dst + c] = vnew[u * kRow + c];
    if (flag && g == 0 && lane == 0) mask[(long long)b * L + (len - 1)] = flag[b] ? 1 : 0;
}

cudaError_t launch_decode_append(const void* k_new, const void* v_new, const uint8_t* flag,
                                 const int32_t* lens, const phsa_shape& s, void* K, void* V,
                                 uint8_t* mask, int* status, cudaStream_t st) {
    const long long units = (long long)s.B * s.Hkv;
    if (units == 0) return cudaSuccess;
    const unsigned grid = (unsigned)((units + kAppendWarps - 1) / kAppendWarps);
    decode_append_kernel<<<grid, kAppendWarps * 32, 0, st>>>(
        static_cast<const int4*>(k_new), static_cast<const int4*>(v_new), flag, lens, s.B, s.Hkv,
        s.L, static_cast<int4*>(K), static_cast<int4*>(V), mask, status);
    return cudaGetLastError();
}

}  // namespace phsa
