// Stage (b) on the tensor cores for GQA pairs (G*64 = 128 query rows):
// query-to-block relevance and Top-K selection (Eq. 8; Algorithm 1 step 3).
//
// This kernel runs at block sizes 16 and 32, and at 64 beyond 1024 query
// blocks (shorter sequences take the one-unit kernel of select_tc_unit.cu).
//
// Work unit: a batch of two 64-token spans of one (batch, KV head) -- each span
// is kSub = 64/m query blocks and fills one 128-row tile (two heads x 64
// tokens). Both spans score the same candidate representative keys (a span's
// candidates are a prefix of Krepr), so one TMA load of a chunk of 128
// candidates serves both. Persistent: one CTA per SM walks the batches,
// heaviest first over all (batch, KV head) pairs.
//
// Each chunk is used twice, and the scores never leave the SM:
//   pass 1  S = Q Kr^T   (M = 128 query rows, N = 128 candidates) in TMEM;
//           the thread owning a row keeps sum 2^(S*scale - m) over the
//           candidates its query block may select, against a shift m that is
//           the row's first maximum and moves only when a later score would
//           overflow the sum; after the last chunk M_r = m + log2(sum).
//   pass 2  S^T = Kr Q^T (M = 128 candidates, N = 128 rows) in TMEM, the
//           chunks in reverse order (the last ones are still in the ring);
//           the thread owning candidate t sums p = 2^(S*scale - M_r) over the
//           rows of each query block of its span, in row order, so equal
//           candidates get bit-identical sums: A[qb][t].
//   top-k   per query block, by one warp of the span's warpgroup: larger A
//           first, lower t on exact ties; output ascending with the forced
//           initial and local blocks, -1 padded.
// The max-logit rule (PHSA_AGG_MAX_LOGIT) needs no softmax statistics: pass 2
// alone, A = max over the query block's rows (rows past L excluded) * scale.
//
// Roles: warps 0-3 own span 0 of a batch, warps 4-7 span 1 (one TMEM lane per
// thread, two 128-column TMEM buffers per span), warp 8 issues TMA (the two Q
// tiles and the chunk ring), warp 9 the MMAs. The chunk ring keeps the last
// chunks of pass 1 for pass 2 (least recently used slot refilled first). The
// ring, the TMEM buffers and every barrier run on counters that continue
// across batches. Every wait is bounded in time.
#include "phsa_common.cuh"
#include "phsa_internal.h"
#include "tc_common.cuh"
#include "topk.cuh"

namespace phsa {

namespace {

using namespace tc;

constexpr int kCand = 128;              // candidates per chunk
constexpr int kHalf = 128 * 64 * 2;     // [128 rows][64 columns] bf16 (16 KB)
constexpr int kTile = 2 * kHalf;        // 128 x 128 bf16 (32 KB)
constexpr int kBox = kHalf / 2;         // a 64-row TMA box of one column half (8 KB)
constexpr int kMaxSlots = 3;            // chunk ring slots (2 when shared memory is short)
constexpr int kThreads = 320;           // 8 elementwise warps, TMA, MMA
constexpr uint32_t kTmemCols = 512;     // 4 buffers of 128 columns: span s uses 2s, 2s + 1

// Q tile slots: span si of a batch uses slot si * nq + (its load count % nq), nq = 2
// when shared memory allows (the next batch's tiles load during this one), else 1.
constexpr int B_QFULL = 0, B_QFREE = 4, B_KFULL = 8, B_KEMPTY = B_KFULL + kMaxSlots,
              B_SFULL = B_KEMPTY + kMaxSlots, B_SFREE = B_SFULL + 4, B_DRAIN = B_SFREE + 4,
              kNumBars = B_DRAIN + 1;

// Shared-memory layout (offsets from the 1024-aligned base).
struct SelLayout {
    int nq;              // Q tile slots per span (1 or 2)
    int slots;           // chunk ring slots
    int a_stride;        // floats per query block's aggregate array (>= NQB, multiple of 4)
    size_t kr, stats, fin, A, bar, misc, total;
};

__host__ __device__ inline SelLayout sel_layout(int nqb, int kSub, int nq, int slots) {
    SelLayout L;
    L.nq = nq;
    L.slots = slots;
    L.a_stride = (nqb + 3) & ~3;
    L.kr = 2 * (size_t)nq * kTile;                  // Q tiles of the two spans first
    L.stats = L.kr + (size_t)slots * kTile;         // -M_r of the 128 rows, per span
    L.fin = L.stats + 2 * 128 * 4;                  // top-k finalists [span][4 warps][32] u64
    L.A = L.fin + 2 * 4 * 32 * 8;                   // A[span][query block of span][candidate]
    L.bar = L.A + (size_t)2 * kSub * L.a_stride * 4;
    L.misc = L.bar + kNumBars * 8;                  // tmem base, abort flag
    L.total = 1024 + L.misc + 16;
    return L;
}

// The largest layout that fits: two Q slots per span first, then ring depth.
__host__ __device__ inline SelLayout sel_layout_fit(int nqb, int kSub) {
    const int cfg[4][2] = {{2, 3}, {2, 2}, {1, 3}, {1, 2}};
    for (int i = 0; i < 3; ++i) {
        const SelLayout l = sel_layout(nqb, kSub, cfg[i][0], cfg[i][1]);
        if (l.total <= kMaxDynSmem) return l;
    }
    return sel_layout(nqb, kSub, 1, 2);
}

struct SelArgs {
    int32_t* idx_out;
    int32_t* cnt_out;
    int* status;
    int Hq, Hkv, L, T, NQB, topk, n_init, n_local, agg;
    int nsb;      // 64-token spans per (b, g)
    int nbat;     // batches per (b, g): ceil(nsb / 2)
    int BG;       // B * Hkv
    int batches;  // BG * nbat
    float scale_log2, scale;
    int nq, slots, a_stride;
    uint32_t off_kr, off_stats, off_fin, off_A, off_bar, off_misc;
};

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

// One span of a batch: its query blocks [s*kSub, s*kSub + nqb), the union of
// their candidate ranges [n_init, c_hi] and the chunks of it that are scored.
struct SpanInfo {
    int s, nqb, c_hi, nC, nch;
    bool present, scored;
};
struct BatchInfo {
    int bg, hq0, n;  // n: chunks of the batch (max over its spans)
    SpanInfo sp[2];
};

template <int kSub>
__device__ __forceinline__ BatchInfo batch_info(const SelArgs& a, int v) {
    BatchInfo B;
    const int k = v / a.BG;
    B.bg = v - k * a.BG;
    B.hq0 = (B.bg / a.Hkv) * a.Hq + (B.bg % a.Hkv) * 2;
    B.n = 0;
#pragma unroll
    for (int si = 0; si < 2; ++si) {
        SpanInfo& p = B.sp[si];
        p.s = a.nsb - 1 - 2 * k - si;  // the heavier (later) span first
        p.present = p.s >= 0;
        p.scored = false;
        p.nqb = 0;
        p.c_hi = -1;
        p.nC = 0;
        p.nch = 0;
        if (!p.present) continue;
        p.nqb = min(kSub, a.NQB - p.s * kSub);
        const int last = p.s * kSub + p.nqb - 1;
        for (int qb = p.s * kSub; qb <= last; ++qb) p.scored |= qb_sel(a, qb).scored;
        p.c_hi = last - a.n_local;
        p.nC = max(0, p.c_hi - a.n_init + 1);
        p.nch = p.scored ? (p.nC + kCand - 1) / kCand : 0;
        B.n = max(B.n, p.nch);
    }
    return B;
}

// The chunk ring as both the TMA and the MMA thread see it: the same sequence
// of chunk uses gives both the same slots. A use finds its chunk still in a
// slot (resident: no load) or refills the least recently used slot. Pass 2
// runs the chunks in reverse order, so its first uses find the last chunks of
// pass 1 (min(n, slots) of them) resident; every other use is a fill.
struct ChunkRing {
    int tag[kMaxSlots];
    uint32_t stamp[kMaxSlots];
    int fills[kMaxSlots];
    uint32_t clock;
    int n;
    __device__ __forceinline__ void init(int slots) {
        n = slots;
        clock = 0;
#pragma unroll
        for (int i = 0; i < kMaxSlots; ++i) {
            tag[i] = -1;
            stamp[i] = 0;
            fills[i] = 0;
        }
    }
    __device__ __forceinline__ int take(int t, bool& load) {
        int s = -1;
#pragma unroll
        for (int i = 0; i < kMaxSlots; ++i)
            if (i < n && tag[i] == t) s = i;
        load = s < 0;
        if (load) {
            s = 0;
#pragma unroll
            for (int i = 1; i < kMaxSlots; ++i)
                if (i < n && stamp[i] < stamp[s]) s = i;
            tag[s] = t;
        }
        stamp[s] = ++clock;
        return s;
    }
};

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

// Top-k of one scored query block by one warp over its aggregates Aq[cj]
// (candidate t = n_init + cj), and its output row.
template <bool kMaxLogit>
__device__ __forceinline__ void topk_write(const SelArgs& a, int bg, int qb, const QbSel& q,
                                           float* Aq, int lane) {
    int32_t* out = a.idx_out + ((long long)bg * a.NQB + qb) * a.topk;
    const int c_lo = a.n_init;
    auto key_of = [&](int cj) { return topk::make_key_agg(Aq[cj], c_lo + cj, kMaxLogit); };
    if (q.ksel <= 32) {
        const unsigned long long mine = topk::warp_topk32(q.nC, q.ksel, key_of, lane);
        const int blk = lane < q.ksel ? topk::key_block(mine) : 0x7fffffff;
        int rank = 0;
        for (int i = 0; i < q.ksel; ++i) rank += __shfl_sync(0xffffffffu, blk, i) < blk;
        if (lane < q.ksel) out[q.n_init_q + rank] = blk;
    } else {
        // a pick is marked by a NaN bit pattern that arithmetic never produces;
        // the marks are then read back in ascending order
        auto taken = [&](int cj) { return __float_as_uint(Aq[cj]) == 0xffffffffu; };
        topk::rounds_mark_one_warp(q.nC, q.ksel, key_of, taken,
                                   [&](int t) { Aq[t - c_lo] = __uint_as_float(0xffffffffu); }, lane);
        __syncwarp();
        int pos = q.n_init_q;
        for (int base = 0; base < q.nC; base += 32) {
            const int cj = base + lane;
            const bool pick = cj < q.nC && taken(cj);
            const unsigned m = __ballot_sync(0xffffffffu, pick);
            if (pick) out[pos + __popc(m & ((1u << lane) - 1u))] = c_lo + cj;
            pos += __popc(m);
        }
    }
    for (int x = lane; x < a.topk; x += 32) {
        if (x < q.n_init_q) out[x] = x;
        else if (x >= q.n_init_q + q.ksel && x < q.nF + q.ksel)
            out[x] = q.loc_lo + (x - q.n_init_q - q.ksel);
        else if (x >= q.nF + q.ksel) out[x] = -1;
    }
    if (lane == 0) a.cnt_out[(long long)bg * a.NQB + qb] = q.nF + q.ksel;
}

// Writes the output row of a scored query block whose picks are held one per
// lane (lane < ksel, in any order): ascending, with the forced initial and local
// blocks, -1 padded, and its count.
__device__ __forceinline__ void write_picks(const SelArgs& a, int bg, int qb, const QbSel& q,
                                            unsigned long long mine, int lane) {
    int32_t* out = a.idx_out + ((long long)bg * a.NQB + qb) * a.topk;
    const int blk = lane < q.ksel ? topk::key_block(mine) : 0x7fffffff;
    int rank = 0;
    for (int i = 0; i < q.ksel; ++i) rank += __shfl_sync(0xffffffffu, blk, i) < blk;
    if (lane < q.ksel) out[q.n_init_q + rank] = blk;
    for (int x = lane; x < a.topk; x += 32) {
        if (x < q.n_init_q) out[x] = x;
        else if (x >= q.n_init_q + q.ksel && x < q.nF + q.ksel)
            out[x] = q.loc_lo + (x - q.n_init_q - q.ksel);
        else if (x >= q.nF + q.ksel) out[x] = -1;
    }
    if (lane == 0) a.cnt_out[(long long)bg * a.NQB + qb] = q.nF + q.ksel;
}

// Top-k of one scored query block (ksel <= 32) by kW warps: warp wi takes a
// kW-th of the candidates and keeps its best min(ksel, slice) in fin[wi],
// sorted (level 1); after the barrier, warp 0 merges the kW sorted lists two
// at a time, keeping the best 32 (level 2): every pick is within the best ksel
// of its own slice.
template <bool kMaxLogit, int kW>
__device__ __forceinline__ void topk_split(const SelArgs& a, int bg, int qb, const QbSel& q,
                                           const float* Aq, unsigned long long* fin, int wi,
                                           int lane, int bar_id, bool ok) {
    const int per = (q.nC + kW - 1) / kW;
    const int lo = min(q.nC, wi * per), hi = min(q.nC, lo + per);
    const int k1 = min(q.ksel, hi - lo);
    unsigned long long mine = 0ull;
    if (k1 > 0)
        mine = topk::warp_topk32(hi - lo, k1, [&](int cj) {
            return topk::make_key_agg(Aq[lo + cj], a.n_init + lo + cj, kMaxLogit);
        }, lane);
    fin[wi * 32 + lane] = lane < k1 ? mine : 0ull;
    named_barrier(bar_id, 32 * kW);
    if (wi == 0) {
        unsigned long long best = fin[lane];
#pragma unroll
        for (int w = 1; w < kW; ++w) best = topk::merge_top32(best, fin[w * 32 + lane], lane);
        if (ok) write_picks(a, bg, qb, q, best, lane);
    }
}

__device__ __forceinline__ float max32(const uint32_t* v) {
    float m[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) m[i] = -INFINITY;
#pragma unroll
    for (int j = 0; j < 32; j += 4) {
        const int i = (j >> 2) & 7;
        m[i] = fmaxf(m[i], fmaxf(fmaxf(__uint_as_float(v[j]), __uint_as_float(v[j + 1])),
                                 fmaxf(__uint_as_float(v[j + 2]), __uint_as_float(v[j + 3]))));
    }
    return fmaxf(fmaxf(fmaxf(m[0], m[1]), fmaxf(m[2], m[3])), fmaxf(fmaxf(m[4], m[5]), fmaxf(m[6], m[7])));
}

// sum over 32 scores of 2^(x * c + o), packed two at a time, fixed order
__device__ __forceinline__ float expsum32(const uint32_t* v, float c, float o) {
    const float2 cc = make_float2(c, c), oo = make_float2(o, o);
    float2 acc[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) acc[i] = make_float2(0.f, 0.f);
#pragma unroll
    for (int j = 0; j < 32; j += 2) {
        float2 e = __ffma2_rn(make_float2(__uint_as_float(v[j]), __uint_as_float(v[j + 1])), cc, oo);
        e.x = ex2_approx(e.x);
        e.y = ex2_approx(e.y);
        acc[(j >> 1) & 3] = __fadd2_rn(acc[(j >> 1) & 3], e);
    }
    const float2 s01 = __fadd2_rn(acc[0], acc[1]), s23 = __fadd2_rn(acc[2], acc[3]);
    const float2 s = __fadd2_rn(s01, s23);
    return s.x + s.y;
}

template <bool kMaxLogit, int kSub>
__global__ void __launch_bounds__(kThreads, 1)
select_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmKr,
                 const SelArgs a) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~uintptr_t(1023));
    const uint32_t sb = smem_u32(smem);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    auto bar = [&](int i) { return sb + a.off_bar + 8u * (uint32_t)i; };
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + a.off_misc + 4);
    constexpr int kTok = 64 / kSub;  // tokens per query block

    if (threadIdx.x == 0) {
        for (int q = 0; q < 4; ++q) {
            mbar_init(bar(B_QFULL + q), 1);
            mbar_init(bar(B_QFREE + q), 1);
        }
        for (int s = 0; s < kMaxSlots; ++s) {
            mbar_init(bar(B_KFULL + s), 1);
            mbar_init(bar(B_KEMPTY + s), 1);
        }
        for (int b = 0; b < 4; ++b) {
            mbar_init(bar(B_SFULL + b), 1);
            mbar_init(bar(B_SFREE + b), 128);
        }
        mbar_init(bar(B_DRAIN), 1);
        fence_barrier_init();
        *abort_flag = 0;
    }
    if (warp == 9) {
        tmem_alloc(sb + a.off_misc, kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(smem + a.off_misc);

    if (warp == 8) {
        // ------------------------------------------------ TMA producer
        if (lane == 0) {
            prefetch_tmap(&tmKr);
            prefetch_tmap(&tmQ);
            ChunkRing ring;
            ring.init(a.slots);
            int qloads[2] = {0, 0};
            bool ok = true;
            int ib = 0;
            for (int v = blockIdx.x; ok && v < a.batches; v += gridDim.x, ++ib) {
                const BatchInfo B = batch_info<kSub>(a, v);
                for (int si = 0; ok && si < 2; ++si) {
                    if (!B.sp[si].scored) continue;
                    const int qs = si * a.nq + qloads[si] % a.nq, use = qloads[si] / a.nq;
                    if (use > 0 &&
                        !mbar_wait(bar(B_QFREE + qs), (use - 1) & 1, abort_flag, a.status)) {
                        ok = false;
                        break;
                    }
                    mbar_expect_tx(bar(B_QFULL + qs), kTile);
                    for (int hl = 0; hl < 2; ++hl)
                        for (int dh = 0; dh < 2; ++dh)
                            tma_load_3d(sb + qs * kTile + dh * kHalf + hl * kBox, &tmQ,
                                        bar(B_QFULL + qs), dh * 64, B.sp[si].s * 64, B.hq0 + hl);
                    ++qloads[si];
                }
                auto use = [&](int c) {
                    bool load;
                    const int sl = ring.take(((ib & 0x7fff) << 16) | c, load);
                    if (load) {
                        // the slot's previous fill is done with (its last use has completed)
                        if (ring.fills[sl] > 0 &&
                            !mbar_wait(bar(B_KEMPTY + sl), (ring.fills[sl] - 1) & 1, abort_flag, a.status))
                            return false;
                        mbar_expect_tx(bar(B_KFULL + sl), kTile);
                        const uint32_t dst = sb + a.off_kr + sl * kTile;
                        for (int dh = 0; dh < 2; ++dh)
                            for (int rh = 0; rh < 2; ++rh)
                                tma_load_3d(dst + dh * kHalf + rh * kBox, &tmKr, bar(B_KFULL + sl),
                                            dh * 64, a.n_init + c * kCand + rh * 64, B.bg);
                        ++ring.fills[sl];
                    }
                    return true;
                };
                if (!kMaxLogit)
                    for (int c = 0; ok && c < B.n; ++c) ok = use(c);
                for (int c = B.n - 1; ok && c >= 0; --c) ok = use(c);
            }
            for (int sl = 0; sl < a.slots; ++sl)
                if (ring.fills[sl] > 0) mbar_wait_drain(bar(B_KFULL + sl), (ring.fills[sl] - 1) & 1);
            for (int si = 0; si < 2; ++si)
                for (int j = 0; j < a.nq && j < qloads[si]; ++j) {
                    const int last = qloads[si] - 1 - j;  // the last load into each slot
                    mbar_wait_drain(bar(B_QFULL + si * a.nq + last % a.nq), (last / a.nq) & 1);
                }
        }
    } else if (warp == 9) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_bf16(128, 128, false);
            const uint64_t dQ0 = sdesc_sw128(sb, 16, 1024);
            const uint64_t dKr0 = sdesc_sw128(sb + a.off_kr, 16, 1024);
            ChunkRing ring;
            ring.init(a.slots);
            int qfulls[2] = {0, 0}, k[2] = {0, 0};
            bool ok = true;
            int ib = 0;
            for (int v = blockIdx.x; ok && v < a.batches; v += gridDim.x, ++ib) {
                const BatchInfo B = batch_info<kSub>(a, v);
                bool need_q[2] = {B.sp[0].scored, B.sp[1].scored};
                auto step = [&](int c, bool pass1) {
                    bool load;
                    const int sl = ring.take(((ib & 0x7fff) << 16) | c, load);
                    if (load) {
                        if (!mbar_wait(bar(B_KFULL + sl), ring.fills[sl] & 1, abort_flag, a.status))
                            return false;
                        ++ring.fills[sl];
                    }
                    tc_fence_after();
                    const uint64_t kr = sdesc_at(dKr0, sl * kTile);
                    for (int si = 0; si < 2; ++si) {
                        if (c >= B.sp[si].nch) continue;
                        const int qs = si * a.nq + qfulls[si] % a.nq;
                        if (need_q[si]) {
                            if (!mbar_wait(bar(B_QFULL + qs), (qfulls[si] / a.nq) & 1, abort_flag,
                                           a.status))
                                return false;
                            need_q[si] = false;
                        }
                        const int b = 2 * si + (k[si] & 1);
                        if (k[si] >= 2 &&
                            !mbar_wait(bar(B_SFREE + b), ((k[si] >> 1) - 1) & 1, abort_flag, a.status))
                            return false;
                        tc_fence_after();
                        const uint64_t q = sdesc_at(dQ0, qs * kTile);
#pragma unroll
                        for (int ks = 0; ks < 8; ++ks) {
                            const uint32_t off = (uint32_t)((ks >> 2) * kHalf + (ks & 3) * 32);
                            // pass 1: rows x candidates; pass 2: candidates x rows
                            mma_ss(tmem + 128u * b, sdesc_at(pass1 ? q : kr, off),
                                   sdesc_at(pass1 ? kr : q, off), idesc, ks > 0 ? 1u : 0u);
                        }
                        mma_commit(bar(B_SFULL + b));
                        ++k[si];
                        if (!pass1 && c == 0) {  // the span's last MMA of the batch
                            mma_commit(bar(B_QFREE + qs));
                            ++qfulls[si];
                        }
                    }
                    // One empty phase per fill, committed after the fill's last use: a
                    // pass-2 use, or a pass-1 use of a chunk that does not stay in the
                    // ring for pass 2 (the last `slots` chunks of pass 1 do). The
                    // producer waits for exactly that phase before refilling the slot,
                    // so the barrier never runs two phases ahead of it.
                    if (!pass1 || c < B.n - a.slots) mma_commit(bar(B_KEMPTY + sl));
                    return true;
                };
                if (!kMaxLogit)
                    for (int c = 0; ok && c < B.n; ++c) ok = step(c, true);
                for (int c = B.n - 1; ok && c >= 0; --c) ok = step(c, false);
            }
            mma_commit(bar(B_DRAIN));
            mbar_wait_drain(bar(B_DRAIN), 0);
        }
    } else {
        // ------------------------------------------------ elementwise: warps 4si .. 4si + 3
        const int si = warp >> 2, wq = warp & 3;
        const int r = wq * 32 + lane;  // TMEM lane: pass 1 query row, pass 2 candidate
        const uint32_t lane_base = tmem + ((uint32_t)(wq * 32) << 16);
        float* negM = reinterpret_cast<float*>(smem + a.off_stats) + si * 128;
        float* Aspan = reinterpret_cast<float*>(smem + a.off_A) + (size_t)si * kSub * a.a_stride;
        const float cs = a.scale_log2;
        bool ok = true;
        int kst = 0;  // this span slot's TMEM steps so far (the MMA thread's k[si])
        // wait for the span's next TMEM buffer, load its 128 columns, release it
        auto next_buffer = [&](uint32_t* v) {
            const int b = 2 * si + (kst & 1);
            if (ok) {
                ok = mbar_wait(bar(B_SFULL + b), (kst >> 1) & 1, abort_flag, a.status);
                ok = __all_sync(0xffffffffu, ok);
            }
            if (ok) {
                tc_fence_after();
                tmem_ld128(lane_base + 128u * b, v);
                tc_fence_before();
                mbar_arrive(bar(B_SFREE + b));
            }
            ++kst;
            return ok;
        };
        for (int v = blockIdx.x; v < a.batches; v += gridDim.x) {
            const BatchInfo B = batch_info<kSub>(a, v);
            const SpanInfo sp = si == 0 ? B.sp[0] : B.sp[1];
            if (!sp.present) continue;
            const int qb0 = sp.s * kSub;
            if (!sp.scored) {  // every query block of the span is covered by its budget
                for (int j = 0; j < sp.nqb; ++j)
                    write_unscored(a, B.bg, qb0 + j, qb_sel(a, qb0 + j), r, 128);
                continue;
            }
            uint32_t val[128];
            if constexpr (!kMaxLogit) {
                // ---- pass 1: row r = (head r / 64, token r % 64) of query block j_r
                const int tok = r & 63, j_r = tok / kTok;
                const bool row_ok = sp.s * 64 + tok < a.L && j_r < sp.nqb;
                const int c_hi_r = qb0 + j_r - a.n_local;  // the row's last candidate
                float m = -INFINITY, z = 0.f;
                for (int c = 0; c < sp.nch; ++c) {
                    if (!next_buffer(val)) continue;
                    const int t0 = a.n_init + c * kCand;
                    const int nv = row_ok ? min(kCand, c_hi_r - t0 + 1) : 0;  // valid columns
#pragma unroll
                    for (int g = 0; g < 4; ++g) {
                        uint32_t* x = val + 32 * g;
                        if (32 * g >= nv) continue;
                        if (32 * g + 31 >= nv) {
#pragma unroll
                            for (int j = 0; j < 32; ++j)
                                if (32 * g + j >= nv) x[j] = __float_as_uint(-INFINITY);
                        }
                        if (m == -INFINITY) m = max32(x) * cs;  // the row's first shift
                        float sg = expsum32(x, cs, -m);
                        if (!(sg <= 3.0e38f)) {  // a score far above the shift: move it
                            const float mn = max32(x) * cs;
                            z *= ex2_approx(m - mn);
                            m = mn;
                            sg = expsum32(x, cs, -m);
                        }
                        z += sg;
                    }
                }
                // a row past L or without candidates contributes 2^-inf = 0 in pass 2
                negM[r] = (row_ok && z > 0.f) ? -(m + log2f(z)) : -INFINITY;
                named_barrier(1 + si, 128);
            }
            // ---- pass 2: candidate t of the chunk against the span's 128 rows
            const bool tail = sp.s * 64 + 63 >= a.L;  // rows past L exist in this span
            for (int c = sp.nch - 1; c >= 0; --c) {
                if (!next_buffer(val)) continue;
                const int cj = c * kCand + r, t = a.n_init + cj;
                if (cj >= sp.nC) continue;
#pragma unroll
                for (int j = 0; j < kSub; ++j) {
                    if (j >= sp.nqb || t > qb0 + j - a.n_local) continue;  // not j's candidate
                    float res;
                    if constexpr (kMaxLogit) {
                        float mx = -INFINITY;
#pragma unroll
                        for (int h = 0; h < 2; ++h)
#pragma unroll
                            for (int k2 = 0; k2 < kTok; ++k2) {
                                const int col = h * 64 + j * kTok + k2;
                                const float x = (!tail || sp.s * 64 + j * kTok + k2 < a.L)
                                                    ? __uint_as_float(val[col]) : -INFINITY;
                                mx = fmaxf(mx, x);
                            }
                        res = mx * a.scale;
                    } else {
                        const float2 cc = make_float2(cs, cs);
                        float2 acc[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
                        for (int h = 0; h < 2; ++h)
#pragma unroll
                            for (int k2 = 0; k2 < kTok; k2 += 4) {
                                const int col = h * 64 + j * kTok + k2;
                                const float4 mm = *reinterpret_cast<const float4*>(negM + col);
                                float2 e0 = __ffma2_rn(make_float2(__uint_as_float(val[col]), __uint_as_float(val[col + 1])), cc,
                                                       make_float2(mm.x, mm.y));
                                float2 e1 = __ffma2_rn(make_float2(__uint_as_float(val[col + 2]), __uint_as_float(val[col + 3])), cc,
                                                       make_float2(mm.z, mm.w));
                                e0.x = ex2_approx(e0.x);
                                e0.y = ex2_approx(e0.y);
                                e1.x = ex2_approx(e1.x);
                                e1.y = ex2_approx(e1.y);
                                acc[0] = __fadd2_rn(acc[0], e0);
                                acc[1] = __fadd2_rn(acc[1], e1);
                            }
                        const float2 s = __fadd2_rn(acc[0], acc[1]);
                        res = s.x + s.y;
                    }
                    Aspan[(size_t)j * a.a_stride + cj] = res;
                }
            }
            named_barrier(1 + si, 128);  // every aggregate of the span is written
            // ---- top-k: kW = 4 / kSub warps per query block of the span
            {
                constexpr int kW = 4 / kSub;
                const int j = wq / kW, wi = wq % kW;
                if (j < sp.nqb) {
                    const int qb = qb0 + j;
                    const QbSel q = qb_sel(a, qb);
                    float* Aq = Aspan + (size_t)j * a.a_stride;
                    if (!q.scored) {
                        if (wi == 0) write_unscored(a, B.bg, qb, q, lane, 32);
                    } else if (kW == 1 || q.ksel > 32) {
                        if (wi == 0 && ok) topk_write<kMaxLogit>(a, B.bg, qb, q, Aq, lane);
                    } else {
                        unsigned long long* fin =
                            reinterpret_cast<unsigned long long*>(smem + a.off_fin) + si * 128 + j * 32 * kW;
                        topk_split<kMaxLogit, kW>(a, B.bg, qb, q, Aq, fin, wi, lane,
                                                  3 + 2 * si + j, ok);
                    }
                }
            }
            // pass 2 of the next batch rewrites A and negM only after the next
            // pass-1 barrier (or, for max logits, the barrier below), which every
            // warp reaches after its top-k
            if constexpr (kMaxLogit) named_barrier(1 + si, 128);
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

namespace {
bool use_unit_kernel(const phsa_shape& s) {
    return s.block_size == 64 && (s.L + 63) / 64 <= kSelectUnitMaxNqb;
}
}  // namespace

size_t select_tc_smem_bytes(const phsa_shape& s, int topk) {
    if (use_unit_kernel(s)) return select_tc_unit_smem_bytes(s, topk);
    const int bm = s.block_size;
    return sel_layout_fit((s.L + bm - 1) / bm, 64 / bm).total;
}

cudaError_t launch_select_tc(const void* Q, const void* Krepr, const phsa_shape& s,
                             const phsa_select_params& p, int32_t* idx, int32_t* cnt, int* status,
                             cudaStream_t st) {
    if (use_unit_kernel(s)) return launch_select_tc_unit(Q, Krepr, s, p, idx, cnt, status, st);
    const int bm = s.block_size, kSub = 64 / bm;
    const int T = s.L / bm, NQB = (s.L + bm - 1) / bm;
    CUtensorMap tq, tkr;
    if (!make_tmap_bf16_rows128(&tq, Q, s.L, (uint64_t)s.B * s.Hq, 64)) return cudaErrorInvalidValue;
    // Krepr may be absent when no query block has a candidate (T < 2): the map is
    // then built over Q, which is never read through it.
    if (!make_tmap_bf16_rows128(&tkr, T > 0 ? Krepr : Q, T > 0 ? T : 1,
                                (uint64_t)s.B * s.Hkv, 64))
        return cudaErrorInvalidValue;
    const SelLayout lay = sel_layout_fit(NQB, kSub);
    const bool mx = p.aggregation == PHSA_AGG_MAX_LOGIT;
    auto kern = kSub == 1 ? (mx ? select_tc_kernel<true, 1> : select_tc_kernel<false, 1>)
                : kSub == 2 ? (mx ? select_tc_kernel<true, 2> : select_tc_kernel<false, 2>)
                            : (mx ? select_tc_kernel<true, 4> : select_tc_kernel<false, 4>);
    cudaError_t e =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)lay.total);
    if (e != cudaSuccess) return e;
    int dev = 0, nsm = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
        return e;
    const int nsb = (NQB + kSub - 1) / kSub;
    const int nbat = (nsb + 1) / 2;
    const int BG = s.B * s.Hkv;
    const long long batches = (long long)BG * nbat;
    if (batches == 0) return cudaSuccess;
    SelArgs args{idx, cnt, status, s.Hq, s.Hkv, s.L, T, NQB, p.topk, p.n_init, p.n_local,
                 p.aggregation, nsb, nbat, BG, (int)batches, p.sm_scale * kLog2e, p.sm_scale,
                 lay.nq, lay.slots, lay.a_stride, (uint32_t)lay.kr, (uint32_t)lay.stats,
                 (uint32_t)lay.fin, (uint32_t)lay.A, (uint32_t)lay.bar, (uint32_t)lay.misc};
    ProfScope prof(K_SELECT, st);
    const unsigned grid = (unsigned)(batches < nsm ? batches : nsm);
    kern<<<grid, kThreads, lay.total, st>>>(tq, tkr, args);
    return cudaGetLastError();
}

}  // namespace phsa
