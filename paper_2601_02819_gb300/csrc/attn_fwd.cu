// Stage (c) forward: causal attention over the selected KV blocks (Eq. 10-11;
// Algorithm 1 step 4), one CTA per (query block qb, KV head g), for block
// sizes m = 16, 32, 64.
//
// The G query heads of the KV group are packed into one G*m-row tile, so each
// gathered m x 128 K/V block is loaded once and used by every head of the
// group. Keys are taken in tiles of 64: a key tile holds 64/m consecutive
// entries of the block list (ascending), slots past its end are masked. Tiles
// are visited in order with a double-buffered cp.async pipeline; S = Q K^T
// and O += P V run as bf16 warp MMAs with fp32 accumulators, and the softmax
// is computed online in the log2 domain
// (FlashAttention-style). Inside the query's own block the token-level causal
// mask applies. Outputs: O in bf16 and the natural-log LSE per row.
#include "phsa_common.cuh"
#include "phsa_internal.h"

namespace phsa {

namespace {

// G query heads x m tokens per unit; keys are taken in tiles of kKT = 64,
// assembled from kNb = kKT / m selected blocks (m rows of K and V each).
// (Tiles of 32 keys at m = 16, which halve the shared memory so that more
// CTAs share an SM, measured slower: 989 us against 942 us at 32k.)
template <int G, int BM>
struct FwdCfg {
    static constexpr int kKT = 64;                     // keys per tile
    static constexpr int kNb = kKT / BM;               // selected blocks per key tile
    static constexpr int kWarps = G * BM / 16;
    static constexpr int kThreads = 32 * kWarps;
    static constexpr int kRows = BM * G;
    static constexpr int kTile = kKT * kD * 2;         // one kKT x 128 bf16 key tile
    static constexpr int kQBytes = kRows * kD * 2;   // Q, then the O rows
    static constexpr int kStage = 2 * kTile;           // K and V of one key tile
    static constexpr int kListOff = kQBytes + 2 * kStage;
    static size_t smem_bytes(int topk) { return (size_t)kListOff + (size_t)(topk + 1) * 4; }
};

template <int G, int BM>
__device__ __forceinline__ void load_key_tile(uint32_t st, const __nv_bfloat16* Kg,
                                              const __nv_bfloat16* Vg, const int* blist, int nblk,
                                              int tile, int L, int tid) {
    using C = FwdCfg<G, BM>;
#pragma unroll
    for (int j = 0; j < C::kNb; ++j) {
        const int e = tile * C::kNb + j;
        // a slot past the list is zero-filled (and masked by the caller)
        const int row0 = e < nblk ? blist[e] * BM : 0;
        const int lim = e < nblk ? L : 0;
        load_rows<C::kThreads, BM>(st + j * BM * kD * 2, Kg, row0, lim, tid);
        load_rows<C::kThreads, BM>(st + C::kTile + j * BM * kD * 2, Vg, row0, lim, tid);
    }
}

template <int G, int BM>
__global__ void __launch_bounds__(FwdCfg<G, BM>::kThreads)
attn_fwd_kernel(const __nv_bfloat16* __restrict__ Q, const __nv_bfloat16* __restrict__ K,
                const __nv_bfloat16* __restrict__ V, const int32_t* __restrict__ idx,
                const int32_t* __restrict__ cnt, int Hq, int Hkv, int L, int NQB, int topk,
                float scale_log2, __nv_bfloat16* __restrict__ O, float* __restrict__ lse,
                int* status) {
    using C = FwdCfg<G, BM>;
    extern __shared__ __align__(128) uint8_t smem[];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int unit = blockIdx.x;
    const int qb = NQB - 1 - (unit % NQB);
    const int bg = unit / NQB;
    const int b = bg / Hkv, g = bg % Hkv;
    const long long lu = (long long)bg * NQB + qb;

    const uint32_t sQ = smem_u32(smem);
    const uint32_t sKV = sQ + C::kQBytes;
    int* blist = reinterpret_cast<int*>(smem + C::kListOff);
    if (tid == 0) blist[topk] = compact_block_list(idx + lu * topk, cnt[lu], topk, qb, blist, status);

    const __nv_bfloat16* Kg = K + (size_t)bg * L * kD;
    const __nv_bfloat16* Vg = V + (size_t)bg * L * kD;
    // rows [hl*BM, hl*BM + BM) hold the query block's tokens of head g*G + hl
#pragma unroll
    for (int hl = 0; hl < G; ++hl)
        load_rows<C::kThreads, BM>(sQ + hl * BM * kD * 2,
                                   Q + (size_t)(b * Hq + g * G + hl) * L * kD, qb * BM, L, tid);
    cp_async_commit();
    __syncthreads();
    const int nblk = blist[topk];
    const int ntile = (nblk + C::kNb - 1) / C::kNb;
    if (ntile > 0) load_key_tile<G, BM>(sKV, Kg, Vg, blist, nblk, 0, L, tid);
    cp_async_commit();

    const int tok0 = (warp * 16) % BM + (lane >> 2);  // token of this lane's rows (and +8)
    const int hl = (warp * 16) / BM;                   // head of the warp's 16 rows
    uint32_t qf[8][4];
    float o[16][4];
#pragma unroll
    for (int n = 0; n < 16; ++n)
#pragma unroll
        for (int e = 0; e < 4; ++e) o[n][e] = 0.f;
    float mrow[2] = {-INFINITY, -INFINITY}, lrow[2] = {0.f, 0.f};

    for (int it = 0; it < ntile; ++it) {
        if (it + 1 < ntile) {
            load_key_tile<G, BM>(sKV + ((it + 1) & 1) * C::kStage, Kg, Vg, blist, nblk, it + 1, L,
                                 tid);
            cp_async_commit();
            cp_async_wait<1>();
        } else {
            cp_async_wait<0>();
        }
        __syncthreads();
        if (it == 0) {
#pragma unroll
            for (int kc = 0; kc < 8; ++kc) load_a_frag(sQ, warp * 16, kc, lane, qf[kc]);
        }
        const uint32_t sK = sKV + (it & 1) * C::kStage;
        const uint32_t sV = sK + C::kTile;

        constexpr int kNs = C::kKT / 8;  // n-tiles of 8 keys
        float s[kNs][4];
#pragma unroll
        for (int n = 0; n < kNs; ++n)
#pragma unroll
            for (int e = 0; e < 4; ++e) s[n][e] = 0.f;
#pragma unroll
        for (int kc = 0; kc < 8; ++kc) {
#pragma unroll
            for (int np = 0; np < kNs / 2; ++np) {
                uint32_t bb[4];
                load_b_nk(sK, np * 16, kc, lane, bb);
                mma16816(s[2 * np], qf[kc], bb[0], bb[1]);
                mma16816(s[2 * np + 1], qf[kc], bb[2], bb[3]);
            }
        }
        // key column -> (slot key / BM of the tile, key % BM inside its block);
        // slots past the list are masked, and so are future tokens of the query's
        // own block, which (the list being ascending, every entry <= qb) can only
        // be the list's last entry
        const int nvalid = nblk - it * C::kNb;
        const int dslot = blist[nblk - 1] == qb ? nblk - 1 - it * C::kNb : -1;
#pragma unroll
        for (int n = 0; n < kNs; ++n)
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int key = n * 8 + (lane & 3) * 2 + (e & 1);
                const int j = key / BM, kk = key % BM;
                const int row = tok0 + ((e >> 1) << 3);
                const bool dead = j >= nvalid || (j == dslot && kk > row);
                s[n][e] = dead ? -INFINITY : s[n][e] * scale_log2;
            }
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            float mx = -INFINITY;
#pragma unroll
            for (int n = 0; n < kNs; ++n) mx = fmaxf(mx, fmaxf(s[n][2 * h], s[n][2 * h + 1]));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
            const float mnew = fmaxf(mrow[h], mx);
            const float base = (mnew == -INFINITY) ? 0.f : mnew;
            const float alpha = ex2_sfu(mrow[h] - base);
            mrow[h] = mnew;
            float rs = 0.f;
#pragma unroll
            for (int n = 0; n < kNs; ++n) {
                s[n][2 * h] = ex2_sfu(s[n][2 * h] - base);
                s[n][2 * h + 1] = ex2_sfu(s[n][2 * h + 1] - base);
                rs += s[n][2 * h] + s[n][2 * h + 1];
            }
            lrow[h] = lrow[h] * alpha + rs;
#pragma unroll
            for (int n = 0; n < 16; ++n) {
                o[n][2 * h] *= alpha;
                o[n][2 * h + 1] *= alpha;
            }
        }
        // O += P V, P re-used from the S accumulators as bf16 A fragments.
#pragma unroll
        for (int ks = 0; ks < kNs / 2; ++ks) {
            uint32_t pa[4];
            pa[0] = pack_bf16(s[2 * ks][0], s[2 * ks][1]);
            pa[1] = pack_bf16(s[2 * ks][2], s[2 * ks][3]);
            pa[2] = pack_bf16(s[2 * ks + 1][0], s[2 * ks + 1][1]);
            pa[3] = pack_bf16(s[2 * ks + 1][2], s[2 * ks + 1][3]);
#pragma unroll
            for (int np = 0; np < 8; ++np) {
                uint32_t bb[4];
                load_b_kn(sV, ks * 16, np * 2, lane, bb);
                mma16816(o[2 * np], pa, bb[0], bb[1]);
                mma16816(o[2 * np + 1], pa, bb[2], bb[3]);
            }
        }
        __syncthreads();
    }
    cp_async_wait<0>();
    __syncthreads();

    // Epilogue: normalise, stage the warp's 16 rows in its own Q rows, store.
    const int h = g * G + hl;
    float inv[2];
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
        float l = lrow[hh];
        l += __shfl_xor_sync(0xffffffffu, l, 1);
        l += __shfl_xor_sync(0xffffffffu, l, 2);
        inv[hh] = l > 0.f ? 1.0f / l : 0.f;
        const int i = qb * BM + tok0 + hh * 8;
        if ((lane & 3) == 0 && i < L) {
            lse[(size_t)(b * Hq + h) * L + i] =
                l > 0.f ? (mrow[hh] + log2f(l)) * kLn2 : -INFINITY;
        }
    }
    uint8_t* sq = smem;
#pragma unroll
    for (int n = 0; n < 16; ++n) {
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
            const int r = warp * 16 + (lane >> 2) + hh * 8;
            const int c = n * 8 + (lane & 3) * 2;  // column
            const uint32_t off = swz(r, c >> 3) + (c & 7) * 2;
            *reinterpret_cast<uint32_t*>(sq + off) =
                pack_bf16(o[n][2 * hh] * inv[hh], o[n][2 * hh + 1] * inv[hh]);
        }
    }
    __syncwarp();
    __nv_bfloat16* Oh = O + (size_t)(b * Hq + h) * L * kD;
#pragma unroll
    for (int k = 0; k < 8; ++k) {
        const int e = k * 32 + lane;
        const int r = e >> 4, c = e & 15;
        const int i = qb * BM + (warp * 16) % BM + r;
        if (i < L) {
            const uint4 v = *reinterpret_cast<const uint4*>(sq + swz(warp * 16 + r, c));
            *reinterpret_cast<uint4*>(Oh + (size_t)i * kD + c * 8) = v;
        }
    }
}

template <int G, int BM>
cudaError_t launch_fwd_g(const void* Q, const void* K, const void* V, const int32_t* idx,
                         const int32_t* cnt, const phsa_shape& s, int topk, float sm_scale,
                         void* O, float* lse, int* status, cudaStream_t st) {
    const int NQB = (s.L + BM - 1) / BM;
    const size_t smem = FwdCfg<G, BM>::smem_bytes(topk);
    auto kern = attn_fwd_kernel<G, BM>;
    cudaError_t e =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const long long grid = (long long)s.B * s.Hkv * NQB;
    ProfScope prof(K_FWD, st);
    kern<<<(unsigned)grid, FwdCfg<G, BM>::kThreads, smem, st>>>(
        static_cast<const __nv_bfloat16*>(Q), static_cast<const __nv_bfloat16*>(K),
        static_cast<const __nv_bfloat16*>(V), idx, cnt, s.Hq, s.Hkv, s.L, NQB, topk,
        sm_scale * kLog2e, static_cast<__nv_bfloat16*>(O), lse, status);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_attn_fwd(const void* Q, const void* K, const void* V, const int32_t* idx,
                            const int32_t* cnt, const phsa_shape& s, int topk, float sm_scale,
                            void* O, float* lse, int* status, cudaStream_t st) {
    if ((long long)s.B * s.Hkv * s.L == 0) return cudaSuccess;
    // Two query heads per KV head fill a 128-row tcgen05 tile at every block size
    // (at m < 64 the tile is a 64-token span; its list union must fit in shared
    // memory); a single head, and larger budgets at m < 64, run on the
    // warp-level MMA kernel in this file.
    const int G = s.Hq / s.Hkv, bm = s.block_size;
    if (G == 2 && (bm == 64 || attn_fwd_tc_smem_bytes(s, topk) <= kMaxDynSmem))
        return launch_attn_fwd_tc(Q, K, V, idx, cnt, s, topk, sm_scale, O, lse, status, st);
#define PHSA_FWD(g_, bm_) launch_fwd_g<g_, bm_>(Q, K, V, idx, cnt, s, topk, sm_scale, O, lse, status, st)
    if (G == 2) return bm == 16 ? PHSA_FWD(2, 16) : PHSA_FWD(2, 32);
    return bm == 16 ? PHSA_FWD(1, 16) : bm == 32 ? PHSA_FWD(1, 32) : PHSA_FWD(1, 64);
#undef PHSA_FWD
}

}  // namespace phsa
