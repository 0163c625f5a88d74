// Stage (b): query-to-block relevance and Top-K block selection (Eq. 8;
// Algorithm 1 step 3), one CTA per (query block qb, KV head g), for block
// sizes m = 16, 32, 64.
//
// The G*m query rows of the group are held as bf16 MMA fragments (one warp
// per 16 rows). The candidate representative keys C = [n_init, qb - n_local]
// are streamed through shared memory in tiles of 64 candidates (double-buffered
// cp.async). Scores never leave the SM:
//   pass 1  S = q . Krepr^T * scale, running row max and row sum (online
//           softmax over the candidates only);
//   pass 2  S recomputed; p = exp(S - max) / sum; the column sums over all rows
//           of the group give A[t] (summed per warp by a fixed shuffle tree,
//           then over warps in warp order, so equal columns get equal sums);
//   top-k   min(topk - |F|, |C|) rounds of a block-wide argmax over the 64-bit
//           key (bits(A) << 32 | ~t): larger A first, lower t on exact ties.
// The max-logit rule (agg = 1) makes one pass: A[t] is the column maximum of
// S = q . Krepr^T * scale over the group's rows (rows past L excluded).
// Forced blocks are never scored; the output is ascending and -1 padded.
#include "phsa_common.cuh"
#include "phsa_internal.h"
#include "topk.cuh"

namespace phsa {

namespace {

constexpr int kCT = 64;  // candidates per Krepr tile

template <int G, int BM>
struct SelCfg {
    static constexpr int kWarps = G * BM / 16;
    static constexpr int kThreads = 32 * kWarps;
    static constexpr int kRows = BM * G;
    static constexpr int kQBytes = kRows * kD * 2;
    static constexpr int kTileBytes = kCT * kD * 2;  // one Krepr tile
    static constexpr int kPartOff = kQBytes + 2 * kTileBytes;          // float [kWarps][64]
    static constexpr int kBestOff = kPartOff + kWarps * 64 * 4;        // u64 [kWarps]
    static constexpr int kAOff = kBestOff + kWarps * 8;                // float [nC]
    static size_t smem_bytes(int nqb, int topk) {
        return (size_t)kAOff + (size_t)nqb * 4 + (size_t)topk * 4 + 16;
    }
};

__device__ __forceinline__ unsigned long long u64_max(unsigned long long a, unsigned long long b) {
    return a > b ? a : b;
}

template <int G, int BM>
__global__ void __launch_bounds__(SelCfg<G, BM>::kThreads)
select_blocks_kernel(const __nv_bfloat16* __restrict__ Q, const __nv_bfloat16* __restrict__ Krepr,
                     int Hq, int Hkv, int L, int T, int NQB, int topk, int n_init, int n_local,
                     int agg, float scale_log2, float scale, int32_t* __restrict__ idx_out,
                     int32_t* __restrict__ cnt_out) {
    using C = SelCfg<G, BM>;
    extern __shared__ __align__(128) uint8_t smem[];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int unit = blockIdx.x;
    const int qb = NQB - 1 - (unit % NQB);  // heaviest query blocks first
    const int bg = unit / NQB;
    const int b = bg / Hkv, g = bg % Hkv;
    const long long out_unit = (long long)bg * NQB + qb;
    int32_t* out = idx_out + out_unit * topk;

    const int n_init_q = min(n_init, qb + 1);            // forced initial blocks [0, n_init_q)
    const int loc_lo = max(n_init_q, qb - n_local + 1);  // forced local blocks [loc_lo, qb]
    const int c_lo = n_init, c_hi = qb - n_local;        // candidates [c_lo, c_hi]
    const int nC = max(0, c_hi - c_lo + 1);
    const int nF = n_init_q + (qb - loc_lo + 1);
    const int ksel = topk - nF;

    if (ksel >= nC) {  // budget covers every candidate: no scoring needed
        const int n = nF + nC;
        for (int j = tid; j < topk; j += C::kThreads) {
            int v = -1;
            if (j < n_init_q) v = j;
            else if (j < n_init_q + nC) v = c_lo + (j - n_init_q);
            else if (j < n) v = loc_lo + (j - n_init_q - nC);
            out[j] = v;
        }
        if (tid == 0) cnt_out[out_unit] = n;
        return;
    }

    const uint32_t sQ = smem_u32(smem);
    const uint32_t sK = sQ + C::kQBytes;
    float* part = reinterpret_cast<float*>(smem + C::kPartOff);
    unsigned long long* wbest = reinterpret_cast<unsigned long long*>(smem + C::kBestOff);
    float* A = reinterpret_cast<float*>(smem + C::kAOff);
    int* sel = reinterpret_cast<int*>(smem + C::kAOff + (size_t)NQB * 4);

    // Query rows of every head of the group: rows [hl*BM, hl*BM + BM) hold head g*G + hl.
#pragma unroll
    for (int hl = 0; hl < G; ++hl) {
        const __nv_bfloat16* Qh = Q + ((size_t)(b * Hq + g * G + hl) * L) * kD;
        load_rows<C::kThreads, BM>(sQ + hl * BM * kD * 2, Qh, qb * BM, L, tid);
    }
    const __nv_bfloat16* Kr = Krepr + (size_t)bg * T * kD;
    const int n_tiles = (nC + kCT - 1) / kCT;
    load_rows<C::kThreads, kCT>(sK, Kr, c_lo, c_hi + 1, tid);
    cp_async_commit();

    // Row bookkeeping: this lane holds rows r0 and r0 + 8 of the warp's 16
    // (row r: token r % BM of head r / BM).
    const int r0 = warp * 16 + (lane >> 2);
    const bool row_ok0 = qb * BM + (r0 & (BM - 1)) < L;
    const bool row_ok1 = qb * BM + ((r0 + 8) & (BM - 1)) < L;

    uint32_t qf[8][4];
    float mrow[2] = {-INFINITY, -INFINITY}, zrow[2] = {0.f, 0.f}, inv_z[2] = {0.f, 0.f};

    const int n_pass = agg ? 1 : 2;
    for (int pass = 0; pass < n_pass; ++pass) {
        for (int j = 0; j < n_tiles; ++j) {
            const int it = pass * n_tiles + j;
            if (it + 1 < n_pass * n_tiles) {
                const int jn = (j + 1 < n_tiles) ? j + 1 : 0;
                load_rows<C::kThreads, kCT>(sK + ((it + 1) & 1) * C::kTileBytes, Kr,
                                            c_lo + jn * kCT, c_hi + 1, tid);
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
            const uint32_t kt = sK + (it & 1) * C::kTileBytes;
            float acc[8][4];
#pragma unroll
            for (int n = 0; n < 8; ++n)
#pragma unroll
                for (int e = 0; e < 4; ++e) acc[n][e] = 0.f;
#pragma unroll
            for (int kc = 0; kc < 8; ++kc) {
#pragma unroll
                for (int np = 0; np < 4; ++np) {
                    uint32_t bb[4];
                    load_b_nk(kt, np * 16, kc, lane, bb);
                    mma16816(acc[2 * np], qf[kc], bb[0], bb[1]);
                    mma16816(acc[2 * np + 1], qf[kc], bb[2], bb[3]);
                }
            }
            // scale (to the log2 domain for the softmax) and mask columns past the
            // candidate range; for max logits also the rows past L
            const int col0 = c_lo + j * kCT + (lane & 3) * 2;
            const float sc = agg ? scale : scale_log2;
#pragma unroll
            for (int n = 0; n < 8; ++n)
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int t = col0 + n * 8 + (e & 1);
                    const bool row_ok = e < 2 ? row_ok0 : row_ok1;
                    acc[n][e] = (t <= c_hi && (row_ok || !agg)) ? acc[n][e] * sc : -INFINITY;
                }
            if (agg) {
                // column maxima over this warp's rows, then over the warps in warp order
#pragma unroll
                for (int n = 0; n < 8; ++n) {
#pragma unroll
                    for (int e = 0; e < 2; ++e) {
                        float v = fmaxf(acc[n][e], acc[n][e + 2]);
                        v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 4));
                        v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 8));
                        v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 16));
                        if (lane < 4) part[warp * 64 + n * 8 + lane * 2 + e] = v;
                    }
                }
                __syncthreads();
                for (int x = tid; x < kCT; x += C::kThreads) {
                    float a = -INFINITY;
#pragma unroll
                    for (int w = 0; w < C::kWarps; ++w) a = fmaxf(a, part[w * 64 + x]);
                    const int c = j * kCT + x;
                    if (c < nC) A[c] = a;
                }
            } else if (pass == 0) {
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    float mx = -INFINITY;
#pragma unroll
                    for (int n = 0; n < 8; ++n) mx = fmaxf(mx, fmaxf(acc[n][2 * h], acc[n][2 * h + 1]));
                    const float mnew = fmaxf(mrow[h], mx);
                    if (mnew == -INFINITY) continue;
                    float s = 0.f;
#pragma unroll
                    for (int n = 0; n < 8; ++n)
                        s += exp2f(acc[n][2 * h] - mnew) + exp2f(acc[n][2 * h + 1] - mnew);
                    zrow[h] = zrow[h] * exp2f(mrow[h] - mnew) + s;
                    mrow[h] = mnew;
                }
            } else {
                // column sums of p over this warp's rows
#pragma unroll
                for (int n = 0; n < 8; ++n) {
#pragma unroll
                    for (int e = 0; e < 2; ++e) {
                        float v = exp2f(acc[n][e] - mrow[0]) * inv_z[0] +
                                  exp2f(acc[n][e + 2] - mrow[1]) * inv_z[1];
                        v += __shfl_xor_sync(0xffffffffu, v, 4);
                        v += __shfl_xor_sync(0xffffffffu, v, 8);
                        v += __shfl_xor_sync(0xffffffffu, v, 16);
                        if (lane < 4) part[warp * 64 + n * 8 + lane * 2 + e] = v;
                    }
                }
                __syncthreads();
                for (int x = tid; x < kCT; x += C::kThreads) {
                    float a = 0.f;
#pragma unroll
                    for (int w = 0; w < C::kWarps; ++w) a += part[w * 64 + x];
                    const int c = j * kCT + x;
                    if (c < nC) A[c] = (a >= 0.f) ? a : 0.f;  // NaN inputs rank as zero
                }
            }
            __syncthreads();
        }
        if (pass == 0) {
            // combine the four lanes that share a row
#pragma unroll
            for (int h = 0; h < 2; ++h) {
#pragma unroll
                for (int off = 1; off <= 2; off <<= 1) {
                    const float mo = __shfl_xor_sync(0xffffffffu, mrow[h], off);
                    const float zo = __shfl_xor_sync(0xffffffffu, zrow[h], off);
                    const float mn = fmaxf(mrow[h], mo);
                    const float za = mrow[h] == -INFINITY ? 0.f : zrow[h] * exp2f(mrow[h] - mn);
                    const float zb = mo == -INFINITY ? 0.f : zo * exp2f(mo - mn);
                    mrow[h] = mn;
                    zrow[h] = za + zb;
                }
            }
            inv_z[0] = (row_ok0 && zrow[0] > 0.f) ? 1.0f / zrow[0] : 0.f;
            inv_z[1] = (row_ok1 && zrow[1] > 0.f) ? 1.0f / zrow[1] : 0.f;
            if (!row_ok0) mrow[0] = 0.f;
            if (!row_ok1) mrow[1] = 0.f;
        }
    }

    // Top-k over A by (A desc, t asc) on keys whose unsigned order is that of
    // A (topk.cuh); a taken candidate is marked by a NaN bit pattern that
    // arithmetic never produces.
    constexpr unsigned kTaken = 0xffffffffu;
    for (int r = 0; r < ksel; ++r) {
        unsigned long long best = 0ull;
        for (int c = tid; c < nC; c += C::kThreads) {
            const float a = A[c];
            if (__float_as_uint(a) != kTaken) best = u64_max(best, topk::make_key_agg(a, c_lo + c, agg != 0));
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
            const unsigned long long o = __shfl_xor_sync(0xffffffffu, best, off);
            best = u64_max(best, o);
        }
        if (lane == 0) wbest[warp] = best;
        __syncthreads();
        if (tid == 0) {
            unsigned long long bb = 0ull;
            for (int w = 0; w < C::kWarps; ++w) bb = u64_max(bb, wbest[w]);
            // every untaken candidate has a nonzero key, so bb != 0 while r < ksel < nC
            const int t = bb ? (int)(0xffffffffu - (unsigned)(bb & 0xffffffffull)) : c_lo;
            sel[r] = t;
            if (t >= c_lo && t <= c_hi) A[t - c_lo] = __uint_as_float(kTaken);
        }
        __syncthreads();
    }

    // Ascending output: initial blocks, the chosen candidates sorted, local blocks.
    for (int j = tid; j < topk; j += C::kThreads) {
        if (j < n_init_q) out[j] = j;
        else if (j >= n_init_q + ksel && j < nF + ksel) out[j] = loc_lo + (j - n_init_q - ksel);
        else if (j >= nF + ksel) out[j] = -1;
    }
    for (int j = tid; j < ksel; j += C::kThreads) {
        const int v = sel[j];
        int rank = 0;
        for (int i = 0; i < ksel; ++i) rank += sel[i] < v;
        out[n_init_q + rank] = v;
    }
    if (tid == 0) cnt_out[out_unit] = nF + ksel;
}

template <int G, int BM>
cudaError_t launch_select_g(const phsa_shape& s, const phsa_select_params& p, const void* Q,
                            const void* Krepr, int32_t* idx, int32_t* cnt, cudaStream_t st) {
    const int T = s.L / BM, NQB = (s.L + BM - 1) / BM;
    const size_t smem = SelCfg<G, BM>::smem_bytes(NQB, p.topk);
    auto kern = select_blocks_kernel<G, BM>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    const long long grid = (long long)s.B * s.Hkv * NQB;
    ProfScope prof(K_SELECT, st);
    kern<<<(unsigned)grid, SelCfg<G, BM>::kThreads, smem, st>>>(
        static_cast<const __nv_bfloat16*>(Q), static_cast<const __nv_bfloat16*>(Krepr), s.Hq,
        s.Hkv, s.L, T, NQB, p.topk, p.n_init, p.n_local, p.aggregation, p.sm_scale * kLog2e,
        p.sm_scale, idx, cnt);
    return cudaGetLastError();
}

}  // namespace

size_t select_smem_bytes(const phsa_shape& s, int topk) {
    const int bm = s.block_size, NQB = (s.L + bm - 1) / bm;
    const int G = s.Hq / s.Hkv;
    if (G == 2 && bm == kM) return select_tc_smem_bytes(s, topk);
    // every instantiation has the same layout apart from the Q rows
    return G == 2 ? SelCfg<2, 64>::smem_bytes(NQB, topk) : SelCfg<1, 64>::smem_bytes(NQB, topk);
}

cudaError_t launch_select_blocks(const void* Q, const void* Krepr, const phsa_shape& s,
                                 const phsa_select_params& p, int32_t* idx, int32_t* cnt,
                                 int* status, cudaStream_t st) {
    const int bm = s.block_size;
    if ((long long)s.B * s.Hkv * ((s.L + bm - 1) / bm) == 0) return cudaSuccess;
    // Two query heads per KV head at m = 64 fill a 128-row tcgen05 tile
    // (select_tc.cu); every other group size and block size runs on the
    // warp-level MMA kernel in this file.
    const int G = s.Hq / s.Hkv;
    if (G == 2 && bm == 64) return launch_select_tc(Q, Krepr, s, p, idx, cnt, status, st);
    if (G == 2)
        return bm == 16 ? launch_select_g<2, 16>(s, p, Q, Krepr, idx, cnt, st)
                        : launch_select_g<2, 32>(s, p, Q, Krepr, idx, cnt, st);
    return bm == 16   ? launch_select_g<1, 16>(s, p, Q, Krepr, idx, cnt, st)
           : bm == 32 ? launch_select_g<1, 32>(s, p, Q, Krepr, idx, cnt, st)
                      : launch_select_g<1, 64>(s, p, Q, Krepr, idx, cnt, st);
}

}  // namespace phsa
