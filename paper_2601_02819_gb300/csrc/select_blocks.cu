// Stage (b): query-to-block relevance and Top-K block selection (Eq. 8;
// Algorithm 1 step 3), one CTA per (query block qb, KV head g), for block
// sizes m = 16, 32, 64.
//
// The G*m query rows of the group are held as bf16 MMA fragments; eight warps
// split each tile of 64 candidates as (groups of 16 rows) x (groups of
// candidates). The candidate representative keys C = [n_init, qb - n_local]
// are streamed through shared memory in those tiles (double-buffered cp.async).
// Scores never leave the SM:
//   pass 1  S = q . Krepr^T * scale, running row max and row sum (online
//           softmax over the candidates only), merged over the candidate
//           groups in group order;
//   pass 2  S recomputed; p = exp(S - max) / sum; the column sums over all rows
//           of the group give A[t] (summed per warp by a fixed shuffle tree,
//           then over the row groups in order, so equal columns get equal sums);
//   top-k   over the 64-bit key (bits(A) << 32 | ~t): larger A first, lower t
//           on exact ties; the two-level selection of topk.cuh (per-warp
//           finalists, then ranks) for budgets <= 32 and <= 2048 candidates,
//           else min(topk - |F|, |C|) rounds of a block-wide argmax.
// The max-logit rule (agg = 1) makes one pass: A[t] is the column maximum of
// S = q . Krepr^T * scale over the group's rows (rows past L excluded).
// Forced blocks are never scored; the output is ascending and -1 padded.
#include <atomic>

#include "phsa_common.cuh"
#include "phsa_internal.h"
#include "topk.cuh"

namespace phsa {

namespace {

constexpr int kCT = 64;  // candidates per Krepr tile

// A CTA takes the kP = 64/m consecutive query blocks of one 64-token span
// (their G*64 query rows) so that every candidate tile is loaded once for all
// of them. Eight warps: kRowWarps groups of 16 rows x kColWarps groups of the
// tile's 64 candidates. Row r = (j*G + hl)*m + tok: query block j of the span,
// head hl, token tok; every row group lies inside one query block.
template <int G, int BM>
struct SelCfg {
    static constexpr int kP = 64 / BM;  // query blocks per CTA
    static constexpr int kRows = 64 * G;
    static constexpr int kRowWarps = kRows / 16;
    static constexpr int kColWarps = 8 / kRowWarps;
    static constexpr int kWarps = kRowWarps * kColWarps;
    static constexpr int kThreads = 32 * kWarps;
    static constexpr int kCols = kCT / kColWarps;
    static constexpr int kNt = kCols / 8;               // n-tiles of 8 candidates per warp
    static constexpr int kRwPerQb = kRowWarps / kP;     // row groups of one query block
    static_assert(kWarps == 8 && kNt % 2 == 0 && kRwPerQb >= 1, "warp split");
    static constexpr int kQBytes = kRows * kD * 2;
    static constexpr int kTileBytes = kCT * kD * 2;                    // one Krepr tile
    static constexpr int kPartOff = kQBytes + 2 * kTileBytes;          // float [kRowWarps][64]
    static constexpr int kStatOff = kPartOff + kRowWarps * kCT * 4;    // float2 [kColWarps][kRows]
    static constexpr int kFinOff = kStatOff + kColWarps * kRows * 8;   // u64 [8 * kFinalMax]
    static constexpr int kAOff = kFinOff + 8 * topk::kFinalMax * 8;    // float [kP][NQB]
    static size_t smem_bytes(int nqb, int topk) {
        return (size_t)kAOff + (size_t)kP * nqb * 4 + (size_t)topk * 4 + 16;
    }
};

__device__ __forceinline__ unsigned long long u64_max(unsigned long long a, unsigned long long b) {
    return a > b ? a : b;
}

// The forced sets and the candidate range of query block qb (Algorithm 1).
struct QbSel {
    int n_init_q, loc_lo, c_hi, nC, nF, ksel;
};
__device__ __forceinline__ QbSel qb_sel(int qb, int topk, int n_init, int n_local) {
    QbSel q;
    q.n_init_q = min(n_init, qb + 1);                  // forced initial blocks [0, n_init_q)
    q.loc_lo = max(q.n_init_q, qb - n_local + 1);      // forced local blocks [loc_lo, qb]
    q.c_hi = qb - n_local;                             // candidates [n_init, c_hi]
    q.nC = max(0, q.c_hi - n_init + 1);
    q.nF = q.n_init_q + (qb - q.loc_lo + 1);
    q.ksel = topk - q.nF;
    return q;
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
    const int rw = warp % C::kRowWarps, cw = warp / C::kRowWarps;
    const int NSB = (NQB + C::kP - 1) / C::kP;
    const int sb = NSB - 1 - (int)(blockIdx.x % NSB);  // heaviest spans first
    const int bg = blockIdx.x / NSB;
    const int b = bg / Hkv, g = bg % Hkv;
    const int qb0 = sb * C::kP;
    const int nq = min(C::kP, NQB - qb0);  // query blocks of this span
    const int c_lo = n_init;

    // Query blocks whose budget covers every candidate need no scoring.
    bool any_scored = false;
    int c_hi_all = c_lo - 1;
    for (int j = 0; j < nq; ++j) {
        const QbSel q = qb_sel(qb0 + j, topk, n_init, n_local);
        const long long ou = (long long)bg * NQB + qb0 + j;
        if (q.ksel >= q.nC) {
            const int n = q.nF + q.nC;
            for (int x = tid; x < topk; x += C::kThreads) {
                int v = -1;
                if (x < q.n_init_q) v = x;
                else if (x < q.n_init_q + q.nC) v = c_lo + (x - q.n_init_q);
                else if (x < n) v = q.loc_lo + (x - q.n_init_q - q.nC);
                idx_out[ou * topk + x] = v;
            }
            if (tid == 0) cnt_out[ou] = n;
        } else {
            any_scored = true;
        }
        c_hi_all = max(c_hi_all, q.c_hi);
    }
    if (!any_scored) return;
    const int nC_all = c_hi_all - c_lo + 1;  // the union of the span's candidate ranges

    const uint32_t sQ = smem_u32(smem);
    const uint32_t sK = sQ + C::kQBytes;
    float* part = reinterpret_cast<float*>(smem + C::kPartOff);
    float2* stat = reinterpret_cast<float2*>(smem + C::kStatOff);
    unsigned long long* fin = reinterpret_cast<unsigned long long*>(smem + C::kFinOff);
    float* Aall = reinterpret_cast<float*>(smem + C::kAOff);  // A of query block j at j * NQB
    int* sel = reinterpret_cast<int*>(smem + C::kAOff + (size_t)C::kP * NQB * 4);

    // Query rows: block j of the span, head hl at rows (j*G + hl)*BM (zero past L).
#pragma unroll
    for (int j = 0; j < C::kP; ++j)
#pragma unroll
        for (int hl = 0; hl < G; ++hl) {
            const __nv_bfloat16* Qh = Q + ((size_t)(b * Hq + g * G + hl) * L) * kD;
            load_rows<C::kThreads, BM>(sQ + (j * G + hl) * BM * kD * 2, Qh, (qb0 + j) * BM, L, tid);
        }
    const __nv_bfloat16* Kr = Krepr + (size_t)bg * T * kD;
    const int n_tiles = (nC_all + kCT - 1) / kCT;
    load_rows<C::kThreads, kCT>(sK, Kr, c_lo, c_hi_all + 1, tid);
    cp_async_commit();

    // Row bookkeeping: this lane holds rows r0 and r0 + 8 of its row group's 16;
    // the group's query block jq bounds its candidates by c_hi_q.
    const int r0 = rw * 16 + (lane >> 2);
    const int jq = rw / C::kRwPerQb;
    const int c_hi_q = qb0 + jq - n_local;
    const int tok0 = r0 % BM;
    const bool row_ok0 = (qb0 + jq) * BM + tok0 < L;
    const bool row_ok1 = (qb0 + jq) * BM + tok0 + 8 < L;

    uint32_t qf[8][4];
    float mrow[2] = {-INFINITY, -INFINITY}, zrow[2] = {0.f, 0.f}, inv_z[2] = {0.f, 0.f};

    const int n_pass = agg ? 1 : 2;
    for (int pass = 0; pass < n_pass; ++pass) {
        for (int jt = 0; jt < n_tiles; ++jt) {
            const int it = pass * n_tiles + jt;
            if (it + 1 < n_pass * n_tiles) {
                const int jn = (jt + 1 < n_tiles) ? jt + 1 : 0;
                load_rows<C::kThreads, kCT>(sK + ((it + 1) & 1) * C::kTileBytes, Kr,
                                            c_lo + jn * kCT, c_hi_all + 1, tid);
                cp_async_commit();
                cp_async_wait<1>();
            } else {
                cp_async_wait<0>();
            }
            __syncthreads();
            if (it == 0) {
#pragma unroll
                for (int kc = 0; kc < 8; ++kc) load_a_frag(sQ, rw * 16, kc, lane, qf[kc]);
            }
            const uint32_t kt = sK + (it & 1) * C::kTileBytes;
            float acc[C::kNt][4];
#pragma unroll
            for (int n = 0; n < C::kNt; ++n)
#pragma unroll
                for (int e = 0; e < 4; ++e) acc[n][e] = 0.f;
#pragma unroll
            for (int kc = 0; kc < 8; ++kc) {
#pragma unroll
                for (int np = 0; np < C::kNt / 2; ++np) {
                    uint32_t bb[4];
                    load_b_nk(kt, cw * C::kCols + np * 16, kc, lane, bb);
                    mma16816(acc[2 * np], qf[kc], bb[0], bb[1]);
                    mma16816(acc[2 * np + 1], qf[kc], bb[2], bb[3]);
                }
            }
            // scale (to the log2 domain for the softmax) and mask columns past this
            // row group's candidate range; for max logits also the rows past L
            const int col0 = c_lo + jt * kCT + cw * C::kCols + (lane & 3) * 2;
            const float sc = agg ? scale : scale_log2;
#pragma unroll
            for (int n = 0; n < C::kNt; ++n)
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int t = col0 + n * 8 + (e & 1);
                    const bool row_ok = e < 2 ? row_ok0 : row_ok1;
                    acc[n][e] = (t <= c_hi_q && (row_ok || !agg)) ? acc[n][e] * sc : -INFINITY;
                }
            if (agg || pass == 1) {
                // column maxima (max logit) or column sums of p (softmax) over this
                // warp's 16 rows, then over the query block's row groups in order
#pragma unroll
                for (int n = 0; n < C::kNt; ++n) {
#pragma unroll
                    for (int e = 0; e < 2; ++e) {
                        float v;
                        if (agg) {
                            v = fmaxf(acc[n][e], acc[n][e + 2]);
                            v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 4));
                            v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 8));
                            v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 16));
                        } else {
                            v = ex2_sfu(acc[n][e] - mrow[0]) * inv_z[0] +
                                ex2_sfu(acc[n][e + 2] - mrow[1]) * inv_z[1];
                            v += __shfl_xor_sync(0xffffffffu, v, 4);
                            v += __shfl_xor_sync(0xffffffffu, v, 8);
                            v += __shfl_xor_sync(0xffffffffu, v, 16);
                        }
                        if (lane < 4) part[rw * kCT + cw * C::kCols + n * 8 + lane * 2 + e] = v;
                    }
                }
                __syncthreads();
                for (int x = tid; x < C::kP * kCT; x += C::kThreads) {
                    const int j = x / kCT, xc = x % kCT;
                    const int c = jt * kCT + xc;
                    if (j < nq && c < nC_all) {
                        float a = agg ? -INFINITY : 0.f;
#pragma unroll
                        for (int w = 0; w < C::kRwPerQb; ++w) {
                            const float v = part[(j * C::kRwPerQb + w) * kCT + xc];
                            a = agg ? fmaxf(a, v) : a + v;
                        }
                        Aall[j * NQB + c] = (agg || a >= 0.f) ? a : 0.f;  // NaN inputs rank as zero
                    }
                }
            } else {
                // pass 1: running max and sum of each row over this lane's columns
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    float mx = -INFINITY;
#pragma unroll
                    for (int n = 0; n < C::kNt; ++n) mx = fmaxf(mx, fmaxf(acc[n][2 * h], acc[n][2 * h + 1]));
                    const float mnew = fmaxf(mrow[h], mx);
                    if (mnew == -INFINITY) continue;
                    float s = 0.f;
#pragma unroll
                    for (int n = 0; n < C::kNt; ++n)
                        s += ex2_sfu(acc[n][2 * h] - mnew) + ex2_sfu(acc[n][2 * h + 1] - mnew);
                    zrow[h] = zrow[h] * ex2_sfu(mrow[h] - mnew) + s;
                    mrow[h] = mnew;
                }
            }
            __syncthreads();
        }
        if (pass == 0 && !agg) {
            // combine the four lanes that share a row, then the column groups in order
#pragma unroll
            for (int h = 0; h < 2; ++h) {
#pragma unroll
                for (int off = 1; off <= 2; off <<= 1) {
                    const float mo = __shfl_xor_sync(0xffffffffu, mrow[h], off);
                    const float zo = __shfl_xor_sync(0xffffffffu, zrow[h], off);
                    const float mn = fmaxf(mrow[h], mo);
                    const float za = mrow[h] == -INFINITY ? 0.f : zrow[h] * ex2_sfu(mrow[h] - mn);
                    const float zb = mo == -INFINITY ? 0.f : zo * ex2_sfu(mo - mn);
                    mrow[h] = mn;
                    zrow[h] = za + zb;
                }
            }
            if ((lane & 3) == 0) {
                stat[cw * C::kRows + r0] = make_float2(mrow[0], zrow[0]);
                stat[cw * C::kRows + r0 + 8] = make_float2(mrow[1], zrow[1]);
            }
            __syncthreads();
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int r = r0 + 8 * h;
                float mx = -INFINITY;
#pragma unroll
                for (int c = 0; c < C::kColWarps; ++c) mx = fmaxf(mx, stat[c * C::kRows + r].x);
                float z = 0.f;
#pragma unroll
                for (int c = 0; c < C::kColWarps; ++c) {
                    const float2 st = stat[c * C::kRows + r];
                    if (st.x != -INFINITY) z += st.y * ex2_sfu(st.x - mx);
                }
                mrow[h] = mx;
                zrow[h] = z;
            }
            inv_z[0] = (row_ok0 && zrow[0] > 0.f) ? 1.0f / zrow[0] : 0.f;
            inv_z[1] = (row_ok1 && zrow[1] > 0.f) ? 1.0f / zrow[1] : 0.f;
            if (!row_ok0) mrow[0] = 0.f;
            if (!row_ok1) mrow[1] = 0.f;
        }
    }

    // Top-k of every scored query block of the span over its own candidates,
    // by (A desc, t asc) on keys whose unsigned order is that of A (topk.cuh):
    // the two-level selection over the eight warps when it applies, else rounds
    // of a block-wide maximum in which a taken candidate is marked by a NaN bit
    // pattern that arithmetic never produces.
    const bool mx_rule = agg != 0;
    for (int j = 0; j < nq; ++j) {
        const int qb = qb0 + j;
        const QbSel q = qb_sel(qb, topk, n_init, n_local);
        if (q.ksel >= q.nC) continue;  // written above
        float* A = Aall + (size_t)j * NQB;
        const int nC = q.nC, ksel = q.ksel, c_hi = q.c_hi;
        if (topk::two_level(nC, ksel)) {
            topk::level1(nC, ksel, [&](int cj) { return topk::make_key_agg(A[cj], c_lo + cj, mx_rule); },
                         fin, warp, lane);
            __syncthreads();
            topk::level2(fin, ksel, sel, tid);
            __syncthreads();
        } else {
            constexpr unsigned kTaken = 0xffffffffu;
            for (int r = 0; r < ksel; ++r) {
                unsigned long long best = 0ull;
                for (int c = tid; c < nC; c += C::kThreads) {
                    const float a = A[c];
                    if (__float_as_uint(a) != kTaken) best = u64_max(best, topk::make_key_agg(a, c_lo + c, mx_rule));
                }
#pragma unroll
                for (int off = 16; off > 0; off >>= 1) {
                    const unsigned long long o = __shfl_xor_sync(0xffffffffu, best, off);
                    best = u64_max(best, o);
                }
                if (lane == 0) fin[warp] = best;
                __syncthreads();
                if (tid == 0) {
                    unsigned long long bb = 0ull;
                    for (int w = 0; w < C::kWarps; ++w) bb = u64_max(bb, fin[w]);
                    // every untaken candidate has a nonzero key, so bb != 0 while r < ksel < nC
                    const int t = bb ? (int)(0xffffffffu - (unsigned)(bb & 0xffffffffull)) : c_lo;
                    sel[r] = t;
                    if (t >= c_lo && t <= c_hi) A[t - c_lo] = __uint_as_float(kTaken);
                }
                __syncthreads();
            }
        }
        // Ascending output: initial blocks, the chosen candidates sorted, local blocks.
        int32_t* out = idx_out + ((long long)bg * NQB + qb) * topk;
        for (int x = tid; x < topk; x += C::kThreads) {
            if (x < q.n_init_q) out[x] = x;
            else if (x >= q.n_init_q + ksel && x < q.nF + ksel) out[x] = q.loc_lo + (x - q.n_init_q - ksel);
            else if (x >= q.nF + ksel) out[x] = -1;
        }
        for (int x = tid; x < ksel; x += C::kThreads) {
            const int v = sel[x];
            int rank = 0;
            for (int i = 0; i < ksel; ++i) rank += sel[i] < v;
            out[q.n_init_q + rank] = v;
        }
        if (tid == 0) cnt_out[(long long)bg * NQB + qb] = q.nF + ksel;
        __syncthreads();  // sel and fin are reused by the next query block
    }
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
    const int NSB = (NQB + SelCfg<G, BM>::kP - 1) / SelCfg<G, BM>::kP;
    const long long grid = (long long)s.B * s.Hkv * NSB;
    ProfScope prof(K_SELECT, st);
    kern<<<(unsigned)grid, SelCfg<G, BM>::kThreads, smem, st>>>(
        static_cast<const __nv_bfloat16*>(Q), static_cast<const __nv_bfloat16*>(Krepr), s.Hq,
        s.Hkv, s.L, T, NQB, p.topk, p.n_init, p.n_local, p.aggregation, p.sm_scale * kLog2e,
        p.sm_scale, idx, cnt);
    return cudaGetLastError();
}

}  // namespace

// Switch point of the GQA-pair selection at m = 16 and 32: the tcgen05 kernel
// while its shared memory stays at or below this many bytes, else the
// warp-MMA kernel. Only phsa_test_set_select_tc_limit lowers it, so that tests
// reach the warp-MMA pair kernels on short sequences.
std::atomic<size_t> g_select_tc_limit{kMaxDynSmem};

bool select_uses_tc(const phsa_shape& s, int topk) {
    if (s.Hq != 2 * s.Hkv) return false;
    return s.block_size == 64 || select_tc_smem_bytes(s, topk) <= g_select_tc_limit.load();
}

size_t select_smem_bytes(const phsa_shape& s, int topk) {
    const int bm = s.block_size, NQB = (s.L + bm - 1) / bm;
    const int G = s.Hq / s.Hkv;
    if (G == 2) {
        // the tcgen05 kernel, unless its per-block sums outgrow shared memory at
        // m < 64 (spans beyond about 64k tokens at m = 16): then the warp-MMA one
        if (select_uses_tc(s, topk)) return select_tc_smem_bytes(s, topk);
        return bm == 16 ? SelCfg<2, 16>::smem_bytes(NQB, topk) : SelCfg<2, 32>::smem_bytes(NQB, topk);
    }
    return bm == 16   ? SelCfg<1, 16>::smem_bytes(NQB, topk)
           : bm == 32 ? SelCfg<1, 32>::smem_bytes(NQB, topk)
                      : SelCfg<1, 64>::smem_bytes(NQB, topk);
}

cudaError_t launch_select_blocks(const void* Q, const void* Krepr, const phsa_shape& s,
                                 const phsa_select_params& p, int32_t* idx, int32_t* cnt,
                                 int* status, cudaStream_t st) {
    const int bm = s.block_size;
    if ((long long)s.B * s.Hkv * ((s.L + bm - 1) / bm) == 0) return cudaSuccess;
    // Two query heads per KV head fill a 128-row tcgen05 tile (select_tc.cu;
    // at m = 16 and 32 the tile holds the query blocks of a 64-token span, as
    // long as their per-block sums fit in shared memory); a single head, and
    // longer sequences at m < 64, run on the warp-level MMA kernel in this file.
    const int G = s.Hq / s.Hkv;
    if (G == 2) {
        if (select_uses_tc(s, p.topk))
            return launch_select_tc(Q, Krepr, s, p, idx, cnt, status, st);
        return bm == 16 ? launch_select_g<2, 16>(s, p, Q, Krepr, idx, cnt, st)
                        : launch_select_g<2, 32>(s, p, Q, Krepr, idx, cnt, st);
    }
    return bm == 16   ? launch_select_g<1, 16>(s, p, Q, Krepr, idx, cnt, st)
           : bm == 32 ? launch_select_g<1, 32>(s, p, Q, Krepr, idx, cnt, st)
                      : launch_select_g<1, 64>(s, p, Q, Krepr, idx, cnt, st);
}

}  // namespace phsa

extern "C" size_t phsa_test_set_select_tc_limit(size_t bytes) {
    const size_t v = bytes == 0 || bytes > phsa::kMaxDynSmem ? phsa::kMaxDynSmem : bytes;
    return phsa::g_select_tc_limit.exchange(v);
}
