// Stage (c) backward: gradients of the block-sparse causal attention with the
// block selection held fixed (the selection is a hard Top-K, so no gradient
// reaches the representative keys, lambda or the scores).
//
// Kernels, in launch order, all on the caller's stream:
//   delta      Delta_i = dO_i . O_i (fp32), half a warp per row.
//   idx_mark   sets bit qb of bitmap[(b,g,t)] for every selected (qb -> t)
//              (inside idx_build, in shared memory, when the bitmap fits).
//   idx_build  one CTA per (b,g): counts each KV block's selecting query
//              blocks, scans, writes the ascending query-block list of every
//              KV block (a CSR transpose of block_idx), and cuts lists longer
//              than kChunk into chunks (one work item each) so that the first
//              block, which every query block selects, does not serialise.
//   dkdv       one CTA per work item (KV block t, chunk): for every listed
//              query block and every query head of the group recomputes
//              S^T = K Q^T, P^T, dP^T = V dO^T, dS^T and accumulates
//              dV += P^T dO, dK += dS^T Q in registers. Single-chunk blocks
//              write bf16 directly; multi-chunk blocks write fp32 partials.
//   dkdv_sum   sums the partials of multi-chunk blocks in chunk order.
//   dq         one CTA per (query block, KV head): recomputes S, P, dP, dS
//              over the selected blocks and accumulates dQ += dS K.
// Every sum runs in a fixed order, so results are bit-reproducible.
#include <atomic>

#include "phsa_common.cuh"
#include "phsa_internal.h"
#include "union.cuh"

namespace phsa {

namespace {

constexpr int kChunk = kBwdChunk;  // query blocks per dK/dV work item
constexpr int kBuildCache = 8192;   // KV blocks whose counts the index build keeps on chip
// Largest bitmap of one (b, g) that the index build keeps in shared memory
// (beside its 32 KB of counts): 160 KB covers 1140 query blocks of 64 and
// 2048 query blocks of 16 (32k tokens at m = 16).
constexpr size_t kIdxSmemBits = 160u * 1024u;
// Which form of the transpose runs. 0, the default: one launch at m = 64 while
// the bitmap fits in kIdxSmemBits, two launches otherwise and at every m < 64,
// where marking the (64/m)-times longer lists is most of the work and the
// separate marking kernel spreads it over the whole GPU instead of one CTA per
// (b, g) (32k at m = 16: 23 + 146 us in one launch, 45 + 78 us in two; at
// m = 64: 31 us against 9 + 24). Nonzero: set by phsa_test_set_idx_smem_limit
// so that tests reach either form at any block size, one launch at every m
// while the bitmap fits in that many bytes.
std::atomic<size_t> g_idx_smem_override{0};

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

// ---------------------------------------------------------------- delta
__global__ void __launch_bounds__(256)
delta_kernel(const __nv_bfloat16* __restrict__ O, const __nv_bfloat16* __restrict__ dO,
             long long rows, float* __restrict__ delta) {
    const long long row = ((long long)blockIdx.x * 256 + threadIdx.x) >> 4;
    const int c = threadIdx.x & 15;
    float acc = 0.f;
    if (row < rows) {
        const uint4 a = __ldg(reinterpret_cast<const uint4*>(O + row * kD + c * 8));
        const uint4 d = __ldg(reinterpret_cast<const uint4*>(dO + row * kD + c * 8));
        const __nv_bfloat162* ha = reinterpret_cast<const __nv_bfloat162*>(&a);
        const __nv_bfloat162* hd = reinterpret_cast<const __nv_bfloat162*>(&d);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const float2 fa = __bfloat1622float2(ha[j]);
            const float2 fd = __bfloat1622float2(hd[j]);
            acc += fa.x * fd.x + fa.y * fd.y;
        }
    }
#pragma unroll
    for (int off = 8; off > 0; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
    if (row < rows && c == 0) delta[row] = acc;
}

// ---------------------------------------------------------------- index transpose
// Rows of the transposed selection are KV spans of 64 keys (kSub = 64/m blocks
// each; one block at m = 64), columns are query blocks of m tokens. At m < 64
// each (span, query block) pair also records which of the span's kSub blocks
// the query block selected: kSub bits in byte qb of the span's mask row. A
// query block's entries in one span are consecutive in its ascending list, so
// the byte is written once, by a plain store; bytes of pairs that are not
// selected are never read and need no clearing.
// Marks the selections of unit u (query block qb of one (b, g)) in the bitmap
// rows `bits` of that (b, g) (global or shared memory) and, at m < 64, in its
// mask rows. The entries are loaded eight at a time (independent loads), then
// checked in list order: -1 is skipped, an index that is negative, in the
// query's future or not ascending is recorded as a device index error.
__device__ __forceinline__ void mark_unit(const int32_t* __restrict__ idx,
                                          const int32_t* __restrict__ cnt, long long u, int qb,
                                          int kSub, int topk, int words, int mrow,
                                          uint32_t* bits, uint8_t* __restrict__ masks,
                                          int* status) {
    int n = cnt[u];
    if (n < 0 || n > topk) {
        set_status(status, PHSA_ERR_DEVICE_INDEX);
        n = n < 0 ? 0 : topk;
    }
    const int32_t* row = idx + u * topk;
    int prev = -1, curT = -1;
    uint32_t curm = 0u;  // the blocks of span curT this query block selected
    for (int j0 = 0; j0 < n; j0 += 8) {
        int tv[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) tv[k] = j0 + k < n ? __ldg(row + j0 + k) : -1;
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const int t = tv[k];
            if (t == -1) continue;
            if (t < 0 || t > qb || t <= prev) {
                set_status(status, PHSA_ERR_DEVICE_INDEX);
                continue;
            }
            prev = t;
            const int T = t / kSub;
            if (T != curT) {
                atomicOr(&bits[T * words + (qb >> 5)], 1u << (qb & 31));
                if (kSub > 1 && curT >= 0) masks[(size_t)curT * mrow + qb] = (uint8_t)curm;
                curT = T;
                curm = 0u;
            }
            curm |= 1u << (t - T * kSub);
        }
    }
    if (kSub > 1 && curT >= 0) masks[(size_t)curT * mrow + qb] = (uint8_t)curm;
}

__global__ void idx_mark_kernel(const int32_t* __restrict__ idx, const int32_t* __restrict__ cnt,
                                long long units, int NQB, int nrows, int kSub, int topk, int words,
                                int mrow, uint32_t* __restrict__ bits, uint8_t* __restrict__ masks,
                                int* status) {
    const long long u = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (u >= units) return;
    const int qb = (int)(u % NQB);
    const long long bg = u / NQB;
    mark_unit(idx, cnt, u, qb, kSub, topk, words, mrow, bits + bg * nrows * words,
              masks + bg * nrows * mrow, status);
}

// The bitmap of one (b, g) in shared memory, rows of rs words: thread q marks
// query block q's selections. The 32 query blocks of a warp share one bitmap
// column (word q / 32), so at each list position the lanes that selected the
// same KV span set their bits with one OR (the lanes of __match_any_sync are
// exactly those bits). The checks are mark_unit's, in list order per lane.
__device__ __forceinline__ void mark_warp(const int32_t* __restrict__ idx,
                                          const int32_t* __restrict__ cnt, long long u0, int NQB,
                                          int kSub, int topk, int rs, int mrow, uint32_t* bits,
                                          uint8_t* __restrict__ masks, int* status) {
    const int lane = threadIdx.x & 31;
    for (int qw = threadIdx.x & ~31; qw < NQB; qw += blockDim.x) {
        const int qb = qw + lane;
        const bool live = qb < NQB;
        int n = live ? cnt[u0 + qb] : 0;
        if (n < 0 || n > topk) {
            set_status(status, PHSA_ERR_DEVICE_INDEX);
            n = n < 0 ? 0 : topk;
        }
        const int nmax = __reduce_max_sync(0xffffffffu, n);
        const int32_t* row = idx + (u0 + (live ? qb : 0)) * topk;
        int prev = -1, curT = -1;
        uint32_t curm = 0u;  // the blocks of span curT this query block selected
        for (int j0 = 0; j0 < nmax; j0 += 8) {
            int tv[8];
#pragma unroll
            for (int k = 0; k < 8; ++k) tv[k] = j0 + k < n ? __ldg(row + j0 + k) : -1;
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                int t = tv[k];
                if (t != -1) {
                    if (t < 0 || t > qb || t <= prev) {
                        set_status(status, PHSA_ERR_DEVICE_INDEX);
                        t = -1;
                    } else {
                        prev = t;
                    }
                }
                // a span is marked once per query block: at its first entry in the list
                const int T = t < 0 ? -1 : t / kSub;
                const int Tn = T == curT ? -1 : T;
                const unsigned grp = __match_any_sync(0xffffffffu, Tn);
                if (Tn >= 0 && lane == __ffs(grp) - 1) atomicOr(&bits[Tn * rs + (qw >> 5)], grp);
                if (T >= 0) {
                    if (T != curT) {
                        if (kSub > 1 && curT >= 0) masks[(size_t)curT * mrow + qb] = (uint8_t)curm;
                        curT = T;
                        curm = 0u;
                    }
                    curm |= 1u << (t - T * kSub);
                }
            }
        }
        if (kSub > 1 && curT >= 0) masks[(size_t)curT * mrow + qb] = (uint8_t)curm;
    }
}

using TInfo = BwdTInfo;

// Block-wide exclusive scan of one int per thread (blockDim.x = 1024).
__device__ int block_excl_scan(int v, int* tmp, int& total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int x = v;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, off);
        if (lane >= off) x += y;
    }
    if (lane == 31) tmp[warp] = x;
    __syncthreads();
    if (warp == 0) {
        int w = tmp[lane];
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, w, off);
            if (lane >= off) w += y;
        }
        tmp[lane] = w;  // inclusive over warps
    }
    __syncthreads();
    const int before = (warp > 0 ? tmp[warp - 1] : 0) + x - v;
    total = tmp[31];
    __syncthreads();
    return before;
}

// One CTA per (b, g): the ascending query-block list of every row (KV span),
// cut into work items of at most kChunk iterations of kSub query blocks each.
// kMark: the CTA first builds its (b, g)'s bitmap in shared memory from the
// block lists itself (mark_warp), so that the transpose is
// one launch and the bitmap never goes through global memory; otherwise it
// reads the bitmap idx_mark_kernel left in `bits`.
template <bool kMark>
__global__ void __launch_bounds__(1024)
idx_build_kernel(const int32_t* __restrict__ idx, const int32_t* __restrict__ cnt,
                 const uint32_t* __restrict__ bits, int NQB, int nrows, int kSub, int topk,
                 int words, int mrow, uint8_t* __restrict__ masks, int work_max, int slot_max,
                 TInfo* __restrict__ tinfo, int32_t* __restrict__ qlist, int2* __restrict__ work,
                 int32_t* __restrict__ nwork, int* __restrict__ arrive, int2* __restrict__ queue,
                 int* __restrict__ qcount, int* status) {
    extern __shared__ uint32_t sbits[];  // kMark: the bitmap of this (b, g)
    __shared__ int tmp[32];
    __shared__ int bin[kChunk + 1];  // items per iteration count, then queue cursors
    __shared__ int ncache[kBuildCache];  // selecting-query count of each KV span
    const int bg = blockIdx.x;
    const int kChunkQ = kChunk * kSub;  // query blocks per work item
    const int per = (nrows + 1023) / 1024;  // KV spans counted by each thread
    const int t0 = threadIdx.x * per;
    const uint32_t* bb;
    int rs;  // words per bitmap row: odd in shared memory, so that rows fall in different banks
    if constexpr (kMark) {
        rs = words | 1;
        for (int i = threadIdx.x; i < nrows * rs; i += blockDim.x) sbits[i] = 0u;
        __syncthreads();
        mark_warp(idx, cnt, (long long)bg * NQB, NQB, kSub, topk, rs, mrow, sbits,
                  masks + (size_t)bg * nrows * mrow, status);
        __syncthreads();
        bb = sbits;
    } else {
        rs = words;
        bb = bits + (size_t)bg * nrows * words;
    }
    // The count of a block: its bitmap row's popcount, read with independent
    // loads. The first kBuildCache blocks keep theirs in shared memory for the
    // later passes (each thread reads back only its own entries); any block
    // beyond is counted again where it is needed.
    auto count_row = [&](int t) {
        const uint32_t* row = bb + (size_t)t * rs;
        int n = 0;
#pragma unroll 8
        for (int w = 0; w < words; ++w) n += __popc(row[w]);
        return n;
    };
    auto count_of = [&](int t) { return t < kBuildCache ? ncache[t] : count_row(t); };
    for (int k = 0; k < per; ++k) {
        const int t = t0 + k;
        if (t >= nrows) break;
        if (t < kBuildCache) ncache[t] = count_row(t);
    }
    int sn = 0, sch = 0, ssl = 0;
    for (int k = 0; k < per; ++k) {
        const int t = t0 + k;
        if (t >= nrows) break;
        const int n = count_of(t);
        const int nch = n <= kChunkQ ? 1 : (n + kChunkQ - 1) / kChunkQ;
        sn += n;
        sch += nch;
        ssl += nch > 1 ? nch : 0;
    }
    int tn, tch, tsl;
    int on = block_excl_scan(sn, tmp, tn);
    int och = block_excl_scan(sch, tmp, tch);
    int osl = block_excl_scan(ssl, tmp, tsl);
    if (threadIdx.x == 0) {
        nwork[bg] = min(tch, work_max);
        if (tch > work_max || tsl > slot_max || tn > NQB * topk) set_status(status, PHSA_ERR_DEVICE_INDEX);
    }
    for (int n = threadIdx.x; n <= kChunk; n += blockDim.x) bin[n] = 0;
    __syncthreads();
    // Items per iteration count (those that fit work_max), then one range of
    // each class's queue for this (b, g), sorted by iteration count, descending
    for (int k = 0, ch = och; k < per; ++k) {
        const int t = t0 + k;
        if (t >= nrows) break;
        const int n = count_of(t);
        const int nch = n <= kChunkQ ? 1 : (n + kChunkQ - 1) / kChunkQ;
        for (int c = 0; c < nch && ch + c < work_max; ++c)
            atomicAdd(&bin[(min(n, kChunkQ * c + kChunkQ) - kChunkQ * c + kSub - 1) / kSub], 1);
        ch += nch;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        int nc[kQueueClasses] = {};
        for (int n = 0; n <= kChunk; ++n) nc[queue_class(n)] += bin[n];
        int pos[kQueueClasses];
        for (int c = 0; c < kQueueClasses; ++c) pos[c] = atomicAdd(qcount + c, nc[c]);
        for (int n = kChunk; n >= 0; --n) {  // bin[n] becomes the cursor of its items
            const int c = queue_class(n), cnt_n = bin[n];
            bin[n] = pos[c];
            pos[c] += cnt_n;
        }
    }
    __syncthreads();
    const size_t qcap = (size_t)gridDim.x * work_max;
    TInfo* ti = tinfo + (size_t)bg * nrows;
    int2* wk = work + (size_t)bg * work_max;
    for (int k = 0; k < per; ++k) {
        const int t = t0 + k;
        if (t >= nrows) break;
        const int n = count_of(t);
        const int nch = n <= kChunkQ ? 1 : (n + kChunkQ - 1) / kChunkQ;
        TInfo info;
        info.off = on;
        info.n = n;
        info.nch = nch;
        info.slot = (nch > 1 && osl + nch <= slot_max) ? osl : -1;
        ti[t] = info;
        if (t < kBuildCache) ncache[t] = on;  // from here on: the list's offset
        arrive[(size_t)bg * nrows + t] = 0;
        for (int c = 0; c < nch && och + c < work_max; ++c) {
            wk[och + c] = make_int2(t, c);
            const int n_it = (min(n, kChunkQ * c + kChunkQ) - kChunkQ * c + kSub - 1) / kSub;
            queue[queue_class(n_it) * qcap + atomicAdd(&bin[n_it], 1)] = make_int2(bg * nrows + t, c);
        }
        on += n;
        och += nch;
        osl += nch > 1 ? nch : 0;
    }
    __syncthreads();  // tinfo of every block is written and visible to the whole CTA
    // List of each KV block: one warp per block, 32 bitmap words per round; a
    // warp scan of the words' popcounts gives every lane its output position.
    // Each warp takes 8 blocks at a time and issues all their loads first.
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int32_t* ql = qlist + (size_t)bg * NQB * topk;
    const int cap = NQB * topk;
    constexpr int kBatch = 8;
    for (int tb = warp; tb < nrows; tb += 32 * kBatch) {
        int pos[kBatch];
#pragma unroll
        for (int j = 0; j < kBatch; ++j) {
            const int t = tb + 32 * j;
            pos[j] = t >= nrows ? 0 : t < kBuildCache ? ncache[t] : ti[t].off;
        }
        for (int w0 = 0; w0 < words; w0 += 32) {
            const int w = w0 + lane;
            uint32_t m[kBatch];
#pragma unroll
            for (int j = 0; j < kBatch; ++j) {
                const int t = tb + 32 * j;
                m[j] = (t < nrows && w < words) ? bb[(size_t)t * rs + w] : 0u;
            }
#pragma unroll
            for (int j = 0; j < kBatch; ++j) {
                const int c = __popc(m[j]);
                int x = c;
#pragma unroll
                for (int off = 1; off < 32; off <<= 1) {
                    const int y = __shfl_up_sync(0xffffffffu, x, off);
                    if (lane >= off) x += y;
                }
                int o = pos[j] + x - c;
                uint32_t mm = m[j];
                while (mm) {
                    const int q = w * 32 + __ffs(mm) - 1;
                    mm &= mm - 1;
                    if (o < cap) ql[o] = q;
                    ++o;
                }
                pos[j] += __shfl_sync(0xffffffffu, x, 31);
            }
        }
    }
}

// ---------------------------------------------------------------- dK / dV
constexpr int kKvThreads = 128;  // 4 warps, 16 keys each
constexpr int kTile = kM * kD * 2;
// smem: K, V (2 tiles) | 2 stages x (Q, dO) | 2 stages x (lse2, delta) [64 floats each]
constexpr int kKvStageOff = 2 * kTile;
constexpr int kKvVecOff = kKvStageOff + 4 * kTile;
constexpr int kKvSmem = kKvVecOff + 2 * 2 * 64 * 4;

__global__ void __launch_bounds__(kKvThreads)
dkdv_kernel(const __nv_bfloat16* __restrict__ Q, const __nv_bfloat16* __restrict__ K,
            const __nv_bfloat16* __restrict__ V, const __nv_bfloat16* __restrict__ dO,
            const float* __restrict__ lse, const float* __restrict__ delta,
            const TInfo* __restrict__ tinfo, const int32_t* __restrict__ qlist,
            const int2* __restrict__ work, const int32_t* __restrict__ nwork, int Hq, int Hkv,
            int L, int NQB, int topk, int work_max, int slot_max, float scale_log2,
            float sm_scale, __nv_bfloat16* __restrict__ dK, __nv_bfloat16* __restrict__ dV,
            float* __restrict__ partial) {
    extern __shared__ __align__(128) uint8_t smem[];
    const int bg = blockIdx.y;
    if ((int)blockIdx.x >= nwork[bg]) return;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int G = Hq / Hkv;
    const int b = bg / Hkv, g = bg % Hkv;
    const int2 wi = work[(size_t)bg * work_max + blockIdx.x];
    const int t = wi.x, chunk = wi.y;
    const TInfo info = tinfo[(size_t)bg * NQB + t];
    const int q_begin = chunk * kChunk;
    const int q_end = min(info.n, q_begin + kChunk);
    const int n_iter = max(0, q_end - q_begin) * G;
    const int32_t* ql = qlist + (size_t)bg * NQB * topk + info.off;

    const uint32_t sK = smem_u32(smem), sV = sK + kTile;
    const uint32_t sStage = sK + kKvStageOff;
    float* vecs = reinterpret_cast<float*>(smem + kKvVecOff);

    const __nv_bfloat16* Kg = K + (size_t)bg * L * kD;
    const __nv_bfloat16* Vg = V + (size_t)bg * L * kD;
    load_tile64<kKvThreads>(sK, Kg, t * kM, L, tid);
    load_tile64<kKvThreads>(sV, Vg, t * kM, L, tid);

    // iteration j -> (query block ql[q_begin + j / G], head g*G + j % G)
    auto issue = [&](int j, int stage) {
        const int qb = ql[q_begin + j / G];
        const int h = g * G + j % G;
        const size_t hoff = (size_t)(b * Hq + h) * L;
        const uint32_t st = sStage + stage * 2 * kTile;
        load_tile64<kKvThreads>(st, Q + hoff * kD, qb * kM, L, tid);
        load_tile64<kKvThreads>(st + kTile, dO + hoff * kD, qb * kM, L, tid);
        if (tid < 64) {
            const int i = qb * kM + tid;
            float* v = vecs + stage * 128;
            v[tid] = i < L ? lse[hoff + i] * kLog2e : 0.f;
            v[64 + tid] = i < L ? delta[hoff + i] : 0.f;
        }
    };
    if (n_iter > 0) issue(0, 0);
    cp_async_commit();

    float dk[16][4], dv[16][4];
#pragma unroll
    for (int n = 0; n < 16; ++n)
#pragma unroll
        for (int e = 0; e < 4; ++e) { dk[n][e] = 0.f; dv[n][e] = 0.f; }

    const int key0 = warp * 16 + (lane >> 2);  // this lane's keys: key0, key0 + 8
    for (int it = 0; it < n_iter; ++it) {
        if (it + 1 < n_iter) {
            issue(it + 1, (it + 1) & 1);
            cp_async_commit();
            cp_async_wait<1>();
        } else {
            cp_async_wait<0>();
        }
        __syncthreads();
        const int qb = ql[q_begin + it / G];
        const uint32_t sQ = sStage + (it & 1) * 2 * kTile;
        const uint32_t sdO = sQ + kTile;
        const float* lse2 = vecs + (it & 1) * 128;
        const float* dl = lse2 + 64;
        const bool diag = (qb == t);
#pragma unroll
        for (int hq = 0; hq < 2; ++hq) {  // two halves of 32 queries
            float sT[4][4], dpT[4][4];
#pragma unroll
            for (int n = 0; n < 4; ++n)
#pragma unroll
                for (int e = 0; e < 4; ++e) { sT[n][e] = 0.f; dpT[n][e] = 0.f; }
#pragma unroll
            for (int kc = 0; kc < 8; ++kc) {
                uint32_t ka[4], va[4];
                load_a_frag(sK, warp * 16, kc, lane, ka);
                load_a_frag(sV, warp * 16, kc, lane, va);
#pragma unroll
                for (int np = 0; np < 2; ++np) {
                    uint32_t qb4[4], ob4[4];
                    load_b_nk(sQ, hq * 32 + np * 16, kc, lane, qb4);
                    load_b_nk(sdO, hq * 32 + np * 16, kc, lane, ob4);
                    mma16816(sT[2 * np], ka, qb4[0], qb4[1]);
                    mma16816(sT[2 * np + 1], ka, qb4[2], qb4[3]);
                    mma16816(dpT[2 * np], va, ob4[0], ob4[1]);
                    mma16816(dpT[2 * np + 1], va, ob4[2], ob4[3]);
                }
            }
            // P^T and dS^T (rows: keys, columns: queries)
#pragma unroll
            for (int n = 0; n < 4; ++n)
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int key = key0 + ((e >> 1) << 3);
                    const int q = hq * 32 + n * 8 + (lane & 3) * 2 + (e & 1);
                    const bool ok = (qb * kM + q < L) && !(diag && key > q);
                    const float p = ok ? exp2f(sT[n][e] * scale_log2 - lse2[q]) : 0.f;
                    sT[n][e] = p;
                    dpT[n][e] = p * (dpT[n][e] - dl[q]);
                }
            // dV += P^T dO, dK += dS^T Q (k = the 32 queries of this half)
#pragma unroll
            for (int ks = 0; ks < 2; ++ks) {
                uint32_t pa[4], sa[4];
                pa[0] = pack_bf16(sT[2 * ks][0], sT[2 * ks][1]);
                pa[1] = pack_bf16(sT[2 * ks][2], sT[2 * ks][3]);
                pa[2] = pack_bf16(sT[2 * ks + 1][0], sT[2 * ks + 1][1]);
                pa[3] = pack_bf16(sT[2 * ks + 1][2], sT[2 * ks + 1][3]);
                sa[0] = pack_bf16(dpT[2 * ks][0], dpT[2 * ks][1]);
                sa[1] = pack_bf16(dpT[2 * ks][2], dpT[2 * ks][3]);
                sa[2] = pack_bf16(dpT[2 * ks + 1][0], dpT[2 * ks + 1][1]);
                sa[3] = pack_bf16(dpT[2 * ks + 1][2], dpT[2 * ks + 1][3]);
#pragma unroll
                for (int np = 0; np < 8; ++np) {
                    uint32_t ob[4], qb2[4];
                    load_b_kn(sdO, hq * 32 + ks * 16, np * 2, lane, ob);
                    load_b_kn(sQ, hq * 32 + ks * 16, np * 2, lane, qb2);
                    mma16816(dv[2 * np], pa, ob[0], ob[1]);
                    mma16816(dv[2 * np + 1], pa, ob[2], ob[3]);
                    mma16816(dk[2 * np], sa, qb2[0], qb2[1]);
                    mma16816(dk[2 * np + 1], sa, qb2[2], qb2[3]);
                }
            }
        }
        __syncthreads();
    }
    cp_async_wait<0>();
    __syncthreads();

    if (info.nch > 1) {
        if (info.slot < 0) return;  // workspace bound exceeded (status already set)
        float* pk = partial + ((size_t)bg * slot_max + info.slot + chunk) * 2 * kM * kD;
        float* pv = pk + kM * kD;
#pragma unroll
        for (int n = 0; n < 16; ++n)
#pragma unroll
            for (int hh = 0; hh < 2; ++hh) {
                const int r = key0 + hh * 8;
                const int c = n * 8 + (lane & 3) * 2;
                *reinterpret_cast<float2*>(pk + r * kD + c) =
                    make_float2(dk[n][2 * hh] * sm_scale, dk[n][2 * hh + 1] * sm_scale);
                *reinterpret_cast<float2*>(pv + r * kD + c) = make_float2(dv[n][2 * hh], dv[n][2 * hh + 1]);
            }
        return;
    }
    // bf16 output through shared memory (K tile <- dK, V tile <- dV)
#pragma unroll
    for (int n = 0; n < 16; ++n)
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
            const int r = key0 + hh * 8;
            const int c = n * 8 + (lane & 3) * 2;
            const uint32_t off = swz(r, c >> 3) + (c & 7) * 2;
            *reinterpret_cast<uint32_t*>(smem + off) =
                pack_bf16(dk[n][2 * hh] * sm_scale, dk[n][2 * hh + 1] * sm_scale);
            *reinterpret_cast<uint32_t*>(smem + kTile + off) = pack_bf16(dv[n][2 * hh], dv[n][2 * hh + 1]);
        }
    __syncthreads();
    __nv_bfloat16* dKg = dK + (size_t)bg * L * kD;
    __nv_bfloat16* dVg = dV + (size_t)bg * L * kD;
    for (int e = tid; e < kM * kRowChunks; e += kKvThreads) {
        const int r = e >> 4, c = e & 15;
        const int i = t * kM + r;
        if (i < L) {
            *reinterpret_cast<uint4*>(dKg + (size_t)i * kD + c * 8) =
                *reinterpret_cast<const uint4*>(smem + swz(r, c));
            *reinterpret_cast<uint4*>(dVg + (size_t)i * kD + c * 8) =
                *reinterpret_cast<const uint4*>(smem + kTile + swz(r, c));
        }
    }
}

__global__ void __launch_bounds__(256)
dkdv_sum_kernel(const TInfo* __restrict__ tinfo, const float* __restrict__ partial, int Hkv,
                int L, int NQB, int slot_max, __nv_bfloat16* __restrict__ dK,
                __nv_bfloat16* __restrict__ dV) {
    const int t = blockIdx.x, bg = blockIdx.y;
    const TInfo info = tinfo[(size_t)bg * NQB + t];
    if (info.nch <= 1 || info.slot < 0) return;
    const float* base = partial + ((size_t)bg * slot_max + info.slot) * 2 * kM * kD;
    for (int e = threadIdx.x * 4; e < 2 * kM * kD; e += 256 * 4) {
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int c = 0; c < info.nch; ++c) {
            const float4 v = *reinterpret_cast<const float4*>(base + (size_t)c * 2 * kM * kD + e);
            acc.x += v.x; acc.y += v.y; acc.z += v.z; acc.w += v.w;
        }
        const int which = e / (kM * kD);
        const int r = (e % (kM * kD)) / kD, col = e % kD;
        const int i = t * kM + r;
        if (i < L) {
            __nv_bfloat16* dst = (which == 0 ? dK : dV) + ((size_t)bg * L + i) * kD + col;
            uint2 pk;
            pk.x = pack_bf16(acc.x, acc.y);
            pk.y = pack_bf16(acc.z, acc.w);
            *reinterpret_cast<uint2*>(dst) = pk;
        }
    }
}

// ---------------------------------------------------------------- dQ
template <int G>
struct DqCfg {
    static constexpr int kWarps = 4 * G;
    static constexpr int kThreads = 32 * kWarps;
    static constexpr int kRows = 64 * G;
    static constexpr int kQOff = 0;
    static constexpr int kdOOff = G * kTile;
    static constexpr int kKVOff = 2 * G * kTile;        // 2 stages x (K, V)
    static constexpr int kVecOff = kKVOff + 4 * kTile;  // lse2[kRows], delta[kRows]
    static constexpr int kListOff = kVecOff + 2 * kRows * 4;
    static size_t smem_bytes(int topk) { return (size_t)kListOff + (size_t)(topk + 1) * 4; }
};

template <int G>
__global__ void __launch_bounds__(DqCfg<G>::kThreads)
dq_kernel(const __nv_bfloat16* __restrict__ Q, const __nv_bfloat16* __restrict__ K,
          const __nv_bfloat16* __restrict__ V, const __nv_bfloat16* __restrict__ dO,
          const float* __restrict__ lse, const float* __restrict__ delta,
          const int32_t* __restrict__ idx, const int32_t* __restrict__ cnt, int Hq, int Hkv,
          int L, int NQB, int topk, float scale_log2, float sm_scale,
          __nv_bfloat16* __restrict__ dQ, int* status) {
    using C = DqCfg<G>;
    extern __shared__ __align__(128) uint8_t smem[];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int unit = blockIdx.x;
    const int qb = NQB - 1 - (unit % NQB);
    const int bg = unit / NQB;
    const int b = bg / Hkv, g = bg % Hkv;
    const long long lu = (long long)bg * NQB + qb;

    const uint32_t sQ = smem_u32(smem) + C::kQOff;
    const uint32_t sdO = smem_u32(smem) + C::kdOOff;
    const uint32_t sKV = smem_u32(smem) + C::kKVOff;
    float* lse2 = reinterpret_cast<float*>(smem + C::kVecOff);
    float* dl = lse2 + C::kRows;
    int* blist = reinterpret_cast<int*>(smem + C::kListOff);
    if (tid == 0) blist[topk] = compact_block_list(idx + lu * topk, cnt[lu], topk, qb, blist, nullptr);

    const __nv_bfloat16* Kg = K + (size_t)bg * L * kD;
    const __nv_bfloat16* Vg = V + (size_t)bg * L * kD;
#pragma unroll
    for (int hl = 0; hl < G; ++hl) {
        const size_t hoff = (size_t)(b * Hq + g * G + hl) * L;
        load_tile64<C::kThreads>(sQ + hl * kTile, Q + hoff * kD, qb * kM, L, tid);
        load_tile64<C::kThreads>(sdO + hl * kTile, dO + hoff * kD, qb * kM, L, tid);
    }
    for (int r = tid; r < C::kRows; r += C::kThreads) {
        const int i = qb * kM + (r & 63);
        const size_t hoff = (size_t)(b * Hq + g * G + (r >> 6)) * L;
        lse2[r] = i < L ? lse[hoff + i] * kLog2e : 0.f;
        dl[r] = i < L ? delta[hoff + i] : 0.f;
    }
    cp_async_commit();
    __syncthreads();
    const int nblk = blist[topk];
    if (nblk > 0) {
        load_tile64<C::kThreads>(sKV, Kg, blist[0] * kM, L, tid);
        load_tile64<C::kThreads>(sKV + kTile, Vg, blist[0] * kM, L, tid);
    }
    cp_async_commit();

    const int rq0 = (warp & 3) * 16 + (lane >> 2);
    const int rw0 = warp * 16 + (lane >> 2);  // row in the stacked G*64 tile
    uint32_t qf[8][4];
    float dq[16][4];
#pragma unroll
    for (int n = 0; n < 16; ++n)
#pragma unroll
        for (int e = 0; e < 4; ++e) dq[n][e] = 0.f;

    for (int it = 0; it < nblk; ++it) {
        if (it + 1 < nblk) {
            const uint32_t st = sKV + ((it + 1) & 1) * 2 * kTile;
            load_tile64<C::kThreads>(st, Kg, blist[it + 1] * kM, L, tid);
            load_tile64<C::kThreads>(st + kTile, Vg, blist[it + 1] * kM, L, tid);
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
        const uint32_t sK = sKV + (it & 1) * 2 * kTile;
        const uint32_t sV = sK + kTile;
        const bool diag = (blist[it] == qb);
        float s[8][4], dp[8][4];
#pragma unroll
        for (int n = 0; n < 8; ++n)
#pragma unroll
            for (int e = 0; e < 4; ++e) { s[n][e] = 0.f; dp[n][e] = 0.f; }
#pragma unroll
        for (int kc = 0; kc < 8; ++kc) {
            uint32_t oa[4];
            load_a_frag(sdO, warp * 16, kc, lane, oa);
#pragma unroll
            for (int np = 0; np < 4; ++np) {
                uint32_t kb[4], vb[4];
                load_b_nk(sK, np * 16, kc, lane, kb);
                load_b_nk(sV, np * 16, kc, lane, vb);
                mma16816(s[2 * np], qf[kc], kb[0], kb[1]);
                mma16816(s[2 * np + 1], qf[kc], kb[2], kb[3]);
                mma16816(dp[2 * np], oa, vb[0], vb[1]);
                mma16816(dp[2 * np + 1], oa, vb[2], vb[3]);
            }
        }
#pragma unroll
        for (int n = 0; n < 8; ++n)
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int key = n * 8 + (lane & 3) * 2 + (e & 1);
                const int hh = e >> 1;
                const int row = rq0 + hh * 8;
                const int rw = rw0 + hh * 8;
                const bool ok = (qb * kM + row < L) && !(diag && key > row);
                const float p = ok ? exp2f(s[n][e] * scale_log2 - lse2[rw]) : 0.f;
                s[n][e] = p * (dp[n][e] - dl[rw]);  // dS
            }
#pragma unroll
        for (int ks = 0; ks < 4; ++ks) {
            uint32_t sa[4];
            sa[0] = pack_bf16(s[2 * ks][0], s[2 * ks][1]);
            sa[1] = pack_bf16(s[2 * ks][2], s[2 * ks][3]);
            sa[2] = pack_bf16(s[2 * ks + 1][0], s[2 * ks + 1][1]);
            sa[3] = pack_bf16(s[2 * ks + 1][2], s[2 * ks + 1][3]);
#pragma unroll
            for (int np = 0; np < 8; ++np) {
                uint32_t kb[4];
                load_b_kn(sK, ks * 16, np * 2, lane, kb);
                mma16816(dq[2 * np], sa, kb[0], kb[1]);
                mma16816(dq[2 * np + 1], sa, kb[2], kb[3]);
            }
        }
        __syncthreads();
    }
    cp_async_wait<0>();
    __syncthreads();

    const int h = g * G + (warp >> 2);
#pragma unroll
    for (int n = 0; n < 16; ++n)
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
            const int r = rw0 + hh * 8;
            const int c = n * 8 + (lane & 3) * 2;
            *reinterpret_cast<uint32_t*>(smem + C::kQOff + swz(r, c >> 3) + (c & 7) * 2) =
                pack_bf16(dq[n][2 * hh] * sm_scale, dq[n][2 * hh + 1] * sm_scale);
        }
    __syncwarp();
    __nv_bfloat16* dQh = dQ + (size_t)(b * Hq + h) * L * kD;
#pragma unroll
    for (int k = 0; k < 8; ++k) {
        const int e = k * 32 + lane;
        const int r = e >> 4, c = e & 15;
        const int i = qb * kM + (warp & 3) * 16 + r;
        if (i < L)
            *reinterpret_cast<uint4*>(dQh + (size_t)i * kD + c * 8) =
                *reinterpret_cast<const uint4*>(smem + C::kQOff + swz(warp * 16 + r, c));
    }
}

template <int G>
cudaError_t launch_dq_g(const void* Q, const void* K, const void* V, const void* dO,
                        const float* lse, const float* delta, const int32_t* idx,
                        const int32_t* cnt, const phsa_shape& s, int topk, float sm_scale,
                        void* dQ, int* status, cudaStream_t st) {
    const int NQB = (s.L + kM - 1) / kM;
    const size_t smem = DqCfg<G>::smem_bytes(topk);
    auto kern = dq_kernel<G>;
    cudaError_t e =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    ProfScope prof(K_BWD_DQ, st);
    kern<<<(unsigned)((long long)s.B * s.Hkv * NQB), DqCfg<G>::kThreads, smem, st>>>(
        static_cast<const __nv_bfloat16*>(Q), static_cast<const __nv_bfloat16*>(K),
        static_cast<const __nv_bfloat16*>(V), static_cast<const __nv_bfloat16*>(dO), lse, delta,
        idx, cnt, s.Hq, s.Hkv, s.L, NQB, topk, sm_scale * kLog2e, sm_scale,
        static_cast<__nv_bfloat16*>(dQ), status);
    return cudaGetLastError();
}

}  // namespace

BwdLayout bwd_layout(const phsa_shape& s, int topk) {
    BwdLayout l{};
    const int bm = s.block_size;
    l.kSub = kM / bm;
    l.nqb = (s.L + bm - 1) / bm;
    l.nrows = (s.L + kM - 1) / kM;
    l.words = (l.nqb + 31) / 32;
    l.mrow = l.kSub > 1 ? l.nqb : 0;  // mask bytes per span row
    l.chunk = kChunk * l.kSub;  // query blocks per dK/dV work item
    l.ucap = l.kSub * topk;
    const long long bgs = (long long)s.B * s.Hkv;
    const long long nnz_max = (long long)l.nqb * topk;  // per (b, g)
    l.work_max = (int)(l.nrows + (nnz_max + l.chunk - 1) / l.chunk);
    l.slot_max = (int)((2 * nnz_max + l.chunk - 1) / l.chunk);
    const long long spans = bgs * l.nrows;
    size_t off = 0;
    l.qctl = off;    off = align256(off + 8 * 4);
    l.bits = off;    off = align256(off + (size_t)spans * l.words * 4);
    l.masks = off;   off = align256(off + (size_t)spans * l.mrow);
    l.tinfo = off;   off = align256(off + (size_t)spans * sizeof(TInfo));
    l.qlist = off;   off = align256(off + (size_t)bgs * nnz_max * 4);
    l.work = off;    off = align256(off + (size_t)bgs * l.work_max * sizeof(int2));
    l.nwork = off;   off = align256(off + (size_t)bgs * 4);
    l.queue = off;   off = align256(off + (size_t)kQueueClasses * bgs * l.work_max * sizeof(int2));
    l.delta = off;   off = align256(off + (size_t)s.B * s.Hq * s.L * 4);
    l.partial = off; off = align256(off + (size_t)bgs * l.slot_max * 2 * kM * kD * 4);
    l.arrive = off;  off = align256(off + (size_t)spans * 4);
    l.ucnt = off;    off = align256(off + (l.kSub > 1 ? (size_t)spans * 4 : 0));
    l.ulist = off;   off = align256(off + (l.kSub > 1 ? (size_t)spans * l.ucap * 4 : 0));
    l.umask = off;   off = align256(off + (l.kSub > 1 ? (size_t)spans * l.ucap : 0));
    l.total = off;
    return l;
}

// The union of the block lists of every span's query blocks (block size
// m < 64), with owner masks, for the dQ pass: one warp per (b, g, span).
template <int kSub>
__global__ void __launch_bounds__(128)
span_union_kernel(const int32_t* __restrict__ idx, const int32_t* __restrict__ cnt, int NQB,
                  int nrows, long long spans, int topk, int ucap, int32_t* __restrict__ ucnt,
                  int32_t* __restrict__ ulist, uint8_t* __restrict__ umask, int* status) {
    extern __shared__ uint32_t ubm[];  // per warp: kSub bitmaps of W words
    const int W = (NQB + 31) / 32;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    uint32_t* bm = ubm + (size_t)warp * kSub * W;
    for (int i = lane; i < kSub * W; i += 32) bm[i] = 0u;
    __syncwarp();
    const long long u = (long long)blockIdx.x * 4 + warp;
    if (u >= spans) return;
    const long long bg = u / nrows;
    const int sp = (int)(u - bg * nrows);
    const int qb0 = sp * kSub;
    build_block_union<kSub>(idx, cnt, bg * NQB + qb0, qb0, min(kSub, NQB - qb0), topk, bm, W,
                            ulist + u * ucap, umask + u * ucap, ucnt + u, status, lane);
}

cudaError_t launch_attn_bwd(const void* Q, const void* K, const void* V, const void* O,
                            const void* dO, const float* lse, const int32_t* idx,
                            const int32_t* cnt, const phsa_shape& s, int topk, float sm_scale,
                            void* ws, void* dQ, void* dK, void* dV, int* status,
                            cudaStream_t st, cudaEvent_t after_dq) {
    if ((long long)s.B * s.Hkv * s.L == 0)
        return after_dq ? cudaEventRecord(after_dq, st) : cudaSuccess;
    const BwdLayout l = bwd_layout(s, topk);
    uint8_t* w = static_cast<uint8_t*>(ws);
    uint32_t* bits = reinterpret_cast<uint32_t*>(w + l.bits);
    uint8_t* masks = w + l.masks;
    int32_t* ucnt = reinterpret_cast<int32_t*>(w + l.ucnt);
    int32_t* ulist = reinterpret_cast<int32_t*>(w + l.ulist);
    uint8_t* umask = reinterpret_cast<uint8_t*>(w + l.umask);
    TInfo* tinfo = reinterpret_cast<TInfo*>(w + l.tinfo);
    int32_t* qlist = reinterpret_cast<int32_t*>(w + l.qlist);
    int2* work = reinterpret_cast<int2*>(w + l.work);
    int32_t* nwork = reinterpret_cast<int32_t*>(w + l.nwork);
    float* delta = reinterpret_cast<float*>(w + l.delta);
    float* partial = reinterpret_cast<float*>(w + l.partial);
    int* arrive = reinterpret_cast<int*>(w + l.arrive);
    int2* queue = reinterpret_cast<int2*>(w + l.queue);
    int* qctl = reinterpret_cast<int*>(w + l.qctl);
    const int bgs = s.B * s.Hkv;
    const long long rows = (long long)s.B * s.Hq * s.L;
    cudaError_t e;

    // Two query heads per KV head: tcgen05 kernels (M = 128 rows per MMA), as
    // long as the block list fits beside dq_tc_kernel's tiles. Block sizes
    // 16 and 32 run on them only (the API rejects them otherwise).
    const bool pair = s.Hq / s.Hkv == 2 && dq_tc_fits(topk, s.block_size);
    if (l.kSub > 1 && !pair) return cudaErrorInvalidValue;
    if (l.kSub > 1) {  // the span unions the dQ pass reads
        const long long spans = (long long)bgs * l.nrows;
        const size_t ush = (size_t)4 * l.kSub * l.words * 4;
        ProfScope prof(K_BWD_MARK, st);
        if (l.kSub == 2)
            span_union_kernel<2><<<(unsigned)((spans + 3) / 4), 128, ush, st>>>(
                idx, cnt, l.nqb, l.nrows, spans, topk, l.ucap, ucnt, ulist, umask, status);
        else
            span_union_kernel<4><<<(unsigned)((spans + 3) / 4), 128, ush, st>>>(
                idx, cnt, l.nqb, l.nrows, spans, topk, l.ucap, ucnt, ulist, umask, status);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    if (pair) {
        // dQ first: it also computes Delta from O and dO, which dK/dV then read.
        e = launch_dq_tc(Q, K, V, O, dO, lse, delta, idx, cnt, ulist, ucnt, umask, s, topk,
                         sm_scale, dQ, status, st);
        if (e != cudaSuccess) return e;
        if (after_dq && (e = cudaEventRecord(after_dq, st)) != cudaSuccess) return e;
    } else {
        ProfScope prof(K_BWD_DELTA, st);
        delta_kernel<<<(unsigned)((rows * 16 + 255) / 256), 256, 0, st>>>(
            static_cast<const __nv_bfloat16*>(O), static_cast<const __nv_bfloat16*>(dO), rows,
            delta);
    }
    if ((e = cudaGetLastError()) != cudaSuccess) return e;

    // the queue counters and the bitmap, in one memset (the mask rows need none)
    if ((e = cudaMemsetAsync(w + l.qctl, 0, l.masks - l.qctl, st)) != cudaSuccess) return e;
    const long long units = (long long)bgs * l.nqb;
    const size_t sbits = (size_t)l.nrows * (l.words | 1) * 4;  // one (b, g)'s bitmap
    const size_t ov = g_idx_smem_override.load();
    if (ov ? sbits <= ov : l.kSub == 1 && sbits <= kIdxSmemBits) {
        // mark and build in one launch, the bitmap in shared memory
        auto kern = idx_build_kernel<true>;
        if ((e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      (int)sbits)) != cudaSuccess)
            return e;
        ProfScope prof(K_BWD_BUILD, st);
        kern<<<bgs, 1024, sbits, st>>>(idx, cnt, bits, l.nqb, l.nrows, l.kSub, topk, l.words,
                                       l.mrow, masks, l.work_max, l.slot_max, tinfo, qlist, work,
                                       nwork, arrive, queue, qctl, status);
    } else {
        {
            ProfScope prof(K_BWD_MARK, st);
            idx_mark_kernel<<<(unsigned)((units + 255) / 256), 256, 0, st>>>(
                idx, cnt, units, l.nqb, l.nrows, l.kSub, topk, l.words, l.mrow, bits, masks,
                status);
        }
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
        ProfScope prof(K_BWD_BUILD, st);
        idx_build_kernel<false><<<bgs, 1024, 0, st>>>(
            idx, cnt, bits, l.nqb, l.nrows, l.kSub, topk, l.words, l.mrow, masks, l.work_max,
            l.slot_max, tinfo, qlist, work, nwork, arrive, queue, qctl, status);
    }
    if ((e = cudaGetLastError()) != cudaSuccess) return e;

    if (pair)  // sums multi-chunk partials itself
        return launch_dkdv_tc(Q, K, V, dO, lse, delta, tinfo, qlist, masks, queue, qctl, s, topk,
                              l, sm_scale, dK, dV, partial, arrive, status, st);

    e = cudaFuncSetAttribute(dkdv_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kKvSmem);
    if (e != cudaSuccess) return e;
    {
        ProfScope prof(K_BWD_DKDV, st);
        dkdv_kernel<<<dim3(l.work_max, bgs), kKvThreads, kKvSmem, st>>>(
            static_cast<const __nv_bfloat16*>(Q), static_cast<const __nv_bfloat16*>(K),
            static_cast<const __nv_bfloat16*>(V), static_cast<const __nv_bfloat16*>(dO), lse,
            delta, tinfo, qlist, work, nwork, s.Hq, s.Hkv, s.L, l.nqb, topk, l.work_max,
            l.slot_max, sm_scale * kLog2e, sm_scale, static_cast<__nv_bfloat16*>(dK),
            static_cast<__nv_bfloat16*>(dV), partial);
    }
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    {
        ProfScope prof(K_BWD_DKDV_SUM, st);
        dkdv_sum_kernel<<<dim3(l.nqb, bgs), 256, 0, st>>>(
            tinfo, partial, s.Hkv, s.L, l.nqb, l.slot_max, static_cast<__nv_bfloat16*>(dK),
            static_cast<__nv_bfloat16*>(dV));
    }
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    e = s.Hq == s.Hkv
            ? launch_dq_g<1>(Q, K, V, dO, lse, delta, idx, cnt, s, topk, sm_scale, dQ, status, st)
            : launch_dq_g<2>(Q, K, V, dO, lse, delta, idx, cnt, s, topk, sm_scale, dQ, status, st);
    if (e != cudaSuccess) return e;
    return after_dq ? cudaEventRecord(after_dq, st) : cudaSuccess;
}

}  // namespace phsa

extern "C" size_t phsa_test_set_idx_smem_limit(size_t bytes) {
    const size_t v = bytes > phsa::kIdxSmemBits ? phsa::kIdxSmemBits : bytes;
    return phsa::g_idx_smem_override.exchange(v);
}
