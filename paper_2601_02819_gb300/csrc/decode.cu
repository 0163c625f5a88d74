// Decode: one new token per sequence. The newest token of sequence b (position
// p = len_b - 1) is the query; the selection rule of Section 3.3 (Algorithm 1
// step 3) is applied to the unit whose rows are that token in each of the
// GQA group's G query heads, and Eq. 10-11 to the token's row. The block
// representations are cached and updated as blocks fill (block_repr.cu).
//
// Both kernels read little per unit and are bound by HBM bandwidth, so they
// run on the CUDA cores: one CTA (8 warps) per (sequence, KV head), with a
// half-warp per 256-byte key row (lane c holds columns 8c..8c+7, 16-byte
// read-only loads, four rows in flight per half-warp).
//
// decode_select_kernel  S[h][t] = q_h . Krepr_t for the candidates, per head
//   the softmax over candidates (max, sum), A_t = sum over heads of the
//   probabilities (head order), then the top-k of topk.cuh.
// decode_attn_kernel  each half-warp runs an online softmax over a share of
//   the selected keys (4 keys per step); the 16 partial states are merged in
//   shared memory. Keys after p (the unfilled part of the local block) are
//   masked.
#include "phsa_common.cuh"
#include "phsa_internal.h"
#include "topk.cuh"

namespace phsa {

namespace {

constexpr int kThreads = 256;

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

__device__ __forceinline__ void load_q8(const __nv_bfloat16* q, float scale, float* out) {
    const uint4 v = __ldg(reinterpret_cast<const uint4*>(q));
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const float2 f = __bfloat1622float2(h[j]);
        out[2 * j] = f.x * scale;
        out[2 * j + 1] = f.y * scale;
    }
}

// Block-wide reduction of one float per thread (max or sum) over 256 threads.
template <bool kMax>
__device__ __forceinline__ float block_reduce(float v, float* red) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
        const float o = __shfl_xor_sync(0xffffffffu, v, off);
        v = kMax ? fmaxf(v, o) : v + o;
    }
    __syncthreads();  // red may still be read from a previous reduction
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
    __syncthreads();
    float r = red[0];
#pragma unroll
    for (int w = 1; w < kThreads / 32; ++w) r = kMax ? fmaxf(r, red[w]) : r + red[w];
    return r;
}

struct DecSelArgs {
    const __nv_bfloat16* q;
    const __nv_bfloat16* Kr;
    const int32_t* lens;
    int32_t* idx;
    int32_t* cnt;
    int* status;
    int Hq, Hkv, L, Tc, topk, n_init, n_local;
    float scale_log2;
};

// Shared memory: S [G][Tc] (scores, log2 units), A [Tc], finalists, picks.
size_t dec_select_smem(int G, int Tc, int topk) {
    return (size_t)(G + 1) * Tc * 4 + 8 * topk::kFinalMax * 8 + (size_t)topk * 4 + 64;
}

template <int G>
__global__ void __launch_bounds__(kThreads)
decode_select_kernel(const DecSelArgs a) {
    extern __shared__ __align__(16) uint8_t smem[];
    unsigned long long* fin = reinterpret_cast<unsigned long long*>(smem);
    float* red = reinterpret_cast<float*>(smem + 8 * topk::kFinalMax * 8);   // 8 floats
    float* S = red + 16;                                                        // [G][Tc]
    float* A = S + (size_t)G * a.Tc;                                            // [Tc]
    int* sel = reinterpret_cast<int*>(A + a.Tc);                                // [topk]
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int u = blockIdx.x;
    const int b = u / a.Hkv, g = u % a.Hkv;
    const int len = a.lens[b];
    int32_t* out = a.idx + (size_t)u * a.topk;
    if (len <= 0 || len > a.L) {  // no query (or a bad length): empty selection
        if (tid == 0 && (len < 0 || len > a.L)) set_status(a.status, PHSA_ERR_DEVICE_INDEX);
        for (int j = tid; j < a.topk; j += kThreads) out[j] = -1;
        if (tid == 0) a.cnt[u] = 0;
        return;
    }
    const int qb = (len - 1) / kM;
    const int n_init_q = min(a.n_init, qb + 1);            // forced initial [0, n_init_q)
    const int loc_lo = max(n_init_q, qb - a.n_local + 1);  // forced local [loc_lo, qb]
    const int c_lo = a.n_init, c_hi = qb - a.n_local;      // candidates, all full blocks
    const int nC = max(0, c_hi - c_lo + 1);
    const int nF = n_init_q + (qb - loc_lo + 1);
    const int ksel = a.topk - nF;
    if (ksel >= nC) {  // the budget covers every candidate
        const int n = nF + nC;
        for (int j = tid; j < a.topk; j += kThreads) {
            int v = -1;
            if (j < n_init_q) v = j;
            else if (j < n_init_q + nC) v = c_lo + (j - n_init_q);
            else if (j < n) v = loc_lo + (j - n_init_q - nC);
            out[j] = v;
        }
        if (tid == 0) a.cnt[u] = n;
        return;
    }

    // ---- scores: half-warp hw takes candidates hw, hw + 16, ... four at a time
    const int hw = tid >> 4, c16 = tid & 15;
    float qv[G][8];
#pragma unroll
    for (int h = 0; h < G; ++h)
        load_q8(a.q + ((size_t)b * a.Hq + g * G + h) * kD + c16 * 8, a.scale_log2, qv[h]);
    const __nv_bfloat16* Krg = a.Kr + ((size_t)u * a.Tc + c_lo) * kD + c16 * 8;
    // The trip count is the same for every thread, so both half-warps of a warp
    // always reach the shuffles of dot8_half together.
    for (int base = hw; base - hw < nC; base += 64) {
        uint4 kv[4];
#pragma unroll
        for (int r = 0; r < 4; ++r) {
            const int cj = base + 16 * r;
            kv[r] = cj < nC ? __ldg(reinterpret_cast<const uint4*>(Krg + (size_t)cj * kD))
                            : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int r = 0; r < 4; ++r) {
            const int cj = base + 16 * r;
#pragma unroll
            for (int h = 0; h < G; ++h) {
                const float s = dot8_half(qv[h], kv[r]);
                if (c16 == 0 && cj < nC) S[h * a.Tc + cj] = s;
            }
        }
    }
    __syncthreads();

    // ---- per head: softmax over the candidates; A_t = sum over heads
    float mx[G], iz[G];
#pragma unroll
    for (int h = 0; h < G; ++h) {
        float m = -INFINITY;
        for (int cj = tid; cj < nC; cj += kThreads) m = fmaxf(m, S[h * a.Tc + cj]);
        mx[h] = block_reduce<true>(m, red);
        float z = 0.f;
        for (int cj = tid; cj < nC; cj += kThreads) z += exp2f(S[h * a.Tc + cj] - mx[h]);
        z = block_reduce<false>(z, red);
        iz[h] = z > 0.f ? 1.0f / z : 0.f;
    }
    for (int cj = tid; cj < nC; cj += kThreads) {
        float acc = 0.f;
#pragma unroll
        for (int h = 0; h < G; ++h) acc += exp2f(S[h * a.Tc + cj] - mx[h]) * iz[h];
        A[cj] = acc;
    }
    __syncthreads();

    // ---- top-k
    auto key_of = [&](int cj) { return topk::make_key(A[cj], c_lo + cj); };
    const bool fast = topk::two_level(nC, ksel);
    if (fast) {
        topk::level1(nC, ksel, key_of, fin, warp, lane);
    } else if (warp == 0) {
        topk::rounds_one_warp(
            nC, ksel, key_of, [&](int cj) { return A[cj] == -1.0f; },
            [&](int t) { A[t - c_lo] = -1.0f; }, sel, lane);
    }
    __syncthreads();
    if (fast) topk::level2(fin, ksel, sel, tid);
    __syncthreads();

    // ---- forced + picked, ascending, -1 padded
    for (int j = tid; j < a.topk; j += kThreads) {
        if (j < n_init_q) out[j] = j;
        else if (j >= n_init_q + ksel && j < nF + ksel) out[j] = loc_lo + (j - n_init_q - ksel);
        else if (j >= nF + ksel) out[j] = -1;
    }
    for (int j = tid; j < ksel; j += kThreads) {
        const int v = sel[j];
        int rank = 0;
        for (int i = 0; i < ksel; ++i) rank += sel[i] < v;
        out[n_init_q + rank] = v;
    }
    if (tid == 0) a.cnt[u] = nF + ksel;
}

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
    int Hq, Hkv, L, topk;
    float scale_log2;
};

// Shared memory: block list [topk] | per half-warp state [16][G][2 + 128].
size_t dec_attn_smem(int G, int topk) {
    return (size_t)((topk + 4) & ~3) * 4 + (size_t)16 * G * 130 * 4;
}

template <int G>
__global__ void __launch_bounds__(kThreads)
decode_attn_kernel(const DecAttnArgs a) {
    extern __shared__ __align__(16) uint8_t smem[];
    int* list = reinterpret_cast<int*>(smem);
    float* part = reinterpret_cast<float*>(smem + (size_t)((a.topk + 4) & ~3) * 4);
    __shared__ int s_n;
    const int tid = threadIdx.x;
    const int u = blockIdx.x;
    const int b = u / a.Hkv, g = u % a.Hkv;
    const int len = a.lens[b];
    const size_t orow = (size_t)b * a.Hq + g * G;  // first query head of the group
    if (len <= 0 || len > a.L) {  // no query: zero output, lse = -inf
        if (tid == 0 && (len < 0 || len > a.L)) set_status(a.status, PHSA_ERR_DEVICE_INDEX);
        for (int e = tid; e < G * kD; e += kThreads)
            a.O[orow * kD + e] = __float2bfloat16_rn(0.f);
        if (tid < G) a.lse[orow + tid] = -INFINITY;
        return;
    }
    const int p = len - 1, qb = p / kM;
    if (tid == 0) s_n = compact_block_list(a.idx + (size_t)u * a.topk, a.cnt[u], a.topk, qb, list, a.status);
    __syncthreads();
    const int nk = s_n * kM;

    const int hw = tid >> 4, c16 = tid & 15;
    float qv[G][8];
#pragma unroll
    for (int h = 0; h < G; ++h) load_q8(a.q + (orow + h) * kD + c16 * 8, a.scale_log2, qv[h]);
    const __nv_bfloat16* Kg = a.K + (size_t)u * a.L * kD + c16 * 8;
    const __nv_bfloat16* Vg = a.V + (size_t)u * a.L * kD + c16 * 8;

    float m[G], l[G], o[G][8];
#pragma unroll
    for (int h = 0; h < G; ++h) {
        m[h] = -INFINITY;
        l[h] = 0.f;
#pragma unroll
        for (int e = 0; e < 8; ++e) o[h][e] = 0.f;
    }
    // Half-warp hw takes keys [4 hw, 4 hw + 4) of every 64: four consecutive rows.
    for (int kb = 4 * hw; kb < nk; kb += 64) {
        uint4 kr[4], vr[4];
        int pos[4];
#pragma unroll
        for (int r = 0; r < 4; ++r) {
            const int key = kb + r;
            pos[r] = list[key >> 6] * kM + (key & 63);
            const bool ok = pos[r] <= p;
            kr[r] = ok ? __ldg(reinterpret_cast<const uint4*>(Kg + (size_t)pos[r] * kD))
                       : make_uint4(0u, 0u, 0u, 0u);
            vr[r] = ok ? __ldg(reinterpret_cast<const uint4*>(Vg + (size_t)pos[r] * kD))
                       : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int h = 0; h < G; ++h) {
            float s[4];
            float mn = m[h];
#pragma unroll
            for (int r = 0; r < 4; ++r) {
                // dot8_half shuffles across the whole warp: call it on every lane
                // (a masked key holds zeros), then mask the score
                const float d = dot8_half(qv[h], kr[r]);
                s[r] = pos[r] <= p ? d : -INFINITY;
                mn = fmaxf(mn, s[r]);
            }
            if (mn == -INFINITY) continue;  // no key of this step is visible
            const float sc = exp2f(m[h] - mn);
            l[h] *= sc;
#pragma unroll
            for (int e = 0; e < 8; ++e) o[h][e] *= sc;
#pragma unroll
            for (int r = 0; r < 4; ++r) {
                const float pr = exp2f(s[r] - mn);
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
    }
    // ---- merge the 16 half-warp states
#pragma unroll
    for (int h = 0; h < G; ++h) {
        float* st = part + ((size_t)hw * G + h) * 130;
        if (c16 == 0) {
            st[0] = m[h];
            st[1] = l[h];
        }
#pragma unroll
        for (int e = 0; e < 8; ++e) st[2 + c16 * 8 + e] = o[h][e];
    }
    __syncthreads();
    if (tid < G * kD) {
        const int h = tid / kD, d = tid % kD;
        float M = -INFINITY;
        for (int w = 0; w < 16; ++w) M = fmaxf(M, part[((size_t)w * G + h) * 130]);
        float Ls = 0.f, acc = 0.f;
        if (M != -INFINITY) {
            for (int w = 0; w < 16; ++w) {
                const float* st = part + ((size_t)w * G + h) * 130;
                const float f = exp2f(st[0] - M);  // 0 for a half-warp that saw no key
                Ls += st[1] * f;
                acc += st[2 + d] * f;
            }
        }
        a.O[(orow + h) * kD + d] = __float2bfloat16_rn(Ls > 0.f ? acc / Ls : 0.f);
        if (d == 0) a.lse[orow + h] = Ls > 0.f ? (M + log2f(Ls)) * kLn2 : -INFINITY;
    }
}

}  // namespace

size_t decode_select_smem_bytes(const phsa_shape& s, int topk) {
    return dec_select_smem(s.Hq / s.Hkv, s.L / kM, topk);
}

cudaError_t launch_decode_select(const void* q, const void* Krepr, const int32_t* lens,
                                 const phsa_shape& s, const phsa_select_params& p, int32_t* idx,
                                 int32_t* cnt, int* status, cudaStream_t st) {
    const int G = s.Hq / s.Hkv, Tc = s.L / kM;
    const size_t smem = dec_select_smem(G, Tc, p.topk);
    DecSelArgs args{static_cast<const __nv_bfloat16*>(q), static_cast<const __nv_bfloat16*>(Krepr),
                    lens, idx, cnt, status, s.Hq, s.Hkv, s.L, Tc, p.topk, p.n_init, p.n_local,
                    p.sm_scale * kLog2e};
    const unsigned grid = (unsigned)((long long)s.B * s.Hkv);
    auto kern = G == 2 ? decode_select_kernel<2> : decode_select_kernel<1>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    ProfScope prof(K_DEC_SELECT, st);
    kern<<<grid, kThreads, smem, st>>>(args);
    return cudaGetLastError();
}

cudaError_t launch_decode_attn(const void* q, const void* K, const void* V, const int32_t* idx,
                               const int32_t* cnt, const int32_t* lens, const phsa_shape& s,
                               int topk, float sm_scale, void* O, float* lse, int* status,
                               cudaStream_t st) {
    const int G = s.Hq / s.Hkv;
    const size_t smem = dec_attn_smem(G, topk);
    DecAttnArgs args{static_cast<const __nv_bfloat16*>(q), static_cast<const __nv_bfloat16*>(K),
                     static_cast<const __nv_bfloat16*>(V), idx, cnt, lens,
                     static_cast<__nv_bfloat16*>(O), lse, status, s.Hq, s.Hkv, s.L, topk,
                     sm_scale * kLog2e};
    const unsigned grid = (unsigned)((long long)s.B * s.Hkv);
    auto kern = G == 2 ? decode_attn_kernel<2> : decode_attn_kernel<1>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    ProfScope prof(K_DEC_ATTN, st);
    kern<<<grid, kThreads, smem, st>>>(args);
    return cudaGetLastError();
}

}  // namespace phsa
