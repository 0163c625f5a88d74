// Stage (a): representative key of every KV block (Section 3.2, Eq. 6-8;
// Algorithm 1 step 2).
//
// One warp reduces one m x 128 bf16 block (m = 64: 16 KB; the kernel is
// instantiated for m = 16, 32, 64). Each half-warp streams one
// 256-byte row per step with 16-byte read-only loads (lane c of the half owns
// columns 8c..8c+7), so a warp keeps up to sixteen 512-byte row pairs in flight. The
// punctuation count of the block comes from warp ballots over its m mask
// bytes. The sum and the punctuation-masked sum are kept in fp32 and combined
// once across the two half-warps; the result is rounded to bf16 once.
// The kernel is bound by HBM: it reads K and the mask once and writes T rows.
// decode_repr_kernel reuses the per-block routine for the block a decode step
// has just filled (block-level caching of the representative keys).
#include "phsa_common.cuh"
#include "phsa_internal.h"

namespace phsa {

namespace {

constexpr int kWarpsPerCta = 8;

__device__ __forceinline__ void add8(float* acc, const uint4& v) {
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        float2 f = __bfloat1622float2(h[j]);
        acc[2 * j] += f.x;
        acc[2 * j + 1] += f.y;
    }
}

// One warp: the representative key of the BM x 128 block at Kb (row stride
// 128) with punctuation bytes mb[0..BM), written as 128 bf16 values to out.
template <int BM>
__device__ __forceinline__ void repr_one_block(const __nv_bfloat16* __restrict__ Kb,
                                               const uint8_t* __restrict__ mb, float lambda,
                                               __nv_bfloat16* __restrict__ out, int lane) {
    static_assert(BM == 16 || BM == 32 || BM == 64, "block size");
    // Punctuation indicator of the block's BM tokens (bit r: token r).
    const unsigned lo = __ballot_sync(0xffffffffu, lane < BM && mb[lane < BM ? lane : 0] != 0);
    const unsigned hi = BM > 32 ? __ballot_sync(0xffffffffu, mb[(BM > 32 ? 32 : 0) + lane] != 0) : 0u;
    const int c = __popc(lo) + __popc(hi);

    const int half = lane >> 4;
    const int col = lane & 15;
    const __nv_bfloat16* kb = Kb + col * 8;

    float s0[8], sp[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) { s0[j] = 0.f; sp[j] = 0.f; }

    // up to 32 rows (16 loads of 16 bytes per lane, 8 KB per warp) in flight per batch
    constexpr int kRB = BM < 32 ? BM : 32;
#pragma unroll
    for (int base = 0; base < BM; base += kRB) {
        uint4 v[kRB / 2];
#pragma unroll
        for (int u = 0; u < kRB / 2; ++u) {
            const int r = base + 2 * u + half;
            v[u] = __ldg(reinterpret_cast<const uint4*>(kb + (size_t)r * kD));
        }
#pragma unroll
        for (int u = 0; u < kRB / 2; ++u) {
            const int r = base + 2 * u + half;
            add8(s0, v[u]);
            const bool p = ((r < 32 ? lo >> r : hi >> (r - 32)) & 1u) != 0;
            if (p) add8(sp, v[u]);
        }
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        s0[j] += __shfl_xor_sync(0xffffffffu, s0[j], 16);
        sp[j] += __shfl_xor_sync(0xffffffffu, sp[j], 16);
    }
    if (half == 0) {
        float o[8];
        const float inv_m = 1.0f / BM;
        const float inv_c = c > 0 ? 1.0f / (float)c : 0.f;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const float m0 = s0[j] * inv_m;                                // Eq. 6
            o[j] = c > 0 ? lambda * m0 + (1.0f - lambda) * (sp[j] * inv_c)  // Eq. 7-8
                         : m0;                                           // no punctuation
        }
        uint4 pk;
        pk.x = pack_bf16(o[0], o[1]);
        pk.y = pack_bf16(o[2], o[3]);
        pk.z = pack_bf16(o[4], o[5]);
        pk.w = pack_bf16(o[6], o[7]);
        *reinterpret_cast<uint4*>(out + col * 8) = pk;
    }
}

template <int BM>
__global__ void __launch_bounds__(kWarpsPerCta * 32)
block_repr_kernel(const __nv_bfloat16* __restrict__ K, const uint8_t* __restrict__ mask, int Hkv,
                  int L, int T, long long n_blocks, float lambda,
                  __nv_bfloat16* __restrict__ Krepr) {
    const int lane = threadIdx.x & 31;
    const long long wid = (long long)blockIdx.x * kWarpsPerCta + (threadIdx.x >> 5);
    if (wid >= n_blocks) return;
    const int t = (int)(wid % T);
    const long long bg = wid / T;  // b * Hkv + g
    const int b = (int)(bg / Hkv);
    repr_one_block<BM>(K + ((size_t)bg * L + (size_t)t * BM) * kD,
                       mask + (size_t)b * L + (size_t)t * BM, lambda,
                       Krepr + ((size_t)bg * T + t) * kD, lane);
}

// Decode: one CTA of four warps per (sequence, KV head). A sequence whose
// length is a positive multiple of m has just filled its last block: that
// block's representative key is computed (Eq. 6-8, the arithmetic of
// repr_one_block); nothing else is touched. Warp w < m / 16 sums rows
// [16w, 16w + 16) with all of its 16-byte loads issued at once; the m / 16
// partial sums are added in warp order in shared memory.
constexpr int kDecReprWarps = 4;

__global__ void __launch_bounds__(kDecReprWarps * 32)
decode_repr_kernel(const __nv_bfloat16* __restrict__ K, const uint8_t* __restrict__ mask,
                   const int32_t* __restrict__ lens, int Hkv, int L, int T, int bm, float lambda,
                   __nv_bfloat16* __restrict__ Krepr, int* status) {
    __shared__ float part[kDecReprWarps][2][kD];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const long long bg = blockIdx.x;
    const int b = (int)(bg / Hkv);
    const int len = lens[b];
    if (len < 0 || len > L) {
        if (threadIdx.x == 0) set_status(status, PHSA_ERR_DEVICE_INDEX);
        return;
    }
    if (len == 0 || len % bm != 0) return;
    const int t = len / bm - 1;
    const uint8_t* mb = mask + (size_t)b * L + (size_t)t * bm;
    const unsigned lo = __ballot_sync(0xffffffffu, lane < bm && mb[lane] != 0);
    const unsigned hi = __ballot_sync(0xffffffffu, bm > 32 && mb[bm > 32 ? 32 + lane : 0] != 0);
    const int c = __popc(lo) + __popc(hi);
    const int half = lane >> 4, col = lane & 15;
    const int nw = bm / 16;  // warps with rows
    if (warp < nw) {
        const __nv_bfloat16* kb = K + ((size_t)bg * L + (size_t)t * bm + 16 * warp) * kD + col * 8;
        uint4 v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u)
            v[u] = __ldg(reinterpret_cast<const uint4*>(kb + (size_t)(2 * u + half) * kD));
        float s0[8], sp[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) { s0[j] = 0.f; sp[j] = 0.f; }
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const int r = 16 * warp + 2 * u + half;
            add8(s0, v[u]);
            if (((r < 32 ? lo >> r : hi >> (r - 32)) & 1u) != 0) add8(sp, v[u]);
        }
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            s0[j] += __shfl_xor_sync(0xffffffffu, s0[j], 16);
            sp[j] += __shfl_xor_sync(0xffffffffu, sp[j], 16);
        }
        if (half == 0) {
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                part[warp][0][col * 8 + j] = s0[j];
                part[warp][1][col * 8 + j] = sp[j];
            }
        }
    }
    __syncthreads();
    const int d = threadIdx.x;  // one column per thread
    float a0 = 0.f, ap = 0.f;
    for (int w = 0; w < nw; ++w) {
        a0 += part[w][0][d];
        ap += part[w][1][d];
    }
    const float m0 = a0 * (1.0f / (float)bm);                        // Eq. 6
    const float o = c > 0 ? lambda * m0 + (1.0f - lambda) * (ap * (1.0f / (float)c))  // Eq. 7-8
                          : m0;                                      // no punctuation
    Krepr[((size_t)bg * T + t) * kD + d] = __float2bfloat16_rn(o);
}

}  // namespace

cudaError_t launch_block_repr(const void* K, const uint8_t* mask, const phsa_shape& s,
                              float lambda, void* Krepr, cudaStream_t st) {
    const int bm = s.block_size;
    if (bm != 16 && bm != 32 && bm != 64) return cudaErrorInvalidValue;
    const int T = s.L / bm;
    const long long n_blocks = (long long)s.B * s.Hkv * T;
    if (n_blocks == 0) return cudaSuccess;
    const long long grid = (n_blocks + kWarpsPerCta - 1) / kWarpsPerCta;
    auto kern = bm == 16 ? block_repr_kernel<16> : bm == 32 ? block_repr_kernel<32> : block_repr_kernel<64>;
    ProfScope prof(K_REPR, st);
    kern<<<(unsigned)grid, kWarpsPerCta * 32, 0, st>>>(
        static_cast<const __nv_bfloat16*>(K), mask, s.Hkv, s.L, T, n_blocks, lambda,
        static_cast<__nv_bfloat16*>(Krepr));
    return cudaGetLastError();
}

}  // namespace phsa

namespace phsa {

cudaError_t launch_decode_repr(const void* K, const uint8_t* mask, const int32_t* lens,
                               const phsa_shape& s, float lambda, void* Krepr, int* status,
                               cudaStream_t st) {
    const int bm = s.block_size;
    if (bm != 16 && bm != 32 && bm != 64) return cudaErrorInvalidValue;
    const int T = s.L / bm;
    const long long n_units = (long long)s.B * s.Hkv;
    if (n_units == 0 || T == 0) return cudaSuccess;
    ProfScope prof(K_DEC_REPR, st);
    decode_repr_kernel<<<(unsigned)n_units, kDecReprWarps * 32, 0, st>>>(
        static_cast<const __nv_bfloat16*>(K), mask, lens, s.Hkv, s.L, T, bm, lambda,
        static_cast<__nv_bfloat16*>(Krepr), status);
    return cudaGetLastError();
}

}  // namespace phsa
