// Prefill into per-sequence caches, one chunk of tokens at a time, with the
// representative keys of the blocks the chunk completes computed from the
// same loads (block-level caching of the representative keys, Section 3.2;
// Eq. 3, 6, 7, 8; Algorithm 1 step 2).
//
// One warp per (sequence b, KV head g, block t touched by the chunk). The
// chunk occupies positions [len - C, len) of sequence b (len = seq_lens[b]
// after the append). The warp copies the chunk's rows of block t (K, V, and
// the punctuation flags, once per sequence) into the caches; if the chunk
// completes block t ((t + 1) m <= len), it also sums all m rows of the block
// -- rows before the chunk read back from the cache, the chunk's rows from
// the registers that carry them to the cache -- and writes the block's
// representative key. The loads and sums follow block_repr_kernel<m>'s order
// exactly (half-warps on alternate rows, eight row pairs per batch, then the
// two halves), so a sequence built chunk by chunk has bit-identical
// representative keys to phsa_build_block_repr over the finished cache, at
// each block size m = 16, 32, 64.
#include "phsa_common.cuh"
#include "phsa_internal.h"

namespace phsa {

namespace {

constexpr int kWarps = 8;

__device__ __forceinline__ void add8(float* acc, const uint4& v) {
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const float2 f = __bfloat1622float2(h[j]);
        acc[2 * j] += f.x;
        acc[2 * j + 1] += f.y;
    }
}

__global__ void __launch_bounds__(kWarps * 32)
prefill_append_kernel(const __nv_bfloat16* __restrict__ kc, const __nv_bfloat16* __restrict__ vc,
                      const uint8_t* __restrict__ fc, const int32_t* __restrict__ lens, int B,
                      int Hkv, int L, int C, int T, int nj, int bm, float lambda,
                      __nv_bfloat16* __restrict__ K, __nv_bfloat16* __restrict__ V,
                      uint8_t* __restrict__ mask, __nv_bfloat16* __restrict__ Krepr, int* status) {
    const int lane = threadIdx.x & 31;
    const long long w = (long long)blockIdx.x * kWarps + (threadIdx.x >> 5);
    if (w >= (long long)B * Hkv * nj) return;
    const int j = (int)(w % nj);
    const long long bg = w / nj;  // b * Hkv + g
    const int b = (int)(bg / Hkv), g = (int)(bg % Hkv);
    const int len = lens[b];
    if (len < C || len > L) {  // the chunk does not fit where the length puts it
        if (g == 0 && j == 0 && lane == 0) set_status(status, PHSA_ERR_DEVICE_INDEX);
        return;
    }
    const int p0 = len - C;           // the chunk's first position
    const int t = p0 / bm + j;        // the block this warp handles
    if (t * bm >= len) return;        // past the chunk
    const bool complete = (t + 1) * bm <= len;
    const size_t blk0 = (size_t)t * bm;  // the block's first position
    const uint8_t* mrow = mask + (size_t)b * L;
    const uint8_t* frow = fc ? fc + (size_t)b * C : nullptr;

    // punctuation flags of the block's rows: the chunk's from the chunk (when
    // given, and written to the cache once per sequence), earlier ones from the cache
    auto flag_of = [&](int r) -> bool {
        const int p = (int)blk0 + r;
        if (p >= len) return false;
        if (p >= p0 && frow) return frow[p - p0] != 0;
        return mrow[p] != 0;
    };
    const unsigned lo = __ballot_sync(0xffffffffu, lane < bm && flag_of(lane));
    const unsigned hi = __ballot_sync(0xffffffffu, bm > 32 && flag_of(32 + lane));
    if (frow && g == 0) {
        for (int r = lane; r < bm; r += 32) {
            const int p = (int)blk0 + r;
            if (p >= p0 && p < len) mask[(size_t)b * L + p] = frow[p - p0] ? 1 : 0;
        }
    }
    const int c = __popc(lo) + __popc(hi);

    const int half = lane >> 4, col = lane & 15;
    const __nv_bfloat16* kcache = K + (size_t)bg * L * kD + col * 8;
    const __nv_bfloat16* kchunk = kc + (size_t)bg * C * kD + col * 8;
    const __nv_bfloat16* vchunk = vc + (size_t)bg * C * kD + col * 8;
    __nv_bfloat16* kdst = K + (size_t)bg * L * kD + col * 8;
    __nv_bfloat16* vdst = V + (size_t)bg * L * kD + col * 8;

    float s0[8], sp[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) { s0[q] = 0.f; sp[q] = 0.f; }
    for (int base = 0; base < bm; base += 16) {
        uint4 v[8], vv[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const int r = base + 2 * u + half;
            const int p = (int)blk0 + r;
            v[u] = make_uint4(0u, 0u, 0u, 0u);
            vv[u] = v[u];
            if (p >= p0 && p < len) {
                v[u] = __ldg(reinterpret_cast<const uint4*>(kchunk + (size_t)(p - p0) * kD));
                vv[u] = __ldg(reinterpret_cast<const uint4*>(vchunk + (size_t)(p - p0) * kD));
            } else if (p < p0 && complete) {
                v[u] = *reinterpret_cast<const uint4*>(kcache + (size_t)p * kD);
            }
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const int r = base + 2 * u + half;
            const int p = (int)blk0 + r;
            if (p >= p0 && p < len) {
                *reinterpret_cast<uint4*>(kdst + (size_t)p * kD) = v[u];
                *reinterpret_cast<uint4*>(vdst + (size_t)p * kD) = vv[u];
            }
            if (complete) {
                add8(s0, v[u]);
                if (((r < 32 ? lo >> r : hi >> (r - 32)) & 1u) != 0) add8(sp, v[u]);
            }
        }
    }
    if (!complete) return;
#pragma unroll
    for (int q = 0; q < 8; ++q) {
        s0[q] += __shfl_xor_sync(0xffffffffu, s0[q], 16);
        sp[q] += __shfl_xor_sync(0xffffffffu, sp[q], 16);
    }
    if (half == 0) {
        float o[8];
        const float inv_m = 1.0f / (float)bm;
        const float inv_c = c > 0 ? 1.0f / (float)c : 0.f;
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            const float m0 = s0[q] * inv_m;                                // Eq. 6
            o[q] = c > 0 ? lambda * m0 + (1.0f - lambda) * (sp[q] * inv_c)  // Eq. 7-8
                         : m0;                                           // no punctuation
        }
        uint4 pk;
        pk.x = pack_bf16(o[0], o[1]);
        pk.y = pack_bf16(o[2], o[3]);
        pk.z = pack_bf16(o[4], o[5]);
        pk.w = pack_bf16(o[6], o[7]);
        *reinterpret_cast<uint4*>(Krepr + ((size_t)bg * T + t) * kD + col * 8) = pk;
    }
}

}  // namespace

cudaError_t launch_prefill_append(const void* k_chunk, const void* v_chunk, const uint8_t* flags,
                                  const int32_t* lens, int C, const phsa_shape& s, float lambda,
                                  void* K, void* V, uint8_t* mask, void* Krepr, int* status,
                                  cudaStream_t st) {
    const int bm = s.block_size;
    if (bm != 16 && bm != 32 && bm != 64) return cudaErrorInvalidValue;
    const int nj = (C + bm - 1) / bm + 1;  // blocks a chunk of C tokens can touch
    const long long warps = (long long)s.B * s.Hkv * nj;
    if (warps == 0 || C == 0) return cudaSuccess;
    const unsigned grid = (unsigned)((warps + kWarps - 1) / kWarps);
    ProfScope prof(K_PREFILL_APPEND, st);
    prefill_append_kernel<<<grid, kWarps * 32, 0, st>>>(
        static_cast<const __nv_bfloat16*>(k_chunk), static_cast<const __nv_bfloat16*>(v_chunk),
        flags, lens, s.B, s.Hkv, s.L, C, s.L / bm, nj, bm, lambda, static_cast<__nv_bfloat16*>(K),
        static_cast<__nv_bfloat16*>(V), mask, static_cast<__nv_bfloat16*>(Krepr), status);
    return cudaGetLastError();
}

}  // namespace phsa
