// The union of the block lists of the kSub = 64/m query blocks of one 64-token
// span (block size m < 64), with owner masks, built by one warp. The
// tcgen05 forward and dQ kernels give the span's 128 query rows (two heads x
// 64 tokens) one key sequence: this union, ascending; an entry's owner mask
// says which of the span's query blocks selected it (bit j: query block j).
#pragma once

#include "phsa_common.cuh"

namespace phsa {

// Warp-collective (all 32 lanes). Lists of query blocks qb0 .. qb0 + nqb - 1
// are rows lu0 .. lu0 + nqb - 1 of idx/cnt (topk entries each). Each list is
// validated as compact_block_list does (-1 entries skipped silently; an entry
// outside [0, qb] or not above the last accepted one skipped and recorded in
// *status): an entry is accepted when it is in range and above every earlier
// in-range entry of its list. bm holds kSub bitmaps of W words (over the
// blocks [0, 32 W)), all zero on entry and left so. Writes the union size to
// *count, the blocks to ul[0 ..) and the owner masks to own[0 ..). Returns the
// size on every lane.
template <int kSub>
__device__ __forceinline__ int build_block_union(const int32_t* __restrict__ idx,
                                                 const int32_t* __restrict__ cnt, long long lu0,
                                                 int qb0, int nqb, int topk, uint32_t* bm, int W,
                                                 int* ul, uint8_t* own, int* count, int* status,
                                                 int lane) {
    int hi = -1;
    for (int j = 0; j < kSub && j < nqb; ++j) {
        const int qbj = qb0 + j;
        const long long lu = lu0 + j;
        int n = __ldg(cnt + lu);
        if (n < 0 || n > topk) {
            if (lane == 0) set_status(status, PHSA_ERR_DEVICE_INDEX);
            n = n < 0 ? 0 : topk;
        }
        int carry = -1;  // the largest in-range entry so far
        for (int e0 = 0; e0 < n; e0 += 32) {
            const int e = e0 + lane;
            const int t = e < n ? __ldg(idx + lu * topk + e) : -1;
            const bool inr = t >= 0 && t <= qbj;
            // exclusive prefix maximum of the in-range entries over the lanes
            int pm = inr ? t : -1;
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
                const int y = __shfl_up_sync(0xffffffffu, pm, off);
                if (lane >= off) pm = max(pm, y);
            }
            int before = __shfl_up_sync(0xffffffffu, pm, 1);
            before = lane == 0 ? carry : max(before, carry);
            const bool accept = inr && t > before;
            if (e < n && t != -1 && !accept) set_status(status, PHSA_ERR_DEVICE_INDEX);
            if (accept) {
                atomicOr(bm + j * W + (t >> 5), 1u << (t & 31));
                hi = max(hi, t);
            }
            carry = max(carry, __shfl_sync(0xffffffffu, pm, 31));
        }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) hi = max(hi, __shfl_xor_sync(0xffffffffu, hi, off));
    __syncwarp();
    const int wn = hi >= 0 ? (hi >> 5) + 1 : 0;
    int pos = 0;
    for (int w0 = 0; w0 < wn; w0 += 32) {
        const int w = w0 + lane;
        uint32_t bj[kSub], u = 0u;
#pragma unroll
        for (int j = 0; j < kSub; ++j) {
            bj[j] = w < wn ? bm[j * W + w] : 0u;
            u |= bj[j];
        }
        const int c = __popc(u);
        int incl = c;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, incl, off);
            if (lane >= off) incl += y;
        }
        int p = pos + incl - c;
        while (u) {
            const int bit = __ffs(u) - 1;
            u &= u - 1;
            uint32_t m = 0;
#pragma unroll
            for (int j = 0; j < kSub; ++j) m |= ((bj[j] >> bit) & 1u) << j;
            ul[p] = 32 * w + bit;
            own[p] = (uint8_t)m;
            ++p;
        }
        pos += __shfl_sync(0xffffffffu, incl, 31);
        if (w < wn)
#pragma unroll
            for (int j = 0; j < kSub; ++j) bm[j * W + w] = 0u;
    }
    if (lane == 0) *count = pos;
    return pos;
}

}  // namespace phsa
