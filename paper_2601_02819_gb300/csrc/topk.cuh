// Top-k block choice shared by the selection kernels (Algorithm 1 step 3):
// the k candidates with the largest aggregate A, ties to the lower block index.
//
// Every candidate gets the 64-bit key bits(A) << 32 | ~t (A >= 0, so the bit
// pattern orders like the value; NaN ranks as zero), and keys are distinct.
//
// Two levels over 8 warps (256 threads):
//   level1  each warp takes an eighth of the candidates, keeps its lanes' keys
//           in registers (at most kLaneKeys per lane) and picks its best
//           min(k, slice) by rounds of a warp-wide maximum; the winners go to
//           fin[warp][0..), the remaining slots stay 0.
//   level2  each finalist counts the finalists with a larger key; rank < k is
//           a pick. The global top k are all finalists, since each of them is
//           within the top k of its own slice.
// Budgets above kFinalMax picks, or more than 8 * 32 * kLaneKeys candidates,
// take one warp's rounds over all candidates instead (rounds_one_warp).
#pragma once

#include <cstdint>

namespace phsa {
namespace topk {

constexpr int kFinalMax = 32;  // picks handled by the two-level path
constexpr int kLaneKeys = 8;   // candidate keys per lane in level 1
constexpr int kMaxCand = 8 * 32 * kLaneKeys;

__device__ __forceinline__ unsigned long long make_key(float a, int t) {
    if (!(a >= 0.f)) a = 0.f;
    return ((unsigned long long)__float_as_uint(a) << 32) |
           (unsigned long long)(0xffffffffu - (unsigned)t);
}

// The key of an aggregate of any sign (the max-logit rule): the float's bits
// mapped so that unsigned order is numeric order (negatives flipped, the sign
// bit set on the rest); -0 counts as +0 and NaN below every number. Every such
// key is nonzero, so 0 still marks an empty slot.
__device__ __forceinline__ unsigned long long make_key_signed(float a, int t) {
    if (a != a) a = -INFINITY;
    if (a == 0.f) a = 0.f;
    unsigned u = __float_as_uint(a);
    u = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
    return ((unsigned long long)u << 32) | (unsigned long long)(0xffffffffu - (unsigned)t);
}

// The key under either rule: summed probabilities (>= 0) or max logits.
__device__ __forceinline__ unsigned long long make_key_agg(float a, int t, bool max_logit) {
    return max_logit ? make_key_signed(a, t) : make_key(a, t);
}

__device__ __forceinline__ int key_block(unsigned long long key) {
    return (int)(0xffffffffu - (unsigned)(key & 0xffffffffull));
}

__device__ __forceinline__ unsigned long long umax64(unsigned long long a, unsigned long long b) {
    return a > b ? a : b;
}

__device__ __forceinline__ bool two_level(int nC, int ksel) {
    return ksel <= kFinalMax && nC <= kMaxCand;
}

// Level 1, called by each of the 8 warps with its warp index; key_of(cj) gives
// the key of candidate cj in [0, nC). fin holds 8 * kFinalMax keys.
template <class KeyOf>
__device__ __forceinline__ void level1(int nC, int ksel, KeyOf key_of, unsigned long long* fin,
                                       int warp, int lane) {
    const int per = (nC + 7) >> 3;
    const int lo = min(nC, warp * per), hi = min(nC, lo + per);
    const int nf = min(ksel, hi - lo);
    unsigned long long key[kLaneKeys];
#pragma unroll
    for (int r = 0; r < kLaneKeys; ++r) {
        const int cj = lo + lane + 32 * r;
        key[r] = cj < hi ? key_of(cj) : 0ull;
    }
    for (int k = lane; k < kFinalMax; k += 32) fin[warp * kFinalMax + k] = 0ull;
    __syncwarp();
    for (int k = 0; k < nf; ++k) {
        unsigned long long best = key[0];
#pragma unroll
        for (int r = 1; r < kLaneKeys; ++r) best = umax64(best, key[r]);
        const unsigned mh = (unsigned)(best >> 32), ml = (unsigned)best;
        const unsigned bh = __reduce_max_sync(0xffffffffu, mh);
        const unsigned bl = __reduce_max_sync(0xffffffffu, mh == bh ? ml : 0u);
        const unsigned long long win = ((unsigned long long)bh << 32) | bl;
        if (lane == 0) fin[warp * kFinalMax + k] = win;
#pragma unroll
        for (int r = 0; r < kLaneKeys; ++r)
            if (key[r] == win) key[r] = 0ull;
    }
}

// Level 2, called by all 256 threads after level 1 is visible to them: writes
// the block index of the pick of rank r to sel[r], r < ksel.
__device__ __forceinline__ void level2(const unsigned long long* fin, int ksel, int* sel,
                                       int tid) {
    const unsigned long long mykey = tid < 8 * kFinalMax ? fin[tid] : 0ull;
    if (mykey == 0ull) return;
    int rank = 0;
    const int pairs = (ksel + 1) >> 1;  // finalists sit at the front of each warp's slots
    for (int w = 0; w < 8; ++w) {
        const ulonglong2* f2 = reinterpret_cast<const ulonglong2*>(fin + w * kFinalMax);
#pragma unroll 4
        for (int j = 0; j < pairs; ++j) {
            const ulonglong2 v = f2[j];
            rank += (v.x > mykey) + (v.y > mykey);
        }
    }
    if (rank < ksel) sel[rank] = key_block(mykey);
}

// One warp, any budget: rounds over all candidates; taken(cj) / take(cj) mark a
// candidate as chosen (the caller's storage). sel[k] = k-th pick.
template <class KeyOf, class Taken, class Take>
__device__ __forceinline__ void rounds_one_warp(int nC, int ksel, KeyOf key_of, Taken taken,
                                                Take take, int* sel, int lane) {
    auto lane_best = [&]() {
        unsigned long long best = 0ull;
        for (int cj = lane; cj < nC; cj += 32)
            if (!taken(cj)) best = umax64(best, key_of(cj));
        return best;
    };
    unsigned long long mine = lane_best();
    for (int k = 0; k < ksel; ++k) {
        const unsigned mh = (unsigned)(mine >> 32), ml = (unsigned)mine;
        const unsigned bh = __reduce_max_sync(0xffffffffu, mh);
        const unsigned bl = __reduce_max_sync(0xffffffffu, mh == bh ? ml : 0u);
        const unsigned long long win = ((unsigned long long)bh << 32) | bl;
        if (lane == 0) sel[k] = key_block(win);
        if (bl != 0u && mine == win) {
            take(key_block(win));
            mine = lane_best();
        }
        __syncwarp();
    }
}

__device__ __forceinline__ unsigned long long warp_max64(unsigned long long v) {
    const unsigned vh = (unsigned)(v >> 32), vl = (unsigned)v;
    const unsigned bh = __reduce_max_sync(0xffffffffu, vh);
    const unsigned bl = __reduce_max_sync(0xffffffffu, vh == bh ? vl : 0u);
    return ((unsigned long long)bh << 32) | bl;
}

__device__ __forceinline__ unsigned long long shfl64(unsigned long long v, int src) {
    const unsigned h = __shfl_sync(0xffffffffu, (unsigned)(v >> 32), src);
    const unsigned l = __shfl_sync(0xffffffffu, (unsigned)v, src);
    return ((unsigned long long)h << 32) | l;
}

__device__ __forceinline__ unsigned long long shfl_up64(unsigned long long v, int d) {
    const unsigned h = __shfl_up_sync(0xffffffffu, (unsigned)(v >> 32), d);
    const unsigned l = __shfl_up_sync(0xffffffffu, (unsigned)v, d);
    return ((unsigned long long)h << 32) | l;
}

__device__ __forceinline__ unsigned long long umin64(unsigned long long a, unsigned long long b) {
    return a < b ? a : b;
}

__device__ __forceinline__ unsigned long long shfl_xor64(unsigned long long v, int m) {
    const unsigned h = __shfl_xor_sync(0xffffffffu, (unsigned)(v >> 32), m);
    const unsigned l = __shfl_xor_sync(0xffffffffu, (unsigned)v, m);
    return ((unsigned long long)h << 32) | l;
}

// The 32 largest keys of two lists sorted descending across the lanes (lane k
// holds the k-th largest of each), sorted descending again: the lane-wise
// maximum of one list and the other reversed holds the 32 largest keys of
// both as a bitonic sequence, and five half-cleaner stages sort it.
__device__ __forceinline__ unsigned long long merge_top32(unsigned long long a, unsigned long long b,
                                                          int lane) {
    unsigned long long v = umax64(a, shfl64(b, 31 - lane));
#pragma unroll
    for (int j = 16; j >= 1; j >>= 1) {
        const unsigned long long o = shfl_xor64(v, j);
        v = (lane & j) ? umin64(v, o) : umax64(v, o);
    }
    return v;
}

// One warp, at most 32 picks, any number of candidates. A first pass takes the
// largest key of each lane's candidates; the ksel-th largest of those 32
// maxima, tau, is at most the ksel-th largest key of all (ksel lanes hold a key
// >= tau), so every pick is >= tau. A second pass inserts the keys >= tau, in
// candidate order, into a list kept sorted across the lanes (lane k holds the
// k-th largest key so far): one ballot finds a key's place and one shuffle
// shifts the keys below it. Only the keys >= tau are inserted, usually a small
// multiple of ksel. Returns this lane's pick (lane < ksel; 0 on the other
// lanes). Requires 1 <= ksel <= 32 and ksel <= nC; keys are nonzero.
template <class KeyOf>
__device__ __forceinline__ unsigned long long warp_topk32_filtered(int nC, int ksel, KeyOf key_of, int lane) {
    unsigned long long lmax = 0ull;
    for (int cj = lane; cj < nC; cj += 32) lmax = umax64(lmax, key_of(cj));
    unsigned long long v = lmax, tau = 0ull;
    for (int k = 0; k < ksel; ++k) {
        const unsigned long long win = warp_max64(v);
        tau = win;
        if (v == win) v = 0ull;
    }
    unsigned long long best = 0ull;
    for (int base = 0; base < nC; base += 32) {
        const int cj = base + lane;
        const unsigned long long x = cj < nC ? key_of(cj) : 0ull;
        unsigned m = __ballot_sync(0xffffffffu, x != 0ull && x >= tau);
        while (m) {
            const int src = __ffs(m) - 1;
            m &= m - 1;
            const unsigned long long y = shfl64(x, src);
            const int pos = __popc(__ballot_sync(0xffffffffu, lane < ksel && best > y));
            const unsigned long long up = shfl_up64(best, 1);
            if (pos < ksel && lane < ksel && lane >= pos) best = lane == pos ? y : up;
        }
    }
    return best;
}

// One warp, at most 32 picks, any number of candidates: the candidates are
// taken 512 at a time (16 keys per lane in registers) together with the picks
// so far (lane k holds the k-th best key, one register), and ksel rounds of a
// warp-wide maximum keep the best ksel of them. Returns this lane's pick
// (lane < ksel; 0 on the other lanes). Requires 1 <= ksel <= 32 and ksel <= nC.
template <class KeyOf>
__device__ __forceinline__ unsigned long long warp_topk32_rounds(int nC, int ksel, KeyOf key_of, int lane) {
    unsigned long long best = 0ull;
    for (int base = 0; base < nC; base += 512) {
        unsigned long long key[16];
#pragma unroll
        for (int r = 0; r < 16; ++r) {
            const int cj = base + lane + 32 * r;
            key[r] = cj < nC ? key_of(cj) : 0ull;
        }
        unsigned long long carry = best;
        best = 0ull;
        for (int k = 0; k < ksel; ++k) {
            unsigned long long m = carry;
#pragma unroll
            for (int r = 0; r < 16; ++r) m = umax64(m, key[r]);
            const unsigned mh = (unsigned)(m >> 32), ml = (unsigned)m;
            const unsigned bh = __reduce_max_sync(0xffffffffu, mh);
            const unsigned bl = __reduce_max_sync(0xffffffffu, mh == bh ? ml : 0u);
            const unsigned long long win = ((unsigned long long)bh << 32) | bl;
            if (lane == k) best = win;
            if (carry == win) carry = 0ull;
#pragma unroll
            for (int r = 0; r < 16; ++r)
                if (key[r] == win) key[r] = 0ull;
        }
    }
    return best;
}

// One warp, at most 32 picks (lane k returns the k-th best, 0 past ksel). The
// rounds cost ksel per 512 candidates, the filtered insertion about 2.6 ksel
// insertions on random aggregates plus two passes over the candidates.
// Measured: at budgets up to 16 the filtered form wins at every length (32k at
// m = 16, ksel 16: the selection 508 -> 408 us); at ksel 30 over slices of
// 512 (131k at m = 64) the rounds do (1897 against 2187 us), and they are kept
// up to 1024 candidates at budgets above 16.
template <class KeyOf>
__device__ __forceinline__ unsigned long long warp_topk32(int nC, int ksel, KeyOf key_of, int lane) {
    return ksel <= 16 || nC > 1024 ? warp_topk32_filtered(nC, ksel, key_of, lane)
                                   : warp_topk32_rounds(nC, ksel, key_of, lane);
}

// One warp, any budget: rounds over all candidates that mark each pick with
// take(t) in the caller's storage (taken(cj) tests the mark); no list of picks
// is kept, so the caller reads the picks back in ascending order.
template <class KeyOf, class Taken, class Take>
__device__ __forceinline__ void rounds_mark_one_warp(int nC, int ksel, KeyOf key_of, Taken taken,
                                                     Take take, int lane) {
    auto lane_best = [&]() {
        unsigned long long best = 0ull;
        for (int cj = lane; cj < nC; cj += 32)
            if (!taken(cj)) best = umax64(best, key_of(cj));
        return best;
    };
    unsigned long long mine = lane_best();
    for (int k = 0; k < ksel; ++k) {
        const unsigned mh = (unsigned)(mine >> 32), ml = (unsigned)mine;
        const unsigned bh = __reduce_max_sync(0xffffffffu, mh);
        const unsigned bl = __reduce_max_sync(0xffffffffu, mh == bh ? ml : 0u);
        const unsigned long long win = ((unsigned long long)bh << 32) | bl;
        if (bl != 0u && mine == win) {
            take(key_block(win));
            mine = lane_best();
        }
        __syncwarp();
    }
}

}  // namespace topk
}  // namespace phsa
