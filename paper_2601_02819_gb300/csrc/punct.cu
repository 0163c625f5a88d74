// Punctuation indicator (Section 3.2, Eq. 4-5): mask[i] = I(ids[i] in P).
// Each CTA sorts the punctuation ids into shared memory (bitonic sort, padded
// to a power of two with INT_MAX) and every thread looks its tokens up by
// binary search. Whether INT_MAX itself is in P is recorded separately, since
// it is also the padding value.
#include <climits>

#include "phsa_common.cuh"
#include "phsa_internal.h"

namespace phsa {

namespace {

constexpr int kThreads = 256;

__global__ void __launch_bounds__(kThreads)
punct_mask_kernel(const int32_t* __restrict__ ids, long long n, const int32_t* __restrict__ pid,
                  int np, int npow, uint8_t* __restrict__ mask) {
    extern __shared__ int set[];  // npow ints
    __shared__ int has_max;
    if (threadIdx.x == 0) has_max = 0;
    __syncthreads();
    for (int i = threadIdx.x; i < npow; i += kThreads) {
        const int v = i < np ? pid[i] : INT_MAX;
        set[i] = v;
        if (i < np && v == INT_MAX) has_max = 1;
    }
    __syncthreads();
    for (int k = 2; k <= npow; k <<= 1)  // ascending bitonic sort
        for (int j = k >> 1; j > 0; j >>= 1) {
            for (int i = threadIdx.x; i < npow; i += kThreads) {
                const int l = i ^ j;
                if (l > i) {
                    const int a = set[i], b = set[l];
                    if ((a > b) == ((i & k) == 0)) {
                        set[i] = b;
                        set[l] = a;
                    }
                }
            }
            __syncthreads();
        }
    for (long long t = (long long)blockIdx.x * kThreads + threadIdx.x; t < n;
         t += (long long)gridDim.x * kThreads) {
        const int x = ids[t];
        int lo = 0, hi = npow;  // first entry >= x
        while (lo < hi) {
            const int mid = (lo + hi) >> 1;
            if (set[mid] < x) lo = mid + 1;
            else hi = mid;
        }
        const bool hit = lo < npow && set[lo] == x && (x != INT_MAX || has_max);
        mask[t] = hit ? 1 : 0;
    }
}

}  // namespace

cudaError_t launch_punct_mask(const int32_t* ids, long long n, const int32_t* punct_ids,
                              int n_punct, uint8_t* mask, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    int npow = 1;
    while (npow < n_punct) npow <<= 1;
    int dev = 0, nsm = 0;
    cudaError_t e;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
        return e;
    long long grid = (n + kThreads * 8 - 1) / (kThreads * 8);  // 8 tokens per thread
    if (grid > 4LL * nsm) grid = 4LL * nsm;
    if (grid < 1) grid = 1;
    punct_mask_kernel<<<(unsigned)grid, kThreads, (size_t)npow * 4, st>>>(ids, n, punct_ids,
                                                                        n_punct, npow, mask);
    return cudaGetLastError();
}

}  // namespace phsa
