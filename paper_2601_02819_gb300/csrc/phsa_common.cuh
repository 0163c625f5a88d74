// Device helpers shared by the PHSA kernels: bf16 tile movement (cp.async,
// ldmatrix), warp-level bf16 MMA, swizzled shared-memory addressing and the
// device status word.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "phsa.h"

namespace phsa {

constexpr int kD = 128;      // head dimension supported by the kernels
constexpr int kM = 64;       // block size (tokens per KV / query block)
constexpr int kRowChunks = kD * 2 / 16;  // 16-byte chunks per 128-wide bf16 row

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

// Records the first device-side error; later ones are dropped.
__device__ __forceinline__ void set_status(int* status, int code) {
    if (status) atomicCAS(status, 0, code);
}

// Byte offset of 16-byte chunk `c` of row `r` in a [rows][128] bf16 tile whose
// chunks are XOR-swizzled by the row's low 3 bits. Eight consecutive rows at
// the same logical chunk land in eight distinct bank groups, so ldmatrix and
// the 16-byte fills are conflict-free.
__device__ __forceinline__ uint32_t swz(int r, int c) {
    return (uint32_t)(r * (kRowChunks * 16) + ((c ^ (r & 7)) << 4));
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}

// 16-byte global -> shared copy; when !pred the destination is zero-filled and
// nothing is read (the source address is still kept in bounds by callers).
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, bool pred) {
    int n = pred ? 16 : 0;
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src), "r"(n)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                          uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

// D = A(16x16, row) * B(16x8, col) + D, bf16 inputs, fp32 accumulate.
__device__ __forceinline__ void mma16816(float* d, const uint32_t* a, uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
        "{%8,%9}, {%0,%1,%2,%3};\n"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// 2^x on the special-function unit (flush-to-zero; 2^-inf = +0).
__device__ __forceinline__ float ex2_sfu(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&v);
}

// ---- fragment loaders over swizzled [rows][128] bf16 tiles ---------------
// A operand (16 rows x 16 k) at (row0, k-chunk pair kc*2): registers in mma order.
__device__ __forceinline__ void load_a_frag(uint32_t base, int row0, int kc, int lane,
                                            uint32_t* a) {
    int r = row0 + (lane & 15);
    int c = kc * 2 + (lane >> 4);
    ldsm_x4(base + swz(r, c), a[0], a[1], a[2], a[3]);
}
// B operand from a tile stored [n][k] (k contiguous), for two n-tiles
// (n0..n0+7, n0+8..n0+15) and one 16-wide k step kc: b[0..1] n-tile 0, b[2..3] n-tile 1.
__device__ __forceinline__ void load_b_nk(uint32_t base, int n0, int kc, int lane, uint32_t* b) {
    int mi = lane >> 3;
    int r = n0 + ((mi >> 1) << 3) + (lane & 7);
    int c = kc * 2 + (mi & 1);
    ldsm_x4(base + swz(r, c), b[0], b[1], b[2], b[3]);
}
// B operand from a tile stored [k][n] (n contiguous), for one 16-wide k step
// starting at row k0 and two n-tiles starting at column chunk nc (8 columns each).
__device__ __forceinline__ void load_b_kn(uint32_t base, int k0, int nc, int lane, uint32_t* b) {
    int mi = lane >> 3;
    int r = k0 + ((mi & 1) << 3) + (lane & 7);
    int c = nc + (mi >> 1);
    ldsm_x4_t(base + swz(r, c), b[0], b[1], b[2], b[3]);
}

// Copies a [64][128] bf16 tile whose first row is `row0` of a [nrows][128]
// matrix into swizzled shared memory; rows >= nrows are zero-filled.
template <int NTHREADS>
__device__ __forceinline__ void load_tile64(uint32_t dst, const __nv_bfloat16* src, int row0,
                                            int nrows, int tid) {
#pragma unroll
    for (int it = 0; it < (kM * kRowChunks) / NTHREADS; ++it) {
        int e = it * NTHREADS + tid;
        int r = e / kRowChunks, c = e % kRowChunks;
        bool ok = row0 + r < nrows;
        const __nv_bfloat16* p = src + (size_t)(ok ? row0 + r : 0) * kD + c * 8;
        cp_async16(dst + swz(r, c), p, ok);
    }
}

// Copies ROWS rows (a [ROWS][128] bf16 tile) starting at row `row0` of a
// [nrows][128] matrix into swizzled shared memory; rows >= nrows are
// zero-filled. ROWS * 16 must be a multiple of NTHREADS.
template <int NTHREADS, int ROWS>
__device__ __forceinline__ void load_rows(uint32_t dst, const __nv_bfloat16* src, int row0,
                                          int nrows, int tid) {
    static_assert((ROWS * kRowChunks) % NTHREADS == 0, "tile split");
#pragma unroll
    for (int it = 0; it < (ROWS * kRowChunks) / NTHREADS; ++it) {
        int e = it * NTHREADS + tid;
        int r = e / kRowChunks, c = e % kRowChunks;
        bool ok = row0 + r < nrows;
        const __nv_bfloat16* p = src + (size_t)(ok ? row0 + r : 0) * kD + c * 8;
        cp_async16(dst + swz(r, c), p, ok);
    }
}

// Copies the valid entries of a selected-block list into shared memory.
// Valid: 0 <= t <= qb and strictly ascending; -1 entries are skipped silently;
// anything else is skipped and recorded in the status word. Returns the count.
__device__ __forceinline__ int compact_block_list(const int32_t* list, int n, int topk, int qb, int* out,
                                  int* status) {
    // The whole row is read first, with independent loads (one memory latency
    // per 16 entries), and compacted afterwards.
    for (int j0 = 0; j0 < topk; j0 += 16) {
        int v[16];
#pragma unroll
        for (int k = 0; k < 16; ++k) v[k] = j0 + k < topk ? __ldg(list + j0 + k) : -1;
#pragma unroll
        for (int k = 0; k < 16; ++k)
            if (j0 + k < topk) out[j0 + k] = v[k];
    }
    if (n < 0 || n > topk) {
        set_status(status, PHSA_ERR_DEVICE_INDEX);
        n = n < 0 ? 0 : topk;
    }
    int k = 0, prev = -1;
    for (int j = 0; j < n; ++j) {
        const int t = out[j];
        if (t == -1) continue;
        if (t < 0 || t > qb || t <= prev) {
            set_status(status, PHSA_ERR_DEVICE_INDEX);
            continue;
        }
        out[k++] = t;
        prev = t;
    }
    return k;
}

}  // namespace phsa
