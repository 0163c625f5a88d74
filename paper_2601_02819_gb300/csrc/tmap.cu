// Host-side TMA tensor maps. The driver's cuTensorMapEncodeTiled is fetched
// once through the runtime's driver entry-point query, so the library needs
// no link-time dependency on libcuda.
#include <cuda.h>
#include <cuda_runtime.h>

#include <mutex>

#include "phsa_internal.h"

namespace phsa {

namespace {

using EncodeTiled = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                 const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                 const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                 CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiled encode_fn() {
    static EncodeTiled fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiled>(p);
    });
    return fn;
}

}  // namespace

// A 3-D bf16 view [planes][rows][128] of a row-major tensor, read or written
// in boxes of {64 columns, box_rows rows, box_planes planes} with the 128-byte
// swizzle (a box lands as box_planes consecutive [box_rows][64] tiles). Rows
// past `rows` (inside a plane) read as zero and are not written.
bool make_tmap_bf16_rows128(CUtensorMap* map, const void* base, uint64_t rows, uint64_t planes,
                            uint32_t box_rows, uint32_t box_planes) {
    EncodeTiled fn = encode_fn();
    if (!fn || !base || rows == 0 || planes == 0) return false;
    const cuuint64_t dims[3] = {128, rows, planes};
    const cuuint64_t strides[2] = {128 * 2, rows * 128 * 2};
    const cuuint32_t box[3] = {64, box_rows, box_planes};
    const cuuint32_t estr[3] = {1, 1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides,
              box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace phsa
