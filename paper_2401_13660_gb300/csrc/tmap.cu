// TMA tensor-map encoding shared by the kernels. cuTensorMapEncodeTiled is
// fetched through the runtime's driver entry point, so the library does not
// link libcuda directly.
#include <cuda.h>
#include <cuda_runtime.h>

#include "internal.h"

namespace mbscan {
namespace {

using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                   const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                   const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = [] {
        void *f = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault,
                                             &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess)
            f = nullptr;
        return reinterpret_cast<EncodeTiledFn>(f);
    }();
    return fn;
}

}  // namespace

bool encode_tmap(CUtensorMap *m, const void *base, int elem_bytes, int rank, const uint64_t *dims,
                 const uint64_t *strides, const uint32_t *box, int swizzle) {
    if (swizzle != 0 && swizzle != 64 && swizzle != 128) return false;
    EncodeTiledFn enc = encode_fn();
    if (!enc || rank < 1 || rank > 5) return false;
    cuuint64_t d[5], st[4];
    cuuint32_t bx[5], es[5];
    for (int i = 0; i < rank; ++i) {
        d[i] = dims[i];
        bx[i] = box[i];
        es[i] = 1;
        if (i + 1 < rank) st[i] = strides[i];
    }
    const CUtensorMapDataType dt = elem_bytes == 2 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16
                                                   : CU_TENSOR_MAP_DATA_TYPE_FLOAT32;
    return enc(m, dt, (cuuint32_t)rank, const_cast<void *>(base), d, st, bx, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE,
               swizzle == 128 ? CU_TENSOR_MAP_SWIZZLE_128B
                              : (swizzle == 64 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_NONE),
               CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace mbscan
