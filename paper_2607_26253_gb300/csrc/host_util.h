// Host helpers: error type carried to the C ABI, CUDA status checks, TMA descriptors.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>

#include <stdexcept>
#include <string>

#include "../../include/sara.h"

namespace sara {

struct SaraError : std::runtime_error {
    int code;
    SaraError(int c, const std::string &m) : std::runtime_error(m), code(c) {}
};

inline void check_cuda(cudaError_t e, const char *what, const char *file, int line) {
    if (e != cudaSuccess) {
        throw SaraError(e == cudaErrorMemoryAllocation ? SARA_ENOMEM : SARA_EDEVICE,
                        std::string(what) + " failed: " + cudaGetErrorString(e) + " (" + file + ":" +
                            std::to_string(line) + ")");
    }
}
#define CK(x) ::sara::check_cuda((x), #x, __FILE__, __LINE__)

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

inline EncodeTiledFn encode_tiled_fn() {
    static EncodeTiledFn fn = nullptr;
    if (!fn) {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        CK(cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q));
        if (q != cudaDriverEntryPointSuccess || !p) throw SaraError(SARA_EDEVICE, "cuTensorMapEncodeTiled is unavailable");
        fn = reinterpret_cast<EncodeTiledFn>(p);
    }
    return fn;
}

// Row-major bf16 matrix [outer][inner] -> 2-D tensor map with box {box_inner, box_outer} and
// 128-byte swizzle (box_inner * 2 bytes must be 128).  Out-of-range rows read as zero.
inline CUtensorMap make_tmap_bf16(const void *base, int inner, int outer, int box_inner, int box_outer) {
    CUtensorMap tm;
    const cuuint64_t dims[2] = {(cuuint64_t)inner, (cuuint64_t)outer};
    const cuuint64_t strides[1] = {(cuuint64_t)inner * 2};
    const cuuint32_t box[2] = {(cuuint32_t)box_inner, (cuuint32_t)box_outer};
    const cuuint32_t estr[2] = {1, 1};
    const CUresult r = encode_tiled_fn()(&tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides,
                                         box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                                         CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) throw SaraError(SARA_EINVAL, "cuTensorMapEncodeTiled failed (" + std::to_string((int)r) + ")");
    return tm;
}

}  // namespace sara
