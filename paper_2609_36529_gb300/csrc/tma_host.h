// Host-side creation of TMA tensor maps (cuTensorMapEncodeTiled through the
// runtime's driver entry point, so the library needs no link-time libcuda).
#pragma once

#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace tla {

inline PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        cudaDriverEntryPointQueryResult q;
        void* p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    }
    return fn;
}

// Token tensor [B, T, H, D] of bf16 (elem_bytes 2) or fp32 (4) viewed as 4-D (D, H, T, B);
// box (box_d, 1, box_t, 1).  Loads read rows past T as zero, stores skip them.  swizzle128:
// 128-byte swizzle (box_d * elem_bytes must be 128).
inline bool make_token_map(CUtensorMap* m, const void* base, int B, int T, int H, int D, int box_d,
                           int box_t, bool swizzle128, int elem_bytes = 2) {
    auto enc = tensor_map_encoder();
    if (!enc) return false;
    cuuint64_t dims[4] = {(cuuint64_t)D, (cuuint64_t)H, (cuuint64_t)T, (cuuint64_t)B};
    const cuuint64_t eb = (cuuint64_t)elem_bytes;
    cuuint64_t strides[3] = {(cuuint64_t)D * eb, (cuuint64_t)H * D * eb, (cuuint64_t)T * H * D * eb};
    cuuint32_t box[4] = {(cuuint32_t)box_d, 1, (cuuint32_t)box_t, 1};
    cuuint32_t es[4] = {1, 1, 1, 1};
    CUresult r = enc(m, elem_bytes == 4 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16,
                     4, const_cast<void*>(base), dims, strides,
                     box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                     swizzle128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

// Token tensor as above (bf16), box (box_d, 1, box_t, 1), the shared-memory side swizzled by
// swizzle_bytes = 2 * box_d (32, 64 or 128): the rows land as the MN-major operand layout of a
// [box_t][box_d] block (tc_common.cuh: blk_offset).
inline bool make_token_map_sw(CUtensorMap* m, const void* base, int B, int T, int H, int D,
                              int box_d, int box_t) {
    auto enc = tensor_map_encoder();
    if (!enc) return false;
    const int sw = 2 * box_d;
    if (sw != 32 && sw != 64 && sw != 128) return false;
    cuuint64_t dims[4] = {(cuuint64_t)D, (cuuint64_t)H, (cuuint64_t)T, (cuuint64_t)B};
    cuuint64_t strides[3] = {(cuuint64_t)D * 2, (cuuint64_t)H * D * 2, (cuuint64_t)T * H * D * 2};
    cuuint32_t box[4] = {(cuuint32_t)box_d, 1, (cuuint32_t)box_t, 1};
    cuuint32_t es[4] = {1, 1, 1, 1};
    CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides,
                     box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                     sw == 32 ? CU_TENSOR_MAP_SWIZZLE_32B
                     : sw == 64 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

// bf16 row-major matrix [rows][cols] as 2-D (cols, rows); box (box_c, box_r); shared-memory
// side swizzled by swizzle_bytes (32, 64 or 128; box_c * 2 must not exceed it).
inline bool make_matrix_map(CUtensorMap* m, const void* base, long long rows, int cols, int box_c,
                            int box_r, int swizzle_bytes = 128) {
    auto enc = tensor_map_encoder();
    if (!enc) return false;
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
    cuuint32_t box[2] = {(cuuint32_t)box_c, (cuuint32_t)box_r};
    cuuint32_t es[2] = {1, 1};
    CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                     box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                     swizzle_bytes == 32   ? CU_TENSOR_MAP_SWIZZLE_32B
                     : swizzle_bytes == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
                                           : CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

// State checkpoints of the tensor-core path: per slab s = ((b * H + h) * NT + chunk) * E + e
// a row-major [128][dv] bf16 hi matrix then the lo matrix.  Viewed as 4-D (column, row,
// slab, hi/lo) with the hi/lo stride inside the slab stride, a box of (box_c, 128, box_s, 2)
// lands in shared memory as [hi/lo][box_s][128][box_c]: the hi blocks of box_s slabs, then
// their lo blocks.  swizzle_bytes: the shared-memory swizzle (box_c * 2 bytes wide).
inline bool make_ckpt_map(CUtensorMap* m, const void* base, long long nslab, int dv, int box_c,
                          int box_s, int swizzle_bytes) {
    auto enc = tensor_map_encoder();
    if (!enc) return false;
    cuuint64_t dims[4] = {(cuuint64_t)dv, 128, (cuuint64_t)nslab, 2};
    cuuint64_t strides[3] = {(cuuint64_t)dv * 2, (cuuint64_t)dv * 2 * 256, (cuuint64_t)dv * 2 * 128};
    cuuint32_t box[4] = {(cuuint32_t)box_c, 128, (cuuint32_t)box_s, 2};
    cuuint32_t es[4] = {1, 1, 1, 1};
    CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides,
                     box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                     swizzle_bytes == 32   ? CU_TENSOR_MAP_SWIZZLE_32B
                     : swizzle_bytes == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
                                           : CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

}  // namespace tla
