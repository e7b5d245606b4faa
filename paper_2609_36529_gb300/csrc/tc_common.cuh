// Device helpers shared by the tensor-core kernels (row stores, split-bf16 stores).
#pragma once

#include <cuda_bf16.h>
#include <stdint.h>

#include "sm100.cuh"

namespace tla {

__device__ __forceinline__ void store_row(void* base, size_t off, const float* v, int n,
                                          int out_f32) {
    if (out_f32) {
        float4* d = reinterpret_cast<float4*>(static_cast<float*>(base) + off);
        for (int i = 0; i < n / 4; ++i) d[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
    } else {
        uint4* d = reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(base) + off);
        for (int i = 0; i < n / 8; ++i) {
            uint32_t u[4];
            for (int j = 0; j < 4; ++j) {
                __nv_bfloat162 pr = __floats2bfloat162_rn(v[8 * i + 2 * j], v[8 * i + 2 * j + 1]);
                u[j] = *reinterpret_cast<uint32_t*>(&pr);
            }
            d[i] = make_uint4(u[0], u[1], u[2], u[3]);
        }
    }
}

__device__ __forceinline__ void store_f32_row(float* dst, const float* v, int n) {
    float4* d = reinterpret_cast<float4*>(dst);
    for (int i = 0; i < n / 4; ++i) d[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
}

// Store v as a bf16 pair: hi = bf16(v) into tile_hi, lo = bf16(v - hi) into tile_lo.
__device__ __forceinline__ void st_split(uint8_t* tile_hi, uint8_t* tile_lo, uint32_t off, float v) {
    const __nv_bfloat16 hi = __float2bfloat16_rn(v);
    *reinterpret_cast<__nv_bfloat16*>(tile_hi + off) = hi;
    *reinterpret_cast<__nv_bfloat16*>(tile_lo + off) = __float2bfloat16_rn(v - __bfloat162float(hi));
}


// State operand blocks.  For a block of TV value columns, each slice e of the state
// (or of its gradient) is a [128 rows][TV] bf16 block of 256 * TV bytes whose rows
// are 2 * TV bytes wide, with the tensor cores' swizzle of that width (16-byte chunks
// XOR-ed with the row's position in its 8-row group: 32-, 64- or 128-byte swizzle for
// TV = 16, 32, 64), which is also the shared-memory layout of a TMA box of TV columns
// with that swizzle.  The recurrences use the blocks of all slices as the MN-major
// operand [dk][E * TV] (one swizzle atom of TV columns per slice) and store each
// block by TMA into the row-major checkpoint of its value columns.
template <int TV>
__host__ __device__ __forceinline__ uint32_t blk_offset(int row, int col) {
    const uint32_t o = uint32_t(row) * (2 * TV) + uint32_t(col) * 2;
    return o ^ (((o >> 7) & (TV / 8 - 1)) << 4);
}
template <int TV>
__host__ __device__ constexpr uint32_t blk_bytes() { return 256u * TV; }

// Token tile of one chunk: 64 rows x dv as bf16 hi (64*dv*2 bytes) then bf16 lo, each in
// SW128 K-major 64-row blocks of 64 columns -- the operand layout of the chunk-gradient
// kernel, which copies a tile into shared memory as is.  Writes columns n0..n0+cnt of row r
// (zeros when !valid, so that padded rows of the last chunk read as zero).
__device__ __forceinline__ void store_tok_tile(float* base, size_t chunk, int dv, int r, int n0,
                                               const float* v, int cnt, bool valid) {
    uint8_t* hi = reinterpret_cast<uint8_t*>(base) + chunk * (size_t(64) * dv * 4);
    uint8_t* lo = hi + size_t(64) * dv * 2;
    for (int i = 0; i < cnt; i += 8) {
        float z[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) z[k] = valid ? v[i + k] : 0.f;
        sm100::st8_split(hi, lo, sm100::sw128_offset(r, n0 + i, 64), z);
    }
}

}  // namespace tla
