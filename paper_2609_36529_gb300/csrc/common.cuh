// Shared device helpers of the CUDA library (not used by the oracle).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/tla.h"

namespace tla {

constexpr int kChunk = 64;  // C of Appendix A

__device__ __forceinline__ float to_f(float x) { return x; }
__device__ __forceinline__ float to_f(__nv_bfloat16 x) { return __bfloat162float(x); }

template <typename T> __device__ __forceinline__ T from_f(float x);
template <> __device__ __forceinline__ float from_f<float>(float x) { return x; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f<__nv_bfloat16>(float x) {
    return __float2bfloat16_rn(x);
}

// Store one result element in the requested output type (fp32 or bf16).
__device__ __forceinline__ void store_out(void* base, size_t i, float v, int out_f32) {
    if (out_f32) static_cast<float*>(base)[i] = v;
    else static_cast<__nv_bfloat16*>(base)[i] = __float2bfloat16_rn(v);
}

// Index of element i of token (b,t,h) in a [B,T,H,D] tensor.
__device__ __forceinline__ size_t tok_idx(int b, int t, int h, int i, int T, int H, int D) {
    return ((size_t(b) * T + t) * H + h) * D + i;
}

// Kernels with bounded waits receive a pointer to the library's device error
// word (owned by tla_api.cu) and record the first failure there.
__device__ __forceinline__ void record_device_error(int* err, int code) {
    if (err) atomicCAS(err, 0, code);
}

}  // namespace tla
