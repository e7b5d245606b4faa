// Activation functions of the layer's input path (Algorithm 2), shared by the
// elementwise prologue kernels and the fused projection GEMM epilogue.
#pragma once

namespace tla {

__device__ __forceinline__ float sigm(float x) { return __fdividef(1.f, 1.f + __expf(-x)); }
// softplus(x) = log(1 + e^x) = max(x, 0) + log(1 + e^-|x|) with fast intrinsics; for
// e^-|x| < 2^-10 the series e (1 - e/2) keeps the relative accuracy that log(1 + e) in fp32
// would lose.  Selects rather than branches, so that unrolled callers interleave elements.
__device__ __forceinline__ float softplus(float x) {
    const float e = __expf(-fabsf(x));
    const float l = e < 0.0009765625f ? e * fmaf(-0.5f, e, 1.f) : __logf(1.f + e);
    return fmaxf(x, 0.f) + l;
}

}  // namespace tla
