// Layer input path and output gate of Algorithm 4 (Appendix A, Input projections):
// the memory-bound steps around the operator, each one kernel per direction.
//
// Prologue (per (b, t, h), C = 2 dk + dv + 2 E channels ordered [q | k | v | q' | k']):
//   causal depthwise convolution of width K of the projection output, SiLU on q, k, v,
//   softplus on q', k', L2 normalisation of q, k, q', k'; log gates
//   -exp(A_log) softplus(gate_in + gate_bias) and beta = sigmoid(beta_in).
// Output gate (per (b, t, h) over dv): RMSNorm(o) * w_norm * sigmoid(z).
// Sums over tokens in the backward passes (weight and bias gradients) are per-CTA
// partials reduced in a fixed order by a second kernel.
#include <cuda_bf16.h>

#include "common.cuh"
#include "internal.h"

namespace tla {
namespace {

constexpr int kThreads = 256;
constexpr int kFwdTok = 16;    // tokens per CTA of the prologue forward
constexpr int kSeg = 256;      // tokens per CTA of the prologue backward
constexpr int kSub = 8;        // tokens per sub-block of the prologue backward
constexpr int kGateRows = 256; // (token, head) rows per CTA of the output gate

__device__ __forceinline__ float sigm(float x) { return 1.f / (1.f + expf(-x)); }
__device__ __forceinline__ float softplus(float x) { return x > 20.f ? x : log1pf(expf(x)); }

template <typename T> __device__ __forceinline__ float ld(const void* p, size_t i) {
    return to_f(static_cast<const T*>(p)[i]);
}
template <typename T> __device__ __forceinline__ void st(void* p, size_t i, float v) {
    static_cast<T*>(p)[i] = from_f<T>(v);
}

// Channel groups of a head: 0 q, 1 k, 2 v, 3 q', 4 k'.
struct Groups {
    int off[6];
    __device__ __forceinline__ int of(int c) const {
        int g = 0;
#pragma unroll
        for (int i = 1; i < 5; ++i) g += c >= off[i];
        return g;
    }
};
__device__ __forceinline__ Groups groups(int dk, int dv, int E) {
    Groups G;
    G.off[0] = 0; G.off[1] = dk; G.off[2] = 2 * dk; G.off[3] = 2 * dk + dv;
    G.off[4] = 2 * dk + dv + E; G.off[5] = 2 * dk + dv + 2 * E;
    return G;
}
// normalised group index (q, k, q', k' -> 0..3) or -1 for v
__device__ __forceinline__ int norm_slot(int g) { return g < 2 ? g : (g == 2 ? -1 : g - 1); }

template <typename Tin>
__global__ void __launch_bounds__(kThreads)
prologue_fwd_kernel(const tla_prologue_args a) {
    extern __shared__ float sm[];
    const int dk = a.dk, dv = a.dv, E = a.E, K = a.K, T = a.T, H = a.H;
    const int C = 2 * dk + dv + 2 * E;
    const Groups G = groups(dk, dv, E);
    const int t0 = blockIdx.x * kFwdTok, h = blockIdx.y, b = blockIdx.z;
    const int nt = min(kFwdTok, T - t0);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    float* ys = sm;                       // [kFwdTok][C] activations
    float* sc = sm + kFwdTok * C;         // [kFwdTok][4] 1 / norm
    for (int c = tid; c < C; c += kThreads) {
        float w[4];
        for (int j = 0; j < K; ++j) w[j] = a.conv_w[(size_t(h) * C + c) * K + j];
        const int g = G.of(c);
        for (int i = 0; i < nt; ++i) {
            const int t = t0 + i;
            float acc = 0.f;
            for (int j = 0; j < K; ++j) {
                const int ts = t - K + 1 + j;
                if (ts >= 0) acc = fmaf(w[j], ld<Tin>(a.P, tok_idx(b, ts, h, c, T, H, C)), acc);
            }
            ys[i * C + c] = g >= 3 ? softplus(acc) : acc * sigm(acc);
        }
    }
    __syncthreads();
    for (int task = warp; task < nt * 4; task += kThreads / 32) {
        const int i = task >> 2, s = task & 3, g = s < 2 ? s : s + 1;
        float ss = 0.f;
        for (int c = G.off[g] + lane; c < G.off[g + 1]; c += 32) ss = fmaf(ys[i * C + c], ys[i * C + c], ss);
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
        if (lane == 0) sc[i * 4 + s] = rsqrtf(ss + a.eps);
    }
    __syncthreads();
    void* dst[5] = {a.q, a.k, a.v, a.q2, a.k2};
    for (int idx = tid; idx < nt * C; idx += kThreads) {
        const int i = idx / C, c = idx - i * C, g = G.of(c), s = norm_slot(g);
        const int width = G.off[g + 1] - G.off[g];
        const float y = ys[idx] * (s >= 0 ? sc[i * 4 + s] : 1.f);
        st<Tin>(dst[g], tok_idx(b, t0 + i, h, c - G.off[g], T, H, width), y);
    }
    for (int idx = tid; idx < nt * E; idx += kThreads) {
        const int i = idx / E, e = idx - i * E;
        const size_t o = tok_idx(b, t0 + i, h, e, T, H, E);
        a.g[o] = -expf(a.A_log[h * E + e]) * softplus(a.gate_in[o] + a.gate_bias[h * E + e]);
    }
    if (a.beta_in && tid < nt) {
        const size_t o = (size_t(b) * T + t0 + tid) * H + h;
        a.beta[o] = sigm(a.beta_in[o]);
    }
}

struct PrologueGrads {
    const void *dq, *dk, *dv, *dq2, *dk2;
    const float *dg, *dbeta;
    void* dP;
    float *dgate_in, *dbeta_in;
    float* part;   // per CTA: [C*K] conv-weight partials, then [E] gate-bias, [E] A_log partials
};

// One CTA per (segment of kSeg tokens, h, b); sub-blocks of kSub tokens, each recomputing
// the activations of its tokens and of the K-1 tokens after them (the transposed
// convolution of a token reads the K-1 following pre-activation gradients).
template <typename Tin, typename Tg>
__global__ void __launch_bounds__(kThreads)
prologue_bwd_kernel(const tla_prologue_args a, const PrologueGrads gr) {
    extern __shared__ float sm[];
    const int dk = a.dk, dv = a.dv, E = a.E, K = a.K, T = a.T, H = a.H;
    const int C = 2 * dk + dv + 2 * E;
    const Groups G = groups(dk, dv, E);
    const int seg = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    constexpr int NE = kSub + 3;            // sub-block tokens + up to K - 1 = 3 after them
    float* ys = sm;                         // [NE][C] activations (then scaled: u = y / n)
    float* das = ys + NE * C;               // [NE][C] pre-activation gradients
    float* inv = das + NE * C;              // [NE][4] 1 / n
    float* udy = inv + NE * 4;              // [NE][4] u . dy
    void* gsrc[5];
    gsrc[0] = const_cast<void*>(gr.dq); gsrc[1] = const_cast<void*>(gr.dk);
    gsrc[2] = const_cast<void*>(gr.dv); gsrc[3] = const_cast<void*>(gr.dq2);
    gsrc[4] = const_cast<void*>(gr.dk2);
    // per-thread partial sums of the conv-weight gradient (channels tid, tid + 256)
    float dwp[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
    float gbp = 0.f, gap = 0.f;              // gate-bias and A_log partials (threads < E)
    const int tbeg = seg * kSeg, tend = min(T, tbeg + kSeg);
    for (int t0 = tbeg; t0 < tend; t0 += kSub) {
        const int nt = min(kSub, tend - t0);
        const int ne = min(nt + K - 1, T - t0);   // tokens whose gradients this block needs
        // pre-activations and activations of tokens t0 .. t0 + ne - 1
        for (int idx = tid; idx < ne * C; idx += kThreads) {
            const int i = idx / C, c = idx - i * C, t = t0 + i;
            float acc = 0.f;
            for (int j = 0; j < K; ++j) {
                const int ts = t - K + 1 + j;
                if (ts >= 0)
                    acc = fmaf(a.conv_w[(size_t(h) * C + c) * K + j],
                               ld<Tin>(a.P, tok_idx(b, ts, h, c, T, H, C)), acc);
            }
            das[idx] = acc;   // pre-activation, replaced by its gradient below
            ys[idx] = G.of(c) >= 3 ? softplus(acc) : acc * sigm(acc);
        }
        __syncthreads();
        for (int task = warp; task < ne * 4; task += kThreads / 32) {   // norms and u . dy
            const int i = task >> 2, s = task & 3, g = s < 2 ? s : s + 1;
            const int width = G.off[g + 1] - G.off[g];
            float ss = 0.f, yd = 0.f;
            for (int c = G.off[g] + lane; c < G.off[g + 1]; c += 32) {
                const float y = ys[i * C + c];
                ss = fmaf(y, y, ss);
                yd = fmaf(y, ld<Tg>(gsrc[g], tok_idx(b, t0 + i, h, c - G.off[g], T, H, width)), yd);
            }
#pragma unroll
            for (int o = 16; o >= 1; o >>= 1) {
                ss += __shfl_xor_sync(0xffffffffu, ss, o);
                yd += __shfl_xor_sync(0xffffffffu, yd, o);
            }
            if (lane == 0) {
                const float r = rsqrtf(ss + a.eps);
                inv[i * 4 + s] = r;
                udy[i * 4 + s] = yd * r;
            }
        }
        __syncthreads();
        for (int idx = tid; idx < ne * C; idx += kThreads) {   // pre-activation gradients
            const int i = idx / C, c = idx - i * C, g = G.of(c), s = norm_slot(g);
            const int width = G.off[g + 1] - G.off[g];
            const float dy = ld<Tg>(gsrc[g], tok_idx(b, t0 + i, h, c - G.off[g], T, H, width));
            float dx = dy;
            if (s >= 0) {   // d(y / n) = (dy - u (u . dy)) / n
                const float r = inv[i * 4 + s];
                dx = (dy - ys[idx] * r * udy[i * 4 + s]) * r;
            }
            const float x = das[idx], sg = sigm(x);
            das[idx] = dx * (g >= 3 ? sg : sg * (1.f + x * (1.f - sg)));
        }
        __syncthreads();
        // dP of the block's own tokens (transposed convolution) and conv-weight partials
        for (int cc = 0; cc < 2; ++cc) {
            const int c = tid + cc * kThreads;
            if (c >= C) break;
            float w[4];
            for (int j = 0; j < K; ++j) w[j] = a.conv_w[(size_t(h) * C + c) * K + j];
            for (int i = 0; i < nt; ++i) {
                const int t = t0 + i;
                float acc = 0.f;
                for (int j = 0; j < K; ++j) {
                    const int td = i + K - 1 - j;   // token t + K - 1 - j, local index
                    if (t + K - 1 - j < T) acc = fmaf(w[j], das[td * C + c], acc);
                }
                st<Tin>(gr.dP, tok_idx(b, t, h, c, T, H, C), acc);
                const float dai = das[i * C + c];
                for (int j = 0; j < K; ++j) {
                    const int ts = t - K + 1 + j;
                    if (ts >= 0) dwp[cc][j] = fmaf(dai, ld<Tin>(a.P, tok_idx(b, ts, h, c, T, H, C)), dwp[cc][j]);
                }
            }
        }
        // gates and beta of the block's own tokens
        if (tid < E) {
            const int e = tid;
            const float sA = -expf(a.A_log[h * E + e]);
            for (int i = 0; i < nt; ++i) {
                const size_t o = tok_idx(b, t0 + i, h, e, T, H, E);
                const float z = a.gate_in[o] + a.gate_bias[h * E + e];
                const float dz = gr.dg[o] * sA * sigm(z);
                gr.dgate_in[o] = dz;
                gbp += dz;
                gap = fmaf(gr.dg[o], sA * softplus(z), gap);
            }
        }
        if (a.beta_in && tid >= 64 && tid < 64 + nt) {
            const size_t o = (size_t(b) * T + t0 + tid - 64) * H + h;
            const float s = sigm(a.beta_in[o]);
            gr.dbeta_in[o] = gr.dbeta[o] * s * (1.f - s);
        }
        __syncthreads();
    }
    float* part = gr.part + ((size_t(b) * gridDim.x + seg) * H + h) * (size_t(C) * K + 2 * E);
    for (int cc = 0; cc < 2; ++cc) {
        const int c = tid + cc * kThreads;
        if (c < C)
            for (int j = 0; j < K; ++j) part[c * K + j] = dwp[cc][j];
    }
    if (tid < E) {
        part[C * K + tid] = gbp;
        part[C * K + E + tid] = gap;
    }
}

// Fixed-order sums of the per-CTA partials: out[h][x] = sum_{b, seg} part[b][seg][h][x].
__global__ void reduce_partials_kernel(const float* __restrict__ part, int nblk, int H, int W,
                                       float* __restrict__ dconv_w, float* __restrict__ dbias,
                                       float* __restrict__ dA, int CK, int E) {
    const int idx = blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= H * W) return;
    const int h = idx / W, x = idx - h * W;
    float acc = 0.f;
    for (int n = 0; n < nblk; ++n) acc += part[(size_t(n) * H + h) * W + x];
    if (x < CK) dconv_w[size_t(h) * CK + x] = acc;
    else if (x < CK + E) dbias[h * E + x - CK] = acc;
    else dA[h * E + x - CK - E] = acc;
}

// Output gate: one warp per (token, head) row, kGateRows rows per CTA.
template <typename To, typename Tz>
__global__ void __launch_bounds__(kThreads)
gate_fwd_kernel(const tla_gate_args a, long long rows) {
    const int dv = a.dv, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (long long r = blockIdx.x * (long long)kGateRows + warp; r < min(rows, (blockIdx.x + 1LL) * kGateRows);
         r += kThreads / 32) {
        const size_t base = size_t(r) * dv;
        float ss = 0.f;
        for (int c = lane; c < dv; c += 32) {
            const float x = ld<To>(a.o, base + c);
            ss = fmaf(x, x, ss);
        }
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
        const float rr = rsqrtf(ss / dv + a.eps);
        for (int c = lane; c < dv; c += 32)
            st<Tz>(a.y, base + c, ld<To>(a.o, base + c) * rr * a.w_norm[c] * sigm(ld<Tz>(a.z, base + c)));
    }
}

template <typename To, typename Tz>
__global__ void __launch_bounds__(kThreads)
gate_bwd_kernel(const tla_gate_args a, long long rows, const void* dy, void* d_o, void* dz,
                float* part) {
    extern __shared__ float sm[];   // [kThreads / 32][dv] dw_norm partials per warp
    const int dv = a.dv, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    float* wp = sm + warp * dv;
    for (int c = lane; c < dv; c += 32) wp[c] = 0.f;
    for (long long r = blockIdx.x * (long long)kGateRows + warp; r < min(rows, (blockIdx.x + 1LL) * kGateRows);
         r += kThreads / 32) {
        const size_t base = size_t(r) * dv;
        float ss = 0.f;
        for (int c = lane; c < dv; c += 32) {
            const float x = ld<To>(a.o, base + c);
            ss = fmaf(x, x, ss);
        }
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
        const float rr = rsqrtf(ss / dv + a.eps);
        float dot = 0.f;
        for (int c = lane; c < dv; c += 32) {
            const float nh = ld<To>(a.o, base + c) * rr, s = sigm(ld<Tz>(a.z, base + c));
            const float g = ld<Tz>(dy, base + c);
            const float dnh = g * a.w_norm[c] * s;
            st<Tz>(dz, base + c, g * nh * a.w_norm[c] * s * (1.f - s));
            wp[c] = fmaf(g * s, nh, wp[c]);
            dot = fmaf(dnh, nh, dot);
        }
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, o);
        for (int c = lane; c < dv; c += 32) {
            const float nh = ld<To>(a.o, base + c) * rr, s = sigm(ld<Tz>(a.z, base + c));
            const float dnh = ld<Tz>(dy, base + c) * a.w_norm[c] * s;
            st<To>(d_o, base + c, rr * (dnh - nh * dot / dv));
        }
    }
    __syncthreads();
    for (int c = threadIdx.x; c < dv; c += kThreads) {
        float acc = 0.f;
        for (int w = 0; w < kThreads / 32; ++w) acc += sm[w * dv + c];
        part[size_t(blockIdx.x) * dv + c] = acc;
    }
}

__global__ void reduce_columns_kernel(const float* __restrict__ part, int nblk, int n,
                                      float* __restrict__ out) {
    const int c = blockIdx.x * blockDim.x + threadIdx.x;
    if (c >= n) return;
    float acc = 0.f;
    for (int i = 0; i < nblk; ++i) acc += part[size_t(i) * n + c];
    out[c] = acc;
}

bool al16(const void* p) { return ((uintptr_t)p & 15) == 0; }
bool dim_ok(int d) { return d >= 16 && d <= 128 && d % 16 == 0; }

tla_status check_prologue(const tla_prologue_args* a) {
    if (!a) return TLA_ERR_INVALID_ARG;
    if (a->B < 1 || a->T < 1 || a->H < 1 || a->E < 1 || a->K < 1) return TLA_ERR_INVALID_ARG;
    if (a->dtype != TLA_BF16 && a->dtype != TLA_FP32) return TLA_ERR_INVALID_ARG;
    if (!a->P || !a->conv_w || !a->gate_in || !a->gate_bias || !a->A_log || !a->q || !a->k ||
        !a->v || !a->q2 || !a->k2 || !a->g)
        return TLA_ERR_INVALID_ARG;
    if ((a->beta_in != nullptr) != (a->beta != nullptr)) return TLA_ERR_INVALID_ARG;
    if (!(a->eps > 0.f)) return TLA_ERR_INVALID_ARG;
    if (!dim_ok(a->dk) || !dim_ok(a->dv) || a->E > 32 || a->K > 4) return TLA_ERR_UNSUPPORTED;
    if ((long long)a->B * a->H > 65535) return TLA_ERR_UNSUPPORTED;
    const void* ptrs[] = {a->P, a->conv_w, a->gate_in, a->gate_bias, a->A_log, a->beta_in,
                          a->q, a->k, a->v, a->q2, a->k2, a->g, a->beta};
    for (const void* p : ptrs)
        if (!al16(p)) return TLA_ERR_INVALID_ARG;
    return TLA_OK;
}

tla_status check_gate(const tla_gate_args* a) {
    if (!a) return TLA_ERR_INVALID_ARG;
    if (a->B < 1 || a->T < 1 || a->H < 1) return TLA_ERR_INVALID_ARG;
    if ((a->dtype != TLA_BF16 && a->dtype != TLA_FP32) ||
        (a->o_dtype != TLA_BF16 && a->o_dtype != TLA_FP32))
        return TLA_ERR_INVALID_ARG;
    if (!a->o || !a->z || !a->w_norm || !a->y || !(a->eps > 0.f)) return TLA_ERR_INVALID_ARG;
    if (!dim_ok(a->dv)) return TLA_ERR_UNSUPPORTED;
    const void* ptrs[] = {a->o, a->z, a->w_norm, a->y};
    for (const void* p : ptrs)
        if (!al16(p)) return TLA_ERR_INVALID_ARG;
    return TLA_OK;
}

int n_segments(const tla_prologue_args* a) { return (a->T + kSeg - 1) / kSeg; }
long long gate_blocks(const tla_gate_args* a) {
    return ((long long)a->B * a->T * a->H + kGateRows - 1) / kGateRows;
}
size_t prologue_part_bytes(const tla_prologue_args* a) {
    const int C = 2 * a->dk + a->dv + 2 * a->E;
    return (size_t)a->B * n_segments(a) * a->H * ((size_t)C * a->K + 2 * a->E) * sizeof(float);
}

tla_status cuda_status(cudaError_t e) { return e == cudaSuccess ? TLA_OK : TLA_ERR_CUDA; }

}  // namespace
}  // namespace tla

using namespace tla;

extern "C" tla_status tla_layer_prologue(const tla_prologue_args* a, void* stream) {
    const tla_status st0 = check_prologue(a);
    if (st0 != TLA_OK) return st0;
    cudaStream_t s = (cudaStream_t)stream;
    const int C = 2 * a->dk + a->dv + 2 * a->E;
    const size_t smem = (size_t(kFwdTok) * C + kFwdTok * 4) * sizeof(float);
    dim3 grid((a->T + kFwdTok - 1) / kFwdTok, a->H, a->B);
    prof_before("layer_prologue", s);
    if (a->dtype == TLA_BF16) prologue_fwd_kernel<__nv_bfloat16><<<grid, kThreads, smem, s>>>(*a);
    else prologue_fwd_kernel<float><<<grid, kThreads, smem, s>>>(*a);
    prof_after(s);
    return cuda_status(cudaGetLastError());
}

extern "C" size_t tla_layer_prologue_bwd_workspace_bytes(const tla_prologue_args* a) {
    if (check_prologue(a) != TLA_OK) return 0;
    return (prologue_part_bytes(a) + 255) & ~size_t(255);
}

extern "C" tla_status tla_layer_prologue_bwd(const tla_prologue_args* a, int grad_dtype,
                                             const void* dq, const void* dk, const void* dv,
                                             const void* dq2, const void* dk2, const float* dg,
                                             const float* dbeta, void* dP, float* dconv_w,
                                             float* dgate_in, float* dgate_bias, float* dA_log,
                                             float* dbeta_in, void* workspace,
                                             size_t workspace_bytes, void* stream) {
    const tla_status st0 = check_prologue(a);
    if (st0 != TLA_OK) return st0;
    if (grad_dtype != TLA_BF16 && grad_dtype != TLA_FP32) return TLA_ERR_INVALID_ARG;
    if (!dq || !dk || !dv || !dq2 || !dk2 || !dg || !dP || !dconv_w || !dgate_in ||
        !dgate_bias || !dA_log)
        return TLA_ERR_INVALID_ARG;
    if ((a->beta_in != nullptr) != (dbeta != nullptr) || (dbeta != nullptr) != (dbeta_in != nullptr))
        return TLA_ERR_INVALID_ARG;
    {
        const void* ptrs[] = {dq, dk, dv, dq2, dk2, dg, dbeta, dP, dconv_w, dgate_in, dgate_bias,
                              dA_log, dbeta_in, workspace};
        for (const void* p : ptrs)
            if (!al16(p)) return TLA_ERR_INVALID_ARG;
    }
    if (!workspace || workspace_bytes < prologue_part_bytes(a)) return TLA_ERR_WORKSPACE;
    cudaStream_t s = (cudaStream_t)stream;
    const int C = 2 * a->dk + a->dv + 2 * a->E;
    PrologueGrads gr{dq, dk, dv, dq2, dk2, dg, dbeta, dP, dgate_in, dbeta_in, (float*)workspace};
    const size_t smem = (2 * size_t(kSub + 3) * C + 8 * (kSub + 3)) * sizeof(float);
    dim3 grid(n_segments(a), a->H, a->B);
    prof_before("layer_prologue_bwd", s);
    if (a->dtype == TLA_BF16) {
        if (grad_dtype == TLA_BF16)
            prologue_bwd_kernel<__nv_bfloat16, __nv_bfloat16><<<grid, kThreads, smem, s>>>(*a, gr);
        else
            prologue_bwd_kernel<__nv_bfloat16, float><<<grid, kThreads, smem, s>>>(*a, gr);
    } else {
        if (grad_dtype == TLA_BF16)
            prologue_bwd_kernel<float, __nv_bfloat16><<<grid, kThreads, smem, s>>>(*a, gr);
        else
            prologue_bwd_kernel<float, float><<<grid, kThreads, smem, s>>>(*a, gr);
    }
    prof_after(s);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return TLA_ERR_CUDA;
    const int W = C * a->K + 2 * a->E;
    const int n = a->H * W;
    prof_before("layer_prologue_reduce", s);
    reduce_partials_kernel<<<(n + 255) / 256, 256, 0, s>>>((const float*)workspace,
                                                           a->B * n_segments(a), a->H, W, dconv_w,
                                                           dgate_bias, dA_log, C * a->K, a->E);
    prof_after(s);
    return cuda_status(cudaGetLastError());
}

extern "C" tla_status tla_output_gate(const tla_gate_args* a, void* stream) {
    const tla_status st0 = check_gate(a);
    if (st0 != TLA_OK) return st0;
    cudaStream_t s = (cudaStream_t)stream;
    const long long rows = (long long)a->B * a->T * a->H;
    const unsigned blocks = (unsigned)gate_blocks(a);
    prof_before("output_gate", s);
    if (a->o_dtype == TLA_FP32) {
        if (a->dtype == TLA_FP32) gate_fwd_kernel<float, float><<<blocks, kThreads, 0, s>>>(*a, rows);
        else gate_fwd_kernel<float, __nv_bfloat16><<<blocks, kThreads, 0, s>>>(*a, rows);
    } else {
        if (a->dtype == TLA_FP32) gate_fwd_kernel<__nv_bfloat16, float><<<blocks, kThreads, 0, s>>>(*a, rows);
        else gate_fwd_kernel<__nv_bfloat16, __nv_bfloat16><<<blocks, kThreads, 0, s>>>(*a, rows);
    }
    prof_after(s);
    return cuda_status(cudaGetLastError());
}

extern "C" size_t tla_output_gate_bwd_workspace_bytes(const tla_gate_args* a) {
    if (check_gate(a) != TLA_OK) return 0;
    return ((size_t)gate_blocks(a) * a->dv * sizeof(float) + 255) & ~size_t(255);
}

extern "C" tla_status tla_output_gate_bwd(const tla_gate_args* a, const void* dy, void* d_o,
                                          void* dz, float* dw_norm, void* workspace,
                                          size_t workspace_bytes, void* stream) {
    const tla_status st0 = check_gate(a);
    if (st0 != TLA_OK) return st0;
    if (!dy || !d_o || !dz || !dw_norm) return TLA_ERR_INVALID_ARG;
    {
        const void* ptrs[] = {dy, d_o, dz, dw_norm, workspace};
        for (const void* p : ptrs)
            if (!al16(p)) return TLA_ERR_INVALID_ARG;
    }
    const long long nblk = gate_blocks(a);
    if (!workspace || workspace_bytes < (size_t)nblk * a->dv * sizeof(float)) return TLA_ERR_WORKSPACE;
    cudaStream_t s = (cudaStream_t)stream;
    const long long rows = (long long)a->B * a->T * a->H;
    const size_t smem = (kThreads / 32) * a->dv * sizeof(float);
    float* part = (float*)workspace;
    prof_before("output_gate_bwd", s);
    if (a->o_dtype == TLA_FP32) {
        if (a->dtype == TLA_FP32)
            gate_bwd_kernel<float, float><<<(unsigned)nblk, kThreads, smem, s>>>(*a, rows, dy, d_o, dz, part);
        else
            gate_bwd_kernel<float, __nv_bfloat16><<<(unsigned)nblk, kThreads, smem, s>>>(*a, rows, dy, d_o, dz, part);
    } else {
        if (a->dtype == TLA_FP32)
            gate_bwd_kernel<__nv_bfloat16, float><<<(unsigned)nblk, kThreads, smem, s>>>(*a, rows, dy, d_o, dz, part);
        else
            gate_bwd_kernel<__nv_bfloat16, __nv_bfloat16><<<(unsigned)nblk, kThreads, smem, s>>>(*a, rows, dy, d_o, dz, part);
    }
    prof_after(s);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return TLA_ERR_CUDA;
    prof_before("output_gate_reduce", s);
    reduce_columns_kernel<<<(a->dv + 127) / 128, 128, 0, s>>>(part, (int)nblk, a->dv, dw_norm);
    prof_after(s);
    return cuda_status(cudaGetLastError());
}
