// Layer input path and output gate of Algorithm 2 (Appendix A, Input projections):
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

#include "act.cuh"
#include "common.cuh"
#include "internal.h"
#include "sm100.cuh"

namespace tla {

// Address of the library's device error word on the current device (tla_api.cu): kernels
// with bounded waits record TLA_ERR_TIMEOUT there.
int* device_error_word();

namespace {

constexpr int kThreads = 256;
constexpr int kFwdRun = 128;   // tokens per CTA of the prologue forward
constexpr int kSeg = 256;      // tokens per CTA of the prologue backward
constexpr int kBwdGroup = 2;   // tokens whose row sums the prologue backward reduces together
constexpr int kGateTile = 64;  // (token, head) rows per CTA of the output gate


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

// Four consecutive channels of one token as fp32: one 8-byte (bf16) or 16-byte (fp32)
// access when VEC (rows and channel offsets multiples of four), else four scalar ones.
template <bool VEC>
__device__ __forceinline__ void ld4(const __nv_bfloat16* p, float* v) {
    if constexpr (VEC) {
        const uint2 u = *reinterpret_cast<const uint2*>(p);
        const float2 lo = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.x));
        const float2 hi = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.y));
        v[0] = lo.x; v[1] = lo.y; v[2] = hi.x; v[3] = hi.y;
    } else {
#pragma unroll
        for (int u = 0; u < 4; ++u) v[u] = __bfloat162float(p[u]);
    }
}
template <bool VEC>
__device__ __forceinline__ void ld4(const float* p, float* v) {
    if constexpr (VEC) {
        const float4 f = *reinterpret_cast<const float4*>(p);
        v[0] = f.x; v[1] = f.y; v[2] = f.z; v[3] = f.w;
    } else {
#pragma unroll
        for (int u = 0; u < 4; ++u) v[u] = p[u];
    }
}
template <bool VEC>
__device__ __forceinline__ void st4(__nv_bfloat16* p, const float* v) {
    if constexpr (VEC) {
        __nv_bfloat162 lo = __floats2bfloat162_rn(v[0], v[1]), hi = __floats2bfloat162_rn(v[2], v[3]);
        *reinterpret_cast<uint2*>(p) = make_uint2(*reinterpret_cast<uint32_t*>(&lo), *reinterpret_cast<uint32_t*>(&hi));
    } else {
#pragma unroll
        for (int u = 0; u < 4; ++u) p[u] = __float2bfloat16_rn(v[u]);
    }
}
template <bool VEC>
__device__ __forceinline__ void st4(float* p, const float* v) {
    if constexpr (VEC) {
        *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
    } else {
#pragma unroll
        for (int u = 0; u < 4; ++u) p[u] = v[u];
    }
}

__device__ __forceinline__ float warp_sum(float x) {
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}
// warp_sum of N values at once, their shuffles interleaved (each value summed in warp_sum's order).
template <int N>
__device__ __forceinline__ void warp_sum_n(float (&v)[N]) {
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1)
#pragma unroll
        for (int i = 0; i < N; ++i) v[i] += __shfl_xor_sync(0xffffffffu, v[i], o);
}

// Layout of the prologue kernels: a CTA of four warps takes one run of tokens of one
// (b, h); warp 0 the q channels, warp 1 k, warp 2 v (four channels per lane) and then the
// gates and beta (v needs no norm), warp 3 the q' and k' channels (one or two per lane).  Each norm
// is then a reduction inside one warp, so the warps never wait on one another.  A warp
// walks its run token by token, keeping the last three projection rows (and, backward,
// the last three pre-activation gradients) in registers: the width-K convolution uses
// K <= 4 taps padded on the left to four with zero weights, so every projection row is
// loaded once plus a halo of three tokens per run.  Tokens are taken four at a time, all
// four loads issued before the first use.
constexpr int kPrWarps = 4;

struct ChanMap {   // the channels of one lane of a q, k or v warp
    int base, width, c;
    bool act;
};
__device__ __forceinline__ ChanMap chan_map(int g, int dk, int dv, int lane) {
    ChanMap m;
    m.base = g == 2 ? 2 * dk : g * dk;
    m.width = g == 2 ? dv : dk;
    m.c = m.base + 4 * lane;
    m.act = 4 * lane < m.width;
    return m;
}

template <typename Tin, bool VEC>
__device__ __forceinline__ void prologue_fwd_qkv(const tla_prologue_args& a, int g, int b, int h,
                                                 int t0, int t1) {
    const int lane = threadIdx.x & 31;
    const int dk = a.dk, dv = a.dv, E = a.E, K = a.K, T = a.T, H = a.H;
    const int C = 2 * dk + dv + 2 * E;
    const ChanMap m = chan_map(g, dk, dv, lane);
    float w[4][4];   // [padded tap][channel]
#pragma unroll
    for (int j = 0; j < 4; ++j)
#pragma unroll
        for (int u = 0; u < 4; ++u)
            w[j][u] = (m.act && j >= 4 - K) ? a.conv_w[(size_t(h) * C + m.c + u) * K + j - (4 - K)] : 0.f;
    const size_t sP = size_t(H) * C, sD = size_t(H) * m.width;
    const Tin* pP = static_cast<const Tin*>(a.P) + (size_t(b) * T * H + h) * C + m.c;
    Tin* pD = static_cast<Tin*>(g == 0 ? a.q : g == 1 ? a.k : a.v) + (size_t(b) * T * H + h) * m.width + 4 * lane;
    float pw[3][4];
#pragma unroll
    for (int i = 0; i < 3; ++i) {
        const int t = t0 - 3 + i;
        if (m.act && t >= 0) ld4<VEC>(pP + t * sP, pw[i]);
        else pw[i][0] = pw[i][1] = pw[i][2] = pw[i][3] = 0.f;
    }
    for (int tb = t0; tb < t1; tb += 4) {
        float xb[4][4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            if (m.act && tb + i < t1) ld4<VEC>(pP + (tb + i) * sP, xb[i]);
            else xb[i][0] = xb[i][1] = xb[i][2] = xb[i][3] = 0.f;
        }
        // the four tokens' activations, then their row sums together (interleaved shuffles),
        // then the scaled rows: no branch per token, so that their latencies overlap
        float y[4][4], rs[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            float ss = 0.f;
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                float x = w[0][u] * pw[0][u];
                x = fmaf(w[1][u], pw[1][u], x);
                x = fmaf(w[2][u], pw[2][u], x);
                x = fmaf(w[3][u], xb[i][u], x);
                y[i][u] = x * sigm(x);
                ss = fmaf(y[i][u], y[i][u], ss);
                pw[0][u] = pw[1][u]; pw[1][u] = pw[2][u]; pw[2][u] = xb[i][u];
            }
            rs[i] = ss;
        }
        if (g != 2) {   // q and k are L2-normalised, v is not
            warp_sum_n(rs);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const float r = rsqrtf(rs[i] + a.eps);
#pragma unroll
                for (int u = 0; u < 4; ++u) y[i][u] *= r;
            }
        }
#pragma unroll
        for (int i = 0; i < 4; ++i)
            if (m.act && tb + i < t1) st4<VEC>(pD + (tb + i) * sD, y[i]);
    }
}

template <typename Tin>
__device__ __forceinline__ void prologue_fwd_small(const tla_prologue_args& a, int b, int h,
                                                   int t0, int t1) {
    const int lane = threadIdx.x & 31;
    const int dk = a.dk, dv = a.dv, E = a.E, K = a.K, T = a.T, H = a.H;
    const int C = 2 * dk + dv + 2 * E, off = 2 * dk + dv;
    // channel slots cc = lane, lane + 32 of the 2E channels [q' | k']
    bool act[2];
    int col[2];
    float w[4][2];
#pragma unroll
    for (int s = 0; s < 2; ++s) {
        const int cc = lane + 32 * s;
        act[s] = cc < 2 * E;
        col[s] = cc < E ? cc : cc - E;
#pragma unroll
        for (int j = 0; j < 4; ++j)
            w[j][s] = (act[s] && j >= 4 - K) ? a.conv_w[(size_t(h) * C + off + cc) * K + j - (4 - K)] : 0.f;
    }
    const size_t sP = size_t(H) * C, sE = size_t(H) * E;
    const Tin* pP = static_cast<const Tin*>(a.P) + (size_t(b) * T * H + h) * C + off + lane;
    const size_t rowE = (size_t(b) * T * H + h) * E;
    float pw[3][2];
#pragma unroll
    for (int i = 0; i < 3; ++i)
#pragma unroll
        for (int s = 0; s < 2; ++s) {
            const int t = t0 - 3 + i;
            pw[i][s] = (act[s] && t >= 0) ? to_f(pP[t * sP + 32 * s]) : 0.f;
        }
    for (int tb = t0; tb < t1; tb += 4) {
        float xb[4][2];
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int s = 0; s < 2; ++s)
                xb[i][s] = (act[s] && tb + i < t1) ? to_f(pP[(tb + i) * sP + 32 * s]) : 0.f;
        float y[4][2], rs[8];   // rs: sq, sk of the four tokens, reduced together
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            float sq = 0.f, sk = 0.f;
#pragma unroll
            for (int s = 0; s < 2; ++s) {
                float x = w[0][s] * pw[0][s];
                x = fmaf(w[1][s], pw[1][s], x);
                x = fmaf(w[2][s], pw[2][s], x);
                x = fmaf(w[3][s], xb[i][s], x);
                y[i][s] = act[s] ? softplus(x) : 0.f;
                if (lane + 32 * s < E) sq = fmaf(y[i][s], y[i][s], sq);
                else sk = fmaf(y[i][s], y[i][s], sk);
                pw[0][s] = pw[1][s]; pw[1][s] = pw[2][s]; pw[2][s] = xb[i][s];
            }
            rs[i] = sq;
            rs[4 + i] = sk;
        }
        warp_sum_n(rs);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float rq = rsqrtf(rs[i] + a.eps), rk = rsqrtf(rs[4 + i] + a.eps);
            if (tb + i < t1) {
                const size_t o = rowE + (tb + i) * sE;
#pragma unroll
                for (int s = 0; s < 2; ++s)
                    if (act[s]) {
                        const bool isq = lane + 32 * s < E;
                        st<Tin>(isq ? a.q2 : a.k2, o + col[s], y[i][s] * (isq ? rq : rk));
                    }
            }
        }
    }
}

// Log gates and beta of tokens [t0, t1) of (b, h) (the v warp, whose channels need no norm).
__device__ __forceinline__ void prologue_fwd_gates(const tla_prologue_args& a, int b, int h, int t0,
                                                   int t1) {
    const int lane = threadIdx.x & 31;
    const int E = a.E, T = a.T, H = a.H;
    const size_t sE = size_t(H) * E;
    const size_t rowE = (size_t(b) * T * H + h) * E;
    const int n = t1 - t0;
    for (int i0 = lane; i0 < n * E; i0 += 32 * 4) {   // log gates, four loads ahead
        float z[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int idx = i0 + 32 * u, i = idx / E, e = idx - i * E;
            z[u] = idx < n * E ? a.gate_in[rowE + (t0 + i) * sE + e] + a.gate_bias[h * E + e] : 0.f;
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int idx = i0 + 32 * u, i = idx / E, e = idx - i * E;
            if (idx < n * E) a.g[rowE + (t0 + i) * sE + e] = -__expf(a.A_log[h * E + e]) * softplus(z[u]);
        }
    }
    if (a.beta_in)
        for (int tb = t0 + lane; tb < t1; tb += 32 * 4) {
            float bi[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int t = tb + 32 * u;
                bi[u] = t < t1 ? a.beta_in[(size_t(b) * T + t) * H + h] : 0.f;
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int t = tb + 32 * u;
                if (t < t1) a.beta[(size_t(b) * T + t) * H + h] = sigm(bi[u]);
            }
        }
}

template <typename Tin, bool VEC>
__global__ void __launch_bounds__(kPrWarps * 32)
prologue_fwd_kernel(const tla_prologue_args a) {
    const int t0 = blockIdx.x * kFwdRun, t1 = min(a.T, t0 + kFwdRun);
    const int g = threadIdx.x >> 5, h = blockIdx.y, b = blockIdx.z;
    if (g < 3) prologue_fwd_qkv<Tin, VEC>(a, g, b, h, t0, t1);
    else prologue_fwd_small<Tin>(a, b, h, t0, t1);
    if (g == 2) prologue_fwd_gates(a, b, h, t0, t1);
}

struct PrologueGrads {
    const void *dq, *dk, *dv, *dq2, *dk2;
    const float *dg, *dbeta;
    void* dP;
    float *dgate_in, *dbeta_in;
    float* part;   // per CTA: [C*K] conv-weight partials, then [E] gate-bias, [E] A_log partials
};

// Backward of one q, k or v warp over tokens [t0, t1): the pre-activation gradients of
// tokens t0 .. t1 + 2 (the transposed convolution of token t reads those of t .. t + 3;
// zero past T), dP of the run's own tokens, and the conv-weight sums over them.
template <typename Tin, typename Tg, bool VEC>
__device__ __forceinline__ void prologue_bwd_qkv(const tla_prologue_args& a, const PrologueGrads& gr,
                                                 int g, int b, int h, int t0, int t1, float* part) {
    const int lane = threadIdx.x & 31;
    const int dk = a.dk, dv = a.dv, E = a.E, K = a.K, T = a.T, H = a.H;
    const int C = 2 * dk + dv + 2 * E;
    const ChanMap m = chan_map(g, dk, dv, lane);
    float w[4][4], dw[4][4];
#pragma unroll
    for (int j = 0; j < 4; ++j)
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            w[j][u] = (m.act && j >= 4 - K) ? a.conv_w[(size_t(h) * C + m.c + u) * K + j - (4 - K)] : 0.f;
            dw[j][u] = 0.f;
        }
    const size_t sP = size_t(H) * C, sG = size_t(H) * m.width;
    const size_t rowP = (size_t(b) * T * H + h) * C + m.c;
    const Tin* pP = static_cast<const Tin*>(a.P) + rowP;
    Tin* pdP = static_cast<Tin*>(gr.dP) + rowP;
    const Tg* pG = static_cast<const Tg*>(g == 0 ? gr.dq : g == 1 ? gr.dk : gr.dv) +
                   (size_t(b) * T * H + h) * m.width + 4 * lane;
    float pw[3][4], dxw[3][4];   // projection rows and pre-activation gradients of t-3 .. t-1
#pragma unroll
    for (int i = 0; i < 3; ++i) {
        const int t = t0 - 3 + i;
        if (m.act && t >= 0) ld4<VEC>(pP + t * sP, pw[i]);
        else pw[i][0] = pw[i][1] = pw[i][2] = pw[i][3] = 0.f;
        dxw[i][0] = dxw[i][1] = dxw[i][2] = dxw[i][3] = 0.f;
    }
    const int tl = t1 + 3, tv = min(tl, T), te = min(t1, T);
    const bool nrm = g != 2;   // q and k are L2-normalised, v is not
    for (int tb = t0; tb < tl; tb += 4) {
        // rows t-3 .. t+3 of the batch's four tokens t = tb .. tb+3: win[i .. i+3] are token
        // i's convolution taps
        float win[7][4], gb[4][4];
#pragma unroll
        for (int i = 0; i < 3; ++i)
#pragma unroll
            for (int u = 0; u < 4; ++u) win[i][u] = pw[i][u];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            if (m.act && tb + i < tv) {
                ld4<VEC>(pP + (tb + i) * sP, win[3 + i]);
                ld4<VEC>(pG + (tb + i) * sG, gb[i]);
            } else {
#pragma unroll
                for (int u = 0; u < 4; ++u) win[3 + i][u] = gb[i][u] = 0.f;
            }
        }
        // The tokens are independent up to the weight sums: a group's activations first, then
        // its row sums together (interleaved shuffles), then its gradients; no branch per
        // token, so that their latencies overlap.  Tokens at or past tv give dx = 0.
        float dwin[7][4];   // pre-activation gradients of t-3 .. t+3
#pragma unroll
        for (int i = 0; i < 3; ++i)
#pragma unroll
            for (int u = 0; u < 4; ++u) dwin[i][u] = dxw[i][u];
#pragma unroll
        for (int i0 = 0; i0 < 4; i0 += kBwdGroup) {
            float fd[kBwdGroup][4], y[kBwdGroup][4], rs[2 * kBwdGroup];   // fd = d silu(x) / dx
#pragma unroll
            for (int j = 0; j < kBwdGroup; ++j) {
                const int i = i0 + j;
                float ss = 0.f, yd = 0.f;
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    float v = w[0][u] * win[i][u];
                    v = fmaf(w[1][u], win[i + 1][u], v);
                    v = fmaf(w[2][u], win[i + 2][u], v);
                    v = fmaf(w[3][u], win[i + 3][u], v);
                    const float sgv = sigm(v);
                    y[j][u] = v * sgv;
                    fd[j][u] = sgv * (1.f + v * (1.f - sgv));
                    ss = fmaf(y[j][u], y[j][u], ss);
                    yd = fmaf(y[j][u], gb[i][u], yd);
                }
                rs[j] = ss;
                rs[kBwdGroup + j] = yd;
            }
            if (nrm) warp_sum_n(rs);
#pragma unroll
            for (int j = 0; j < kBwdGroup; ++j) {
                const int i = i0 + j, t = tb + i;
                float dy[4] = {gb[i][0], gb[i][1], gb[i][2], gb[i][3]};
                if (nrm) {   // through u = y / n:  (dy - u (u . dy)) / n
                    const float r = rsqrtf(rs[j] + a.eps), kk = r * r * rs[kBwdGroup + j];
#pragma unroll
                    for (int u = 0; u < 4; ++u) dy[u] = (dy[u] - y[j][u] * kk) * r;
                }
                const bool live = t < tv, own = t < t1;
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const float dx = dy[u] * fd[j][u];
                    dwin[3 + i][u] = live ? dx : 0.f;
                    const float dxo = own ? dx : 0.f;   // the conv-weight sums take the run's own tokens
                    dw[0][u] = fmaf(dxo, win[i][u], dw[0][u]);
                    dw[1][u] = fmaf(dxo, win[i + 1][u], dw[1][u]);
                    dw[2][u] = fmaf(dxo, win[i + 2][u], dw[2][u]);
                    dw[3][u] = fmaf(dxo, win[i + 3][u], dw[3][u]);
                }
            }
        }
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int tp = tb + i - 3;   // dP of token t - 3 reads dx of t - 3 .. t
            if (m.act && tp >= t0 && tp < te) {
                float d[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    float v = w[0][u] * dwin[i + 3][u];
                    v = fmaf(w[1][u], dwin[i + 2][u], v);
                    v = fmaf(w[2][u], dwin[i + 1][u], v);
                    v = fmaf(w[3][u], dwin[i][u], v);
                    d[u] = v;
                }
                st4<VEC>(pdP + tp * sP, d);
            }
        }
#pragma unroll
        for (int i = 0; i < 3; ++i)
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                pw[i][u] = win[4 + i][u];
                dxw[i][u] = dwin[4 + i][u];
            }
    }
    if (m.act)
#pragma unroll
        for (int u = 0; u < 4; ++u)
#pragma unroll
            for (int j = 0; j < 4; ++j)
                if (j >= 4 - K) part[(m.c + u) * K + j - (4 - K)] = dw[j][u];
}

template <typename Tin, typename Tg>
__device__ __forceinline__ void prologue_bwd_small(const tla_prologue_args& a, const PrologueGrads& gr,
                                                   int b, int h, int t0, int t1, float* part) {
    const int lane = threadIdx.x & 31;
    const int dk = a.dk, dv = a.dv, E = a.E, K = a.K, T = a.T, H = a.H;
    const int C = 2 * dk + dv + 2 * E, off = 2 * dk + dv;
    bool act[2], isq[2];
    int col[2];
    float w[4][2], dw[4][2];
#pragma unroll
    for (int s = 0; s < 2; ++s) {
        const int cc = lane + 32 * s;
        act[s] = cc < 2 * E;
        isq[s] = cc < E;
        col[s] = cc < E ? cc : cc - E;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            w[j][s] = (act[s] && j >= 4 - K) ? a.conv_w[(size_t(h) * C + off + cc) * K + j - (4 - K)] : 0.f;
            dw[j][s] = 0.f;
        }
    }
    const size_t sP = size_t(H) * C, sE = size_t(H) * E;
    const size_t rowP = (size_t(b) * T * H + h) * C + off + lane;
    const Tin* pP = static_cast<const Tin*>(a.P) + rowP;
    Tin* pdP = static_cast<Tin*>(gr.dP) + rowP;
    const size_t rowE = (size_t(b) * T * H + h) * E;
    const Tg* gq = static_cast<const Tg*>(gr.dq2);
    const Tg* gk = static_cast<const Tg*>(gr.dk2);
    float pw[3][2], dxw[3][2];
#pragma unroll
    for (int i = 0; i < 3; ++i)
#pragma unroll
        for (int s = 0; s < 2; ++s) {
            const int t = t0 - 3 + i;
            pw[i][s] = (act[s] && t >= 0) ? to_f(pP[t * sP + 32 * s]) : 0.f;
            dxw[i][s] = 0.f;
        }
    const int tl = t1 + 3, tv = min(tl, T), te = min(t1, T);
    for (int tb = t0; tb < tl; tb += 4) {
        // as in prologue_bwd_qkv: rows t-3 .. t+3 in win, the four tokens' activations, then
        // their row sums together, then their gradients, with no branch per token
        float win[7][2], gb[4][2];
#pragma unroll
        for (int i = 0; i < 3; ++i)
#pragma unroll
            for (int s = 0; s < 2; ++s) win[i][s] = pw[i][s];
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int s = 0; s < 2; ++s) {
                const bool ok = act[s] && tb + i < tv;
                const size_t o = rowE + (tb + i) * sE + col[s];
                win[3 + i][s] = ok ? to_f(pP[(tb + i) * sP + 32 * s]) : 0.f;
                gb[i][s] = ok ? to_f(isq[s] ? gq[o] : gk[o]) : 0.f;
            }
        float sx[4][2], y[4][2], rs[16];   // sx = sigmoid(x); rs: sq, sk, dq, dk of the four tokens
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            float sq = 0.f, sk = 0.f, dq = 0.f, dkk = 0.f;
#pragma unroll
            for (int s = 0; s < 2; ++s) {
                float v = w[0][s] * win[i][s];
                v = fmaf(w[1][s], win[i + 1][s], v);
                v = fmaf(w[2][s], win[i + 2][s], v);
                v = fmaf(w[3][s], win[i + 3][s], v);
                sx[i][s] = sigm(v);
                y[i][s] = act[s] ? softplus(v) : 0.f;
                if (isq[s]) { sq = fmaf(y[i][s], y[i][s], sq); dq = fmaf(y[i][s], gb[i][s], dq); }
                else { sk = fmaf(y[i][s], y[i][s], sk); dkk = fmaf(y[i][s], gb[i][s], dkk); }
            }
            rs[i] = sq;
            rs[4 + i] = sk;
            rs[8 + i] = dq;
            rs[12 + i] = dkk;
        }
        warp_sum_n(rs);
        float dwin[7][2];
#pragma unroll
        for (int i = 0; i < 3; ++i)
#pragma unroll
            for (int s = 0; s < 2; ++s) dwin[i][s] = dxw[i][s];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int t = tb + i;
            const float rq = rsqrtf(rs[i] + a.eps), rk = rsqrtf(rs[4 + i] + a.eps);
            const float kq = rq * rq * rs[8 + i], kk = rk * rk * rs[12 + i];
            const bool live = t < tv, own = t < t1;
#pragma unroll
            for (int s = 0; s < 2; ++s) {
                const float r = isq[s] ? rq : rk, k2 = isq[s] ? kq : kk;
                const float dx = act[s] ? (gb[i][s] - y[i][s] * k2) * r * sx[i][s] : 0.f;
                dwin[3 + i][s] = live ? dx : 0.f;
                const float dxo = own ? dx : 0.f;
                dw[0][s] = fmaf(dxo, win[i][s], dw[0][s]);
                dw[1][s] = fmaf(dxo, win[i + 1][s], dw[1][s]);
                dw[2][s] = fmaf(dxo, win[i + 2][s], dw[2][s]);
                dw[3][s] = fmaf(dxo, win[i + 3][s], dw[3][s]);
            }
        }
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int tp = tb + i - 3;
            if (tp >= t0 && tp < te)
#pragma unroll
                for (int s = 0; s < 2; ++s)
                    if (act[s]) {
                        float v = w[0][s] * dwin[i + 3][s];
                        v = fmaf(w[1][s], dwin[i + 2][s], v);
                        v = fmaf(w[2][s], dwin[i + 1][s], v);
                        v = fmaf(w[3][s], dwin[i][s], v);
                        pdP[tp * sP + 32 * s] = from_f<Tin>(v);
                    }
        }
#pragma unroll
        for (int i = 0; i < 3; ++i)
#pragma unroll
            for (int s = 0; s < 2; ++s) {
                pw[i][s] = win[4 + i][s];
                dxw[i][s] = dwin[4 + i][s];
            }
    }
#pragma unroll
    for (int s = 0; s < 2; ++s)
        if (act[s])
#pragma unroll
            for (int j = 0; j < 4; ++j)
                if (j >= 4 - K) part[(off + lane + 32 * s) * K + j - (4 - K)] = dw[j][s];
}

// Gradients through the log gates and beta of tokens [t0, t1) of (b, h), with the gate-bias
// and A_log partials of this CTA (the v warp, whose channels need no norm).
__device__ __forceinline__ void prologue_bwd_gates(const tla_prologue_args& a, const PrologueGrads& gr,
                                                   int b, int h, int t0, int t1, float* part) {
    const int lane = threadIdx.x & 31;
    const int dk = a.dk, dv = a.dv, E = a.E, K = a.K, T = a.T, H = a.H;
    const int C = 2 * dk + dv + 2 * E;
    const size_t sE = size_t(H) * E;
    const size_t rowE = (size_t(b) * T * H + h) * E;
    const int te = min(t1, T);
    // log gates: lane p * E + e takes gate e of tokens t0 + p, t0 + p + NP, ... (NP = 32 / E
    // phases), eight tokens' loads at a time; the phases' sums are added in order after.
    __shared__ float red[2][32];
    const int NP = 32 / E, p = lane / E, e = lane - p * E;
    float gbp = 0.f, gap = 0.f;
    if (p < NP) {
        const float sA = -__expf(a.A_log[h * E + e]), bias = a.gate_bias[h * E + e];
        for (int tb = t0 + p; tb < te; tb += 8 * NP) {
            float z[8], dgv[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const int t = tb + i * NP;
                const size_t o = rowE + t * sE + e;
                z[i] = t < te ? a.gate_in[o] + bias : 0.f;
                dgv[i] = t < te ? gr.dg[o] : 0.f;
            }
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const int t = tb + i * NP;
                if (t < te) {
                    const float dz = dgv[i] * sA * sigm(z[i]);
                    gr.dgate_in[rowE + t * sE + e] = dz;
                    gbp += dz;
                    gap = fmaf(dgv[i], sA * softplus(z[i]), gap);
                }
            }
        }
    }
    red[0][lane] = gbp;
    red[1][lane] = gap;
    __syncwarp();
    if (lane < E) {
        float sb = 0.f, sa = 0.f;
        for (int q = 0; q < NP; ++q) {
            sb += red[0][q * E + lane];
            sa += red[1][q * E + lane];
        }
        part[C * K + lane] = sb;
        part[C * K + E + lane] = sa;
    }
    if (a.beta_in)
        for (int tb = t0 + lane; tb < te; tb += 32 * 8) {
            float bi[8], db[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const int t = tb + 32 * i;
                const size_t o = (size_t(b) * T + t) * H + h;
                bi[i] = t < te ? a.beta_in[o] : 0.f;
                db[i] = t < te ? gr.dbeta[o] : 0.f;
            }
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const int t = tb + 32 * i;
                if (t < te) {
                    const float s = sigm(bi[i]);
                    gr.dbeta_in[(size_t(b) * T + t) * H + h] = db[i] * s * (1.f - s);
                }
            }
        }
}

template <typename Tin, typename Tg, bool VEC>
__global__ void __launch_bounds__(kPrWarps * 32, 4)
prologue_bwd_kernel(const tla_prologue_args a, const PrologueGrads gr) {
    const int seg = blockIdx.x, h = blockIdx.y, b = blockIdx.z, g = threadIdx.x >> 5;
    const int t0 = seg * kSeg, t1 = min(a.T, t0 + kSeg);
    const int C = 2 * a.dk + a.dv + 2 * a.E;
    float* part = gr.part + ((size_t(b) * gridDim.x + seg) * a.H + h) * (size_t(C) * a.K + 2 * a.E);
    if (g < 3) prologue_bwd_qkv<Tin, Tg, VEC>(a, gr, g, b, h, t0, t1, part);
    else prologue_bwd_small<Tin, Tg>(a, gr, b, h, t0, t1, part);
    if (g == 2) prologue_bwd_gates(a, gr, b, h, t0, t1, part);
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

// Bulk copy shared -> global (16-byte aligned addresses, size a multiple of 16) in the issuing
// thread's bulk async-group.
__device__ __forceinline__ void bulk_store_g(void* dst, const void* src, uint32_t bytes) {
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(
                     reinterpret_cast<uint64_t>(dst)),
                 "r"(sm100::smem_u32(src)), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void bulk_commit_g() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read_g() {
    asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}

// Output gate through shared memory (dv <= 128 and a multiple of 16): the kGateTile
// consecutive (token, head) rows of a CTA are contiguous in o, z and y, so they arrive by one
// bulk copy per tensor; one warp per row (four channels per lane) normalises and gates in
// shared memory, y over z in place, and y leaves by one bulk copy.  With little register
// state several CTAs' copies are in flight on an SM.
template <typename To, typename Tz>
__global__ void __launch_bounds__(kThreads)
gate_fwd_kernel(const tla_gate_args a, long long rows, int* err) {
    using namespace sm100;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 127) & ~uintptr_t(127));
    __shared__ __align__(8) uint64_t bar;
    const int dv = a.dv, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const long long r0 = blockIdx.x * (long long)kGateTile;
    const int nr = (int)min((long long)kGateTile, rows - r0);
    To* so = reinterpret_cast<To*>(sm);
    Tz* sz = reinterpret_cast<Tz*>(sm + size_t(kGateTile) * dv * sizeof(To));
    const uint32_t bo = uint32_t(nr) * dv * sizeof(To), bz = uint32_t(nr) * dv * sizeof(Tz);
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        fence_barrier_init();
        mbar_arrive_expect_tx(&bar, bo + bz);
        bulk_load(so, static_cast<const To*>(a.o) + r0 * dv, bo, &bar);
        bulk_load(sz, static_cast<const Tz*>(a.z) + r0 * dv, bz, &bar);
    }
    const bool act = 4 * lane < dv;
    float wn[4] = {0.f, 0.f, 0.f, 0.f};
    if (act) ld4<true>(a.w_norm + 4 * lane, wn);
    __syncthreads();
    const bool ok = mbar_wait(&bar, 0);
    if (__syncthreads_or(!ok)) {
        if (threadIdx.x == 0) {
            record_device_error(err, TLA_ERR_TIMEOUT);
            mbar_wait(&bar, 0);   // bounded drain of the copies
        }
        return;
    }
    for (int r = warp; r < nr; r += kThreads / 32) {
        float o[4] = {0.f, 0.f, 0.f, 0.f}, z[4] = {0.f, 0.f, 0.f, 0.f};
        if (act) {
            ld4<true>(so + r * dv + 4 * lane, o);
            ld4<true>(sz + r * dv + 4 * lane, z);
        }
        float ss = 0.f;
#pragma unroll
        for (int u = 0; u < 4; ++u) ss = fmaf(o[u], o[u], ss);
        const float rr = rsqrtf(warp_sum(ss) / dv + a.eps);
        float y[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) y[u] = o[u] * rr * wn[u] * sigm(z[u]);
        if (act) st4<true>(sz + r * dv + 4 * lane, y);
    }
    fence_proxy_async_smem();
    __syncthreads();
    if (threadIdx.x == 0) {   // the CTA's shared memory must outlive the copy's read
        bulk_store_g(static_cast<Tz*>(a.y) + r0 * dv, sz, bz);
        bulk_commit_g();
        bulk_wait_read_g();
    }
}

// Backward of the output gate through shared memory, kGateBwdTiles tiles of kGateTile rows per
// CTA in turn: a tile's rows of o, z and dy arrive by one bulk copy each; do and dz are written
// in place over o and z and leave by one bulk copy each; the w_norm gradient is summed per lane
// over the CTA's rows, then over its warps in order into part[blk][dv].
constexpr int kGateBwdTiles = 4;
template <typename To, typename Tz>
__global__ void __launch_bounds__(kThreads)
gate_bwd_kernel(const tla_gate_args a, long long rows, const void* dy, void* d_o, void* dz,
                float* part, int* err) {
    using namespace sm100;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 127) & ~uintptr_t(127));
    __shared__ __align__(8) uint64_t bar;
    __shared__ float wsm[kThreads / 32][128];
    const int dv = a.dv, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    To* so = reinterpret_cast<To*>(sm);                                          // o, then do
    Tz* sz = reinterpret_cast<Tz*>(sm + size_t(kGateTile) * dv * sizeof(To));    // z, then dz
    Tz* sg = sz + size_t(kGateTile) * dv;                                        // dy
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        fence_barrier_init();
    }
    const bool act = 4 * lane < dv;
    float wn[4] = {0.f, 0.f, 0.f, 0.f}, wacc[4] = {0.f, 0.f, 0.f, 0.f};
    if (act) ld4<true>(a.w_norm + 4 * lane, wn);
    const float inv_dv = 1.f / dv;
    __syncthreads();
    for (int j = 0; j < kGateBwdTiles; ++j) {
        const long long r0 = (blockIdx.x * (long long)kGateBwdTiles + j) * kGateTile;
        if (r0 >= rows) break;
        const int nr = (int)min((long long)kGateTile, rows - r0);
        const uint32_t bo = uint32_t(nr) * dv * sizeof(To), bz = uint32_t(nr) * dv * sizeof(Tz);
        if (threadIdx.x == 0) {
            mbar_arrive_expect_tx(&bar, bo + 2 * bz);
            bulk_load(so, static_cast<const To*>(a.o) + r0 * dv, bo, &bar);
            bulk_load(sz, static_cast<const Tz*>(a.z) + r0 * dv, bz, &bar);
            bulk_load(sg, static_cast<const Tz*>(dy) + r0 * dv, bz, &bar);
        }
        const bool ok = mbar_wait(&bar, uint32_t(j) & 1u);
        if (__syncthreads_or(!ok)) {
            if (threadIdx.x == 0) {
                record_device_error(err, TLA_ERR_TIMEOUT);
                mbar_wait(&bar, uint32_t(j) & 1u);   // bounded drain of the copies
            }
            return;
        }
        for (int r = warp; r < nr; r += kThreads / 32) {
            float o[4] = {0.f, 0.f, 0.f, 0.f}, z[4] = {0.f, 0.f, 0.f, 0.f}, g[4] = {0.f, 0.f, 0.f, 0.f};
            if (act) {
                ld4<true>(so + r * dv + 4 * lane, o);
                ld4<true>(sz + r * dv + 4 * lane, z);
                ld4<true>(sg + r * dv + 4 * lane, g);
            }
            float ss = 0.f;
#pragma unroll
            for (int u = 0; u < 4; ++u) ss = fmaf(o[u], o[u], ss);
            const float rr = rsqrtf(warp_sum(ss) * inv_dv + a.eps);
            float nh[4], dnh[4], dzv[4], dot = 0.f;
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const float sgm = sigm(z[u]);
                nh[u] = o[u] * rr;
                dnh[u] = g[u] * wn[u] * sgm;
                dzv[u] = g[u] * nh[u] * wn[u] * sgm * (1.f - sgm);
                wacc[u] = fmaf(g[u] * sgm, nh[u], wacc[u]);
                dot = fmaf(dnh[u], nh[u], dot);
            }
            dot = warp_sum(dot) * inv_dv;
            float dov[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) dov[u] = rr * (dnh[u] - nh[u] * dot);
            if (act) {
                st4<true>(sz + r * dv + 4 * lane, dzv);
                st4<true>(so + r * dv + 4 * lane, dov);
            }
        }
        fence_proxy_async_smem();
        __syncthreads();
        if (threadIdx.x == 0) {   // the next tile's copies overwrite these buffers
            bulk_store_g(static_cast<To*>(d_o) + r0 * dv, so, bo);
            bulk_store_g(static_cast<Tz*>(dz) + r0 * dv, sz, bz);
            bulk_commit_g();
            bulk_wait_read_g();
        }
    }
    if (act)
#pragma unroll
        for (int u = 0; u < 4; ++u) wsm[warp][4 * lane + u] = wacc[u];
    __syncthreads();
    for (int c = threadIdx.x; c < dv; c += kThreads) {
        float acc = 0.f;
        for (int w = 0; w < kThreads / 32; ++w) acc += wsm[w][c];
        part[size_t(blockIdx.x) * dv + c] = acc;
    }
}

// Fixed-order column sums out[c] = sum_i part[i][c]: block of 8 warps per 32 columns,
// warp w summing the rows i = w, w + 8, ...; the eight sums then added in order.
__global__ void __launch_bounds__(256) reduce_columns_kernel(const float* __restrict__ part, int nblk,
                                                             int n, float* __restrict__ out) {
    __shared__ float sm[8][32];
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, c = blockIdx.x * 32 + lane;
    float acc = 0.f;
    if (c < n)
        for (int i = w; i < nblk; i += 8) acc += part[size_t(i) * n + c];
    sm[w][lane] = acc;
    __syncthreads();
    if (w == 0 && c < n) {
        float t = 0.f;
        for (int j = 0; j < 8; ++j) t += sm[j][lane];
        out[c] = t;
    }
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
// forward: one CTA per kGateTile (token, head) rows; backward: kGateBwdTiles such tiles per
// CTA, each CTA writing one partial w_norm gradient
long long gate_blocks(const tla_gate_args* a) {
    return ((long long)a->B * a->T * a->H + kGateTile - 1) / kGateTile;
}
long long gate_bwd_blocks(const tla_gate_args* a) {
    const long long per = (long long)kGateTile * kGateBwdTiles;
    return ((long long)a->B * a->T * a->H + per - 1) / per;
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
    dim3 grid((a->T + kFwdRun - 1) / kFwdRun, a->H, a->B);
    const bool vec = (C % 4) == 0;   // every row and channel group starts on four channels
    prof_before("layer_prologue", s);
    if (a->dtype == TLA_BF16) {
        if (vec) prologue_fwd_kernel<__nv_bfloat16, true><<<grid, kPrWarps * 32, 0, s>>>(*a);
        else prologue_fwd_kernel<__nv_bfloat16, false><<<grid, kPrWarps * 32, 0, s>>>(*a);
    } else {
        if (vec) prologue_fwd_kernel<float, true><<<grid, kPrWarps * 32, 0, s>>>(*a);
        else prologue_fwd_kernel<float, false><<<grid, kPrWarps * 32, 0, s>>>(*a);
    }
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
    dim3 grid(n_segments(a), a->H, a->B);
    const bool vec = (C % 4) == 0;
    prof_before("layer_prologue_bwd", s);
#define TLA_PROLOGUE_BWD(TI, TG)                                                        \
    do {                                                                                \
        if (vec) prologue_bwd_kernel<TI, TG, true><<<grid, kPrWarps * 32, 0, s>>>(*a, gr); \
        else prologue_bwd_kernel<TI, TG, false><<<grid, kPrWarps * 32, 0, s>>>(*a, gr);    \
    } while (0)
    if (a->dtype == TLA_BF16) {
        if (grad_dtype == TLA_BF16) TLA_PROLOGUE_BWD(__nv_bfloat16, __nv_bfloat16);
        else TLA_PROLOGUE_BWD(__nv_bfloat16, float);
    } else {
        if (grad_dtype == TLA_BF16) TLA_PROLOGUE_BWD(float, __nv_bfloat16);
        else TLA_PROLOGUE_BWD(float, float);
    }
#undef TLA_PROLOGUE_BWD
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
    const size_t so = a->o_dtype == TLA_FP32 ? 4 : 2, sz = a->dtype == TLA_FP32 ? 4 : 2;
    const size_t smem = 128 + size_t(kGateTile) * a->dv * (so + sz);
    int* err = device_error_word();
    if (!err) return TLA_ERR_CUDA;
    prof_before("output_gate", s);
#define TLA_GATE_LAUNCH(TO, TZ)                                                                    \
    do {                                                                                           \
        auto kern = gate_fwd_kernel<TO, TZ>;                                                       \
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);        \
        kern<<<blocks, kThreads, smem, s>>>(*a, rows, err);                                        \
    } while (0)
    if (a->o_dtype == TLA_FP32) {
        if (a->dtype == TLA_FP32) TLA_GATE_LAUNCH(float, float);
        else TLA_GATE_LAUNCH(float, __nv_bfloat16);
    } else {
        if (a->dtype == TLA_FP32) TLA_GATE_LAUNCH(__nv_bfloat16, float);
        else TLA_GATE_LAUNCH(__nv_bfloat16, __nv_bfloat16);
    }
#undef TLA_GATE_LAUNCH
    prof_after(s);
    return cuda_status(cudaGetLastError());
}

extern "C" size_t tla_output_gate_bwd_workspace_bytes(const tla_gate_args* a) {
    if (check_gate(a) != TLA_OK) return 0;
    return ((size_t)gate_bwd_blocks(a) * a->dv * sizeof(float) + 255) & ~size_t(255);
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
    const long long nblk = gate_bwd_blocks(a);
    if (!workspace || workspace_bytes < (size_t)nblk * a->dv * sizeof(float)) return TLA_ERR_WORKSPACE;
    cudaStream_t s = (cudaStream_t)stream;
    const long long rows = (long long)a->B * a->T * a->H;
    float* part = (float*)workspace;
    const unsigned g = (unsigned)nblk;
    const size_t so = a->o_dtype == TLA_FP32 ? 4 : 2, sz = a->dtype == TLA_FP32 ? 4 : 2;
    const size_t smem = 128 + size_t(kGateTile) * a->dv * (so + 2 * sz);
    int* err = device_error_word();
    if (!err) return TLA_ERR_CUDA;
    prof_before("output_gate_bwd", s);
#define TLA_GATE_BWD_LAUNCH(TO, TZ)                                                                \
    do {                                                                                           \
        auto kern = gate_bwd_kernel<TO, TZ>;                                                       \
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);        \
        kern<<<g, kThreads, smem, s>>>(*a, rows, dy, d_o, dz, part, err);                          \
    } while (0)
    if (a->o_dtype == TLA_FP32) {
        if (a->dtype == TLA_FP32) TLA_GATE_BWD_LAUNCH(float, float);
        else TLA_GATE_BWD_LAUNCH(float, __nv_bfloat16);
    } else {
        if (a->dtype == TLA_FP32) TLA_GATE_BWD_LAUNCH(__nv_bfloat16, float);
        else TLA_GATE_BWD_LAUNCH(__nv_bfloat16, __nv_bfloat16);
    }
#undef TLA_GATE_BWD_LAUNCH
    prof_after(s);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return TLA_ERR_CUDA;
    prof_before("output_gate_reduce", s);
    reduce_columns_kernel<<<(a->dv + 31) / 32, 256, 0, s>>>(part, (int)nblk, a->dv, dw_norm);
    prof_after(s);
    return cuda_status(cudaGetLastError());
}
