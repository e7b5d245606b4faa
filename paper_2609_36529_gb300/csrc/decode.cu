// Single-token decode step (Algorithm 2, one iteration), HBM-bound.
//
// Per (b, h) and block of TV value columns one CTA streams its E x dk x TV
// slab of the fp32 state once from HBM into registers (16-byte loads, rows of
// TV contiguous floats), and writes the updated slab back once:
//   Shat_e = alpha_e S_e                                   (Eq. forget3)
//   r      = sum_e k'_e Shat_e^T k,  u = beta (v - r)      (Eq. gdn3; sGLA: u = beta v)
//   S_e    = Shat_e + k'_e k u^T                           (triadic write)
//   o      = sum_e q'_e S_e^T q = p + (q'.k')(q.k) u,  p = sum_e q'_e Shat_e^T q
// The last identity lets o come from the same single read of the slab.
// Reductions over (e, d) use warp shuffles then a fixed-order pass over warps,
// so results are deterministic.
#include "common.cuh"
#include "internal.h"

namespace tla {

constexpr int kDecThreads = 256;

// TPR threads per slab row (TV = 4 * TPR columns); MAXP float4 registers per thread.
// Two or more CTAs per SM let one CTA's loads overlap another's stores.
template <typename Tin, int TPR, int MAXP>
__global__ void __launch_bounds__(kDecThreads, (MAXP <= 16 ? 2 : 1))
decode_step_kernel(const Tin* __restrict__ q, const Tin* __restrict__ k,
                   const Tin* __restrict__ v, const Tin* __restrict__ q2,
                   const Tin* __restrict__ k2, const float* __restrict__ g,
                   const float* __restrict__ beta, float* __restrict__ state,
                   Tin* __restrict__ o, int dk, int dv, int E, int use_delta) {
    constexpr int TV = 4 * TPR;
    constexpr int RPP = kDecThreads / TPR;  // slab rows per pass
    constexpr int NW = kDecThreads / 32;
    const int nb = blockIdx.x;
    const int bh = blockIdx.y;
    const int n0 = nb * TV;
    const int tid = threadIdx.x;
    const int quad = tid % TPR;       // which 4 columns
    const int row0 = tid / TPR;       // first slab row of this thread
    const int rows = E * dk;
    const int passes = (rows + RPP - 1) / RPP;

    __shared__ float qs[128], ks[128], q2s[32], k2s[32], al[32];
    __shared__ float4 red_r[NW][TPR], red_p[NW][TPR];
    __shared__ __align__(16) float us[TV];
    __shared__ float qk_s, q2k2_s;

    for (int i = tid; i < dk; i += kDecThreads) {
        qs[i] = to_f(q[size_t(bh) * dk + i]);
        ks[i] = to_f(k[size_t(bh) * dk + i]);
    }
    if (tid < E) {
        q2s[tid] = to_f(q2[size_t(bh) * E + tid]);
        k2s[tid] = to_f(k2[size_t(bh) * E + tid]);
        al[tid] = expf(g[size_t(bh) * E + tid]);
    }
    float4* S4 = reinterpret_cast<float4*>(state + size_t(bh) * rows * dv + n0) + quad;
    const int row_stride4 = dv / 4;

    // stream the slab in: all loads issued before any use
    float4 reg[MAXP];
#pragma unroll
    for (int p = 0; p < MAXP; ++p) {
        int row = row0 + p * RPP;
        if (p < passes && row < rows) reg[p] = __ldcs(S4 + size_t(row) * row_stride4);
        else reg[p] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
    __syncthreads();
    if (tid == 0) {
        float a = 0.f, c = 0.f;
        for (int i = 0; i < dk; ++i) a = fmaf(qs[i], ks[i], a);
        for (int e = 0; e < E; ++e) c = fmaf(q2s[e], k2s[e], c);
        qk_s = a;
        q2k2_s = c;
    }
    // decay, then partial reads at the joint key (k, k') and the joint query (q, q')
    float4 pr = make_float4(0.f, 0.f, 0.f, 0.f), pp = pr;
#pragma unroll
    for (int p = 0; p < MAXP; ++p) {
        int row = row0 + p * RPP;
        if (p < passes && row < rows) {
            int e = row / dk, d = row - e * dk;
            float a = al[e];
            float4 s = reg[p];
            s.x *= a; s.y *= a; s.z *= a; s.w *= a;
            reg[p] = s;
            float ck = k2s[e] * ks[d], cq = q2s[e] * qs[d];
            pr.x = fmaf(ck, s.x, pr.x); pr.y = fmaf(ck, s.y, pr.y);
            pr.z = fmaf(ck, s.z, pr.z); pr.w = fmaf(ck, s.w, pr.w);
            pp.x = fmaf(cq, s.x, pp.x); pp.y = fmaf(cq, s.y, pp.y);
            pp.z = fmaf(cq, s.z, pp.z); pp.w = fmaf(cq, s.w, pp.w);
        }
    }
#pragma unroll
    for (int off = TPR; off < 32; off <<= 1) {
        pr.x += __shfl_xor_sync(0xffffffffu, pr.x, off);
        pr.y += __shfl_xor_sync(0xffffffffu, pr.y, off);
        pr.z += __shfl_xor_sync(0xffffffffu, pr.z, off);
        pr.w += __shfl_xor_sync(0xffffffffu, pr.w, off);
        pp.x += __shfl_xor_sync(0xffffffffu, pp.x, off);
        pp.y += __shfl_xor_sync(0xffffffffu, pp.y, off);
        pp.z += __shfl_xor_sync(0xffffffffu, pp.z, off);
        pp.w += __shfl_xor_sync(0xffffffffu, pp.w, off);
    }
    const int lane = tid & 31, warp = tid >> 5;
    if (lane < TPR) {
        red_r[warp][lane] = pr;
        red_p[warp][lane] = pp;
    }
    __syncthreads();
    if (tid < TV) {
        const int qd = tid / 4, comp = tid % 4;
        float r = 0.f, pq = 0.f;
        for (int w = 0; w < NW; ++w) {
            const float* a = reinterpret_cast<const float*>(&red_r[w][qd]);
            const float* b = reinterpret_cast<const float*>(&red_p[w][qd]);
            r += a[comp];
            pq += b[comp];
        }
        const int col = n0 + tid;
        float vv = to_f(v[size_t(bh) * dv + col]);
        float bt = beta ? beta[bh] : 1.f;
        float u = use_delta ? bt * (vv - r) : bt * vv;
        us[tid] = u;
        o[size_t(bh) * dv + col] = from_f<Tin>(fmaf(q2k2_s * qk_s, u, pq));
    }
    __syncthreads();
    const float4 u4 = reinterpret_cast<const float4*>(us)[quad];
#pragma unroll
    for (int p = 0; p < MAXP; ++p) {
        int row = row0 + p * RPP;
        if (p < passes && row < rows) {
            int e = row / dk, d = row - e * dk;
            float c = k2s[e] * ks[d];
            float4 s = reg[p];
            s.x = fmaf(c, u4.x, s.x); s.y = fmaf(c, u4.y, s.y);
            s.z = fmaf(c, u4.z, s.z); s.w = fmaf(c, u4.w, s.w);
            __stcs(S4 + size_t(row) * row_stride4, s);
        }
    }
}

cudaError_t launch_decode_step(int B, int H, int dk, int dv, int E, int use_delta, int dtype,
                               const void* q, const void* k, const void* v, const void* q2,
                               const void* k2, const float* g, const float* beta,
                               float* state, void* o, cudaStream_t s) {
    // TV = 16 columns (64-byte row segments): the slab of E x dk rows takes
    // rows / 64 float4 registers per thread (16 for E*dk <= 1024, else 32).
    const int rows = E * dk;
    const int TV = 16;
    dim3 grid(dv / TV, B * H);
    prof_before("decode_step", s);
    if (dtype == TLA_BF16) {
        using Tb = __nv_bfloat16;
        if (rows <= 16 * 64)
            decode_step_kernel<Tb, 4, 16><<<grid, kDecThreads, 0, s>>>(
                (const Tb*)q, (const Tb*)k, (const Tb*)v, (const Tb*)q2, (const Tb*)k2, g, beta,
                state, (Tb*)o, dk, dv, E, use_delta);
        else
            decode_step_kernel<Tb, 4, 32><<<grid, kDecThreads, 0, s>>>(
                (const Tb*)q, (const Tb*)k, (const Tb*)v, (const Tb*)q2, (const Tb*)k2, g, beta,
                state, (Tb*)o, dk, dv, E, use_delta);
    } else {
        if (rows <= 16 * 64)
            decode_step_kernel<float, 4, 16><<<grid, kDecThreads, 0, s>>>(
                (const float*)q, (const float*)k, (const float*)v, (const float*)q2,
                (const float*)k2, g, beta, state, (float*)o, dk, dv, E, use_delta);
        else
            decode_step_kernel<float, 4, 32><<<grid, kDecThreads, 0, s>>>(
                (const float*)q, (const float*)k, (const float*)v, (const float*)q2,
                (const float*)k2, g, beta, state, (float*)o, dk, dv, E, use_delta);
    }
    prof_after(s);
    return cudaGetLastError();
}

}  // namespace tla
