// SIMT (fp32 CUDA-core) kernels of the chunkwise forward, Appendix A.
//
// These kernels compute every step in fp32 and serve the fp32 problems (whose
// tolerance rules out bf16/tf32 tensor-core operands) and every shape the
// tensor-core path does not cover.  Steps:
//   gate_cumsum_kernel   G_{r,e} = sum_{j<=r} log alpha_{j,e}, chunk-local      (Eq. joint-gram, gamma)
//   chunk_prep_kernel    R, R' element by element (Eq. joint-gram, "Numerical
//                        stability"), A = Q K^T (.) R' (Eq. separate / joint-chunk),
//                        N = (I + tril(diag(beta)(K K^T (.) R), -1))^{-1}  (Eq. joint-solve;
//                        T = N diag(beta))
//   fwd_recurrence_kernel  the chunk step of Eq. joint-chunk carried over chunks,
//                        one CTA per (b, h, block of tv value columns): value
//                        columns never interact (Section 2.5, Eq. slices).
#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace tla {

// ---------------------------------------------------------------------------
__global__ void gate_cumsum_kernel(const float* __restrict__ g, float* __restrict__ G,
                                   const int2* __restrict__ ctab, int B, int T, int H, int E,
                                   int NT, int per_head) {
    long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x;
    long long total = (long long)B * NT * H * E;
    if (idx >= total) return;
    int e = int(idx % E);
    long long x = idx / E;
    int h = int(x % H);
    x /= H;
    int c = int(x % NT);
    int b = int(x / NT);
    int t0 = c * kChunk;
    int n = min(kChunk, T - t0);
    if (ctab) {   // packed documents: the chunk's first token and rows
        const int2 cr = ctab[c];
        t0 = cr.x;
        n = cr.y;
    }
    float acc = 0.f;
    for (int r = 0; r < n; ++r) {
        size_t off = tok_idx(b, t0 + r, h, e, T, H, E);
        acc += per_head ? g[(size_t(b) * T + t0 + r) * H + h] : g[off];   // per-head gate: every slice
        G[off] = acc;
    }
}

cudaError_t launch_gate_cumsum(const tla_problem& p, const FwdPlan& fp, const char* ws, float* G,
                               cudaStream_t s) {
    const int NT = fp.NT;
    long long total = (long long)p.B * NT * p.H * p.E;
    if (total == 0) return cudaSuccess;
    int threads = 256;
    long long blocks = (total + threads - 1) / threads;
    const int2* ctab = p.cu_seqlens ? (const int2*)(ws + fp.ctab) : nullptr;
    prof_before("gate_cumsum", s);
    gate_cumsum_kernel<<<(unsigned)blocks, threads, 0, s>>>(p.g, G, ctab, p.B, p.T, p.H, p.E, NT,
                                                            p.gate_per_head);
    prof_after(s);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Per (b, h, chunk): A (64x64, lower incl. diagonal) and N = (I + L)^{-1}.
template <typename Tin>
__global__ void __launch_bounds__(256)
chunk_prep_kernel(const Tin* __restrict__ q, const Tin* __restrict__ k, const Tin* __restrict__ q2,
                  const Tin* __restrict__ k2, const float* __restrict__ G,
                  const float* __restrict__ beta, float* __restrict__ Aout,
                  float* __restrict__ Nout, int T, int H, int dk, int E, int use_delta) {
    const int c = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
    const int NT = gridDim.x;
    const int tid = threadIdx.x;
    const int t0 = c * kChunk;
    const int n = min(kChunk, T - t0);
    const int DKP = dk + 1;
    extern __shared__ float sm[];
    float* Ks = sm;
    float* Qs = Ks + kChunk * DKP;
    float* Gs = Qs + kChunk * DKP;
    float* k2s = Gs + kChunk * E;
    float* q2s = k2s + kChunk * E;
    float* bs = q2s + kChunk * E;
    float* Ls = bs + kChunk;
    float* Xs = Ls + kChunk * 65;
    float* As = Xs + kChunk * 65;
    float* part = As + kChunk * 65;

    for (int i = tid; i < kChunk * dk; i += blockDim.x) {
        int r = i / dk, d = i % dk;
        float kv = 0.f, qv = 0.f;
        if (r < n) {
            kv = to_f(k[tok_idx(b, t0 + r, h, d, T, H, dk)]);
            qv = to_f(q[tok_idx(b, t0 + r, h, d, T, H, dk)]);
        }
        Ks[r * DKP + d] = kv;
        Qs[r * DKP + d] = qv;
    }
    for (int i = tid; i < kChunk * E; i += blockDim.x) {
        int r = i / E, e = i % E;
        int rr = r < n ? r : n - 1;
        Gs[i] = G[tok_idx(b, t0 + rr, h, e, T, H, E)];
        k2s[i] = r < n ? to_f(k2[tok_idx(b, t0 + r, h, e, T, H, E)]) : 0.f;
        q2s[i] = r < n ? to_f(q2[tok_idx(b, t0 + r, h, e, T, H, E)]) : 0.f;
    }
    for (int r = tid; r < kChunk; r += blockDim.x)
        bs[r] = r < n ? (beta ? beta[(size_t(b) * T + t0 + r) * H + h] : 1.f) : 0.f;
    __syncthreads();

    const size_t mat = ((size_t(b) * H + h) * NT + c) * (kChunk * kChunk);
    for (int i = tid; i < kChunk * kChunk; i += blockDim.x) {
        int r = i >> 6, s = i & 63;
        float a = 0.f, l = 0.f;
        if (r >= s) {
            float qk = 0.f, kk = 0.f;
            for (int d = 0; d < dk; ++d) {
                float ksd = Ks[s * DKP + d];
                qk = fmaf(Qs[r * DKP + d], ksd, qk);
                kk = fmaf(Ks[r * DKP + d], ksd, kk);
            }
            float R = 0.f, Rq = 0.f;
            for (int e = 0; e < E; ++e) {
                // exp of a non-positive difference of accumulated log gates
                float gam = expf(Gs[r * E + e] - Gs[s * E + e]);
                float ks2 = k2s[s * E + e] * gam;
                R = fmaf(k2s[r * E + e], ks2, R);
                Rq = fmaf(q2s[r * E + e], ks2, Rq);
            }
            a = qk * Rq;
            if (r > s) l = bs[r] * kk * R;
        }
        Aout[mat + i] = a;
        As[r * 65 + s] = a;
        Ls[r * 65 + s] = l;
    }
    __syncthreads();
    if (use_delta) {
        // Forward substitution, one row at a time: X[r][s] = delta_rs - sum_{j<r} L[r][j] X[j][s].
        const int s = tid & 63, pp = tid >> 6;  // 4 partial sums per column
        for (int r = 0; r < kChunk; ++r) {
            float acc = 0.f;
            for (int j = pp; j < r; j += 4) acc = fmaf(Ls[r * 65 + j], Xs[j * 65 + s], acc);
            part[pp * 64 + s] = acc;
            __syncthreads();
            if (pp == 0) {
                float x = (r == s ? 1.f : 0.f) - ((part[s] + part[64 + s]) + (part[128 + s] + part[192 + s]));
                Xs[r * 65 + s] = x;
            }
            __syncthreads();
        }
        for (int i = tid; i < kChunk * kChunk; i += blockDim.x) Nout[mat + i] = Xs[(i >> 6) * 65 + (i & 63)];
    }
}

static size_t prep_smem(const tla_problem& p) {
    return sizeof(float) * (2 * kChunk * (p.dk + 1) + 3 * kChunk * p.E + kChunk + 3 * kChunk * 65 + 256);
}

cudaError_t launch_chunk_prep(const tla_problem& p, const float* G, float* A, float* N,
                              cudaStream_t s) {
    int NT = (p.T + kChunk - 1) / kChunk;
    dim3 grid(NT, p.H, p.B);
    size_t smem = prep_smem(p);
    prof_before("chunk_prep_simt", s);
    if (p.dtype == TLA_BF16) {
        auto kern = chunk_prep_kernel<__nv_bfloat16>;
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        kern<<<grid, 256, smem, s>>>((const __nv_bfloat16*)p.q, (const __nv_bfloat16*)p.k,
                                     (const __nv_bfloat16*)p.q2, (const __nv_bfloat16*)p.k2, G,
                                     p.beta, A, N, p.T, p.H, p.dk, p.E, p.use_delta);
    } else {
        auto kern = chunk_prep_kernel<float>;
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        kern<<<grid, 256, smem, s>>>((const float*)p.q, (const float*)p.k, (const float*)p.q2,
                                     (const float*)p.k2, G, p.beta, A, N, p.T, p.H, p.dk, p.E,
                                     p.use_delta);
    }
    prof_after(s);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Recurrence over chunks for one (b, h, block of tv value columns).
//   a_e[r] = k'_{r,e} gamma_{r,e},  b_e[r] = q'_{r,e} gamma_{r,e},
//   w_e[r] = k'_{r,e} gamma^C_e / gamma_{r,e}
//   Res = V - sum_e diag(a_e) K S_e       (delta rule; sGLA: U = diag(beta) V)
//   U   = N diag(beta) Res
//   O   = sum_e diag(b_e) Q S_e + A U
//   S_e = gamma^C_e S_e + K^T diag(w_e) U
template <typename Tin>
__global__ void __launch_bounds__(256)
fwd_recurrence_kernel(const Tin* __restrict__ q, const Tin* __restrict__ k,
                      const Tin* __restrict__ v, const Tin* __restrict__ q2,
                      const Tin* __restrict__ k2, const float* __restrict__ G,
                      const float* __restrict__ beta, const float* __restrict__ h0,
                      const float* __restrict__ Amat, const float* __restrict__ Nmat,
                      void* __restrict__ o, float* __restrict__ ht, float* __restrict__ Sck,
                      float* __restrict__ Ubuf, float* __restrict__ Rbuf, int T, int H, int dk,
                      int dv, int E, int tv, int use_delta, int save, int out_f32) {
    const int nb = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
    const int n0 = nb * tv;
    const int tid = threadIdx.x;
    const int NT = (T + kChunk - 1) / kChunk;
    const int DKP = dk + 1, TVP = tv + 1;
    const int SE = dk * tv;  // one slice of the slab
    extern __shared__ float sm[];
    float* Ss = sm;                        // [E][dk][tv]
    float* Ks = Ss + E * SE;               // [64][DKP]
    float* Qs = Ks + kChunk * DKP;
    float* Vs = Qs + kChunk * DKP;         // [64][TVP]
    float* Rs = Vs + kChunk * TVP;         // residual
    float* Us = Rs + kChunk * TVP;
    float* Os = Us + kChunk * TVP;         // inter-chunk part of O
    float* As = Os + kChunk * TVP;         // [64][65]
    float* Ns = As + kChunk * 65;          // [64][65]
    float* ae = Ns + kChunk * 65;          // [64][E]
    float* be = ae + kChunk * E;
    float* we = be + kChunk * E;
    float* bs = we + kChunk * E;           // [64]
    float* gc = bs + kChunk;               // [E] gamma^C

    const size_t head_state = (size_t(b) * H + h) * E;
    for (int i = tid; i < E * SE; i += blockDim.x) {
        int e = i / SE, rem = i % SE, d = rem / tv, nn = rem % tv;
        Ss[i] = h0 ? h0[((head_state + e) * dk + d) * dv + n0 + nn] : 0.f;
    }

    for (int c = 0; c < NT; ++c) {
        const int t0 = c * kChunk;
        const int n = min(kChunk, T - t0);
        __syncthreads();  // previous chunk finished with every buffer
        for (int i = tid; i < kChunk * dk; i += blockDim.x) {
            int r = i / dk, d = i % dk;
            float kv = 0.f, qv = 0.f;
            if (r < n) {
                kv = to_f(k[tok_idx(b, t0 + r, h, d, T, H, dk)]);
                qv = to_f(q[tok_idx(b, t0 + r, h, d, T, H, dk)]);
            }
            Ks[r * DKP + d] = kv;
            Qs[r * DKP + d] = qv;
        }
        for (int i = tid; i < kChunk * tv; i += blockDim.x) {
            int r = i / tv, nn = i % tv;
            Vs[r * TVP + nn] = r < n ? to_f(v[tok_idx(b, t0 + r, h, n0 + nn, T, H, dv)]) : 0.f;
        }
        for (int i = tid; i < kChunk * E; i += blockDim.x) {
            int r = i / E, e = i % E;
            int rr = r < n ? r : n - 1;
            float Gr = G[tok_idx(b, t0 + rr, h, e, T, H, E)];
            float GC = G[tok_idx(b, t0 + n - 1, h, e, T, H, E)];
            float kk2 = r < n ? to_f(k2[tok_idx(b, t0 + r, h, e, T, H, E)]) : 0.f;
            float qq2 = r < n ? to_f(q2[tok_idx(b, t0 + r, h, e, T, H, E)]) : 0.f;
            float gam = expf(Gr);
            ae[i] = kk2 * gam;
            be[i] = qq2 * gam;
            we[i] = kk2 * expf(GC - Gr);
            if (r == 0) gc[e] = expf(GC);
        }
        for (int r = tid; r < kChunk; r += blockDim.x)
            bs[r] = r < n ? (beta ? beta[(size_t(b) * T + t0 + r) * H + h] : 1.f) : 0.f;
        const size_t mat = ((size_t(b) * H + h) * NT + c) * (kChunk * kChunk);
        for (int i = tid; i < kChunk * kChunk; i += blockDim.x) {
            As[(i >> 6) * 65 + (i & 63)] = Amat[mat + i];
            if (use_delta) Ns[(i >> 6) * 65 + (i & 63)] = Nmat[mat + i];
        }
        __syncthreads();

        // chunk-start state to the backward's checkpoint
        if (save) {
            size_t base = ((size_t(b) * H + h) * NT + c) * E;
            for (int i = tid; i < E * SE; i += blockDim.x) {
                int e = i / SE, rem = i % SE, d = rem / tv, nn = rem % tv;
                Sck[((base + e) * dk + d) * dv + n0 + nn] = Ss[i];
            }
        }
        // W (keys) and the inter-chunk read (queries) against the chunk-start state
        for (int i = tid; i < kChunk * tv; i += blockDim.x) {
            int r = i / tv, nn = i % tv;
            float w = 0.f, oi = 0.f;
            for (int e = 0; e < E; ++e) {
                const float* Se = Ss + e * SE + nn;
                float sk = 0.f, sq = 0.f;
                for (int d = 0; d < dk; ++d) {
                    float sv = Se[d * tv];
                    sk = fmaf(Ks[r * DKP + d], sv, sk);
                    sq = fmaf(Qs[r * DKP + d], sv, sq);
                }
                w = fmaf(ae[r * E + e], sk, w);
                oi = fmaf(be[r * E + e], sq, oi);
            }
            Rs[r * TVP + nn] = use_delta ? Vs[r * TVP + nn] - w : Vs[r * TVP + nn];
            Os[r * TVP + nn] = oi;
        }
        __syncthreads();
        // U = N diag(beta) Res  (sGLA: diag(beta) V)
        for (int i = tid; i < kChunk * tv; i += blockDim.x) {
            int r = i / tv, nn = i % tv;
            float u;
            if (use_delta) {
                u = 0.f;
                for (int s2 = 0; s2 <= r; ++s2) u = fmaf(Ns[r * 65 + s2] * bs[s2], Rs[s2 * TVP + nn], u);
            } else {
                u = bs[r] * Vs[r * TVP + nn];
            }
            Us[r * TVP + nn] = u;
            if (save && r < n) {
                Ubuf[tok_idx(b, t0 + r, h, n0 + nn, T, H, dv)] = u;
                if (use_delta) Rbuf[tok_idx(b, t0 + r, h, n0 + nn, T, H, dv)] = Rs[r * TVP + nn];
            }
        }
        __syncthreads();
        // O = inter + A U
        for (int i = tid; i < kChunk * tv; i += blockDim.x) {
            int r = i / tv, nn = i % tv;
            if (r >= n) continue;
            float acc = Os[r * TVP + nn];
            for (int s2 = 0; s2 <= r; ++s2) acc = fmaf(As[r * 65 + s2], Us[s2 * TVP + nn], acc);
            store_out(o, tok_idx(b, t0 + r, h, n0 + nn, T, H, dv), acc, out_f32);
        }
        // S_e = gamma^C_e S_e + K^T diag(w_e) U
        for (int i = tid; i < E * SE; i += blockDim.x) {
            int e = i / SE, rem = i % SE, d = rem / tv, nn = rem % tv;
            float acc = 0.f;
            for (int r = 0; r < n; ++r) acc = fmaf(Ks[r * DKP + d] * we[r * E + e], Us[r * TVP + nn], acc);
            Ss[i] = fmaf(gc[e], Ss[i], acc);
        }
    }
    __syncthreads();
    if (ht) {
        for (int i = tid; i < E * SE; i += blockDim.x) {
            int e = i / SE, rem = i % SE, d = rem / tv, nn = rem % tv;
            ht[((head_state + e) * dk + d) * dv + n0 + nn] = Ss[i];
        }
    }
}

static size_t fwd_smem(const tla_problem& p, int tv) {
    return sizeof(float) * ((size_t)p.E * p.dk * tv + 2 * kChunk * (p.dk + 1) +
                            4 * kChunk * (tv + 1) + 2 * kChunk * 65 + 3 * kChunk * p.E + kChunk +
                            p.E);
}

cudaError_t launch_fwd_recurrence(const tla_problem& p, const FwdPlan& fp, char* ws,
                                  int save_for_bwd, cudaStream_t s) {
    const int tv = fp.tv;
    dim3 grid(p.dv / tv, p.H, p.B);
    size_t smem = fwd_smem(p, tv);
    const float* G = (const float*)(ws + fp.G);
    const float* A = (const float*)(ws + fp.A);
    const float* N = p.use_delta ? (const float*)(ws + fp.N) : nullptr;
    float* Sck = save_for_bwd ? (float*)(ws + fp.S) : nullptr;
    float* U = save_for_bwd ? (float*)(ws + fp.U) : nullptr;
    float* R = (save_for_bwd && p.use_delta) ? (float*)(ws + fp.Res) : nullptr;
    prof_before("fwd_recurrence_simt", s);
    if (p.dtype == TLA_BF16) {
        using Tb = __nv_bfloat16;
        auto kern = fwd_recurrence_kernel<Tb>;
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        kern<<<grid, 256, smem, s>>>((const Tb*)p.q, (const Tb*)p.k, (const Tb*)p.v,
                                     (const Tb*)p.q2, (const Tb*)p.k2, G, p.beta, p.h0, A, N,
                                     p.o, p.ht, Sck, U, R, p.T, p.H, p.dk, p.dv, p.E, tv,
                                     p.use_delta, save_for_bwd, p.out_dtype == TLA_FP32);
    } else {
        auto kern = fwd_recurrence_kernel<float>;
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        kern<<<grid, 256, smem, s>>>((const float*)p.q, (const float*)p.k, (const float*)p.v,
                                     (const float*)p.q2, (const float*)p.k2, G, p.beta, p.h0, A,
                                     N, p.o, p.ht, Sck, U, R, p.T, p.H, p.dk, p.dv, p.E,
                                     tv, p.use_delta, save_for_bwd, p.out_dtype == TLA_FP32);
    }
    prof_after(s);
    return cudaGetLastError();
}

}  // namespace tla
