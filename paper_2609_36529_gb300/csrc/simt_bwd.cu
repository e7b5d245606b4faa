// SIMT (fp32 CUDA-core) kernels of the chunkwise backward (Appendix A, Kernels).
// The backward first walks the chunks in reverse to obtain the gradient of every
// state slice at each chunk boundary, then derives all other gradients with one
// independent CTA per chunk.  Reductions run in a fixed order and use no
// floating-point atomics, so repeated runs give identical bits.
//
// Forward chunk step being differentiated (per chunk, per value column block):
//   a_e = k'_e (.) gamma_e,  b_e = q'_e (.) gamma_e,  w_e = k'_e (.) gamma^C_e / gamma_e
//   Res = V - sum_e diag(a_e) K S_e   (sGLA: Res = V)
//   U   = T Res,  T = N diag(beta),  N = (I + L)^{-1},
//   L   = tril(diag(beta)(K K^T (.) R), -1)               (sGLA: T = diag(beta))
//   O   = sum_e diag(b_e) Q S_e + A U,  A = (Q K^T) (.) R'
//   S'_e = gamma^C_e S_e + K^T diag(w_e) U
// Reverse recurrence (bwd_recurrence_kernel), given dS' = dL/dS'_e:
//   dU   = A^T dO + sum_e diag(w_e) K dS'_e
//   dRes = T^T dU            (this is dV)
//   dS_e = gamma^C_e dS'_e + Q^T diag(b_e) dO - K^T diag(a_e) dRes
// Chunk-parallel gradients (bwd_chunk_grads_kernel): see the kernel.
#include "common.cuh"
#include "internal.h"

namespace tla {

template <typename Tin>
__global__ void __launch_bounds__(256)
bwd_recurrence_kernel(const Tin* __restrict__ q, const Tin* __restrict__ k,
                      const Tin* __restrict__ q2, const Tin* __restrict__ k2,
                      const float* __restrict__ G, const float* __restrict__ beta,
                      const float* __restrict__ Amat, const float* __restrict__ Nmat,
                      const Tin* __restrict__ dO, const float* __restrict__ dht,
                      void* __restrict__ dv_out, float* __restrict__ dh0,
                      float* __restrict__ dUbuf, float* __restrict__ dRbuf,
                      float* __restrict__ dSck, int T, int H, int dk, int dv, int E, int tv,
                      int use_delta, int out_f32) {
    const int nb = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
    const int n0 = nb * tv;
    const int tid = threadIdx.x;
    const int NT = (T + kChunk - 1) / kChunk;
    const int DKP = dk + 1, TVP = tv + 1;
    const int SE = dk * tv;
    extern __shared__ float sm[];
    float* dSs = sm;                       // [E][dk][tv]
    float* Ks = dSs + E * SE;
    float* Qs = Ks + kChunk * DKP;
    float* dOs = Qs + kChunk * DKP;        // [64][TVP]
    float* dUs = dOs + kChunk * TVP;
    float* dRs = dUs + kChunk * TVP;
    float* As = dRs + kChunk * TVP;        // [64][65]
    float* Ns = As + kChunk * 65;
    float* ae = Ns + kChunk * 65;
    float* be = ae + kChunk * E;
    float* we = be + kChunk * E;
    float* bs = we + kChunk * E;
    float* gc = bs + kChunk;

    const size_t head_state = (size_t(b) * H + h) * E;
    for (int i = tid; i < E * SE; i += blockDim.x) {
        int e = i / SE, rem = i % SE, d = rem / tv, nn = rem % tv;
        dSs[i] = dht ? dht[((head_state + e) * dk + d) * dv + n0 + nn] : 0.f;
    }
    for (int c = NT - 1; c >= 0; --c) {
        const int t0 = c * kChunk;
        const int n = min(kChunk, T - t0);
        __syncthreads();
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
            dOs[r * TVP + nn] = r < n ? to_f(dO[tok_idx(b, t0 + r, h, n0 + nn, T, H, dv)]) : 0.f;
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
        // gradient of the state at the end of chunk c, kept for the chunk-parallel pass
        {
            size_t base = ((size_t(b) * H + h) * NT + c) * E;
            for (int i = tid; i < E * SE; i += blockDim.x) {
                int e = i / SE, rem = i % SE, d = rem / tv, nn = rem % tv;
                dSck[((base + e) * dk + d) * dv + n0 + nn] = dSs[i];
            }
        }
        // dU = A^T dO + sum_e diag(w_e) K dS'_e
        for (int i = tid; i < kChunk * tv; i += blockDim.x) {
            int r = i / tv, nn = i % tv;
            float acc = 0.f;
            for (int s2 = r; s2 < kChunk; ++s2) acc = fmaf(As[s2 * 65 + r], dOs[s2 * TVP + nn], acc);
            for (int e = 0; e < E; ++e) {
                const float* dSe = dSs + e * SE + nn;
                float sk = 0.f;
                for (int d = 0; d < dk; ++d) sk = fmaf(Ks[r * DKP + d], dSe[d * tv], sk);
                acc = fmaf(we[r * E + e], sk, acc);
            }
            dUs[r * TVP + nn] = acc;
        }
        __syncthreads();
        // dRes = T^T dU = diag(beta) N^T dU   (sGLA: diag(beta) dU)
        for (int i = tid; i < kChunk * tv; i += blockDim.x) {
            int r = i / tv, nn = i % tv;
            float acc;
            if (use_delta) {
                acc = 0.f;
                for (int s2 = r; s2 < kChunk; ++s2) acc = fmaf(Ns[s2 * 65 + r], dUs[s2 * TVP + nn], acc);
                acc *= bs[r];
            } else {
                acc = bs[r] * dUs[r * TVP + nn];
            }
            dRs[r * TVP + nn] = acc;
            if (r < n) {
                size_t off = tok_idx(b, t0 + r, h, n0 + nn, T, H, dv);
                dUbuf[off] = dUs[r * TVP + nn];
                dRbuf[off] = acc;
                store_out(dv_out, off, acc, out_f32);
            }
        }
        __syncthreads();
        // dS_e = gamma^C_e dS'_e + Q^T diag(b_e) dO - K^T diag(a_e) dRes
        for (int i = tid; i < E * SE; i += blockDim.x) {
            int e = i / SE, rem = i % SE, d = rem / tv, nn = rem % tv;
            float acc = 0.f;
            for (int r = 0; r < n; ++r) {
                acc = fmaf(Qs[r * DKP + d] * be[r * E + e], dOs[r * TVP + nn], acc);
                if (use_delta) acc = fmaf(-Ks[r * DKP + d] * ae[r * E + e], dRs[r * TVP + nn], acc);
            }
            dSs[i] = fmaf(gc[e], dSs[i], acc);
        }
    }
    __syncthreads();
    if (dh0) {
        for (int i = tid; i < E * SE; i += blockDim.x) {
            int e = i / SE, rem = i % SE, d = rem / tv, nn = rem % tv;
            dh0[((head_state + e) * dk + d) * dv + n0 + nn] = dSs[i];
        }
    }
}

static size_t bwd_rec_smem(const tla_problem& p, int tv) {
    return sizeof(float) * ((size_t)p.E * p.dk * tv + 2 * kChunk * (p.dk + 1) +
                            3 * kChunk * (tv + 1) + 2 * kChunk * 65 + 3 * kChunk * p.E + kChunk +
                            p.E);
}

cudaError_t launch_bwd_recurrence(const tla_problem& p, const FwdPlan& fp, const char* fws,
                                  const BwdPlan& bp, char* bws, const void* dO,
                                  const float* dht, void* dv, float* dh0, cudaStream_t s) {
    const int tv = bp.tv;
    dim3 grid(p.dv / tv, p.H, p.B);
    size_t smem = bwd_rec_smem(p, tv);
    const float* G = (const float*)(fws + fp.G);
    const float* A = (const float*)(fws + fp.A);
    const float* N = p.use_delta ? (const float*)(fws + fp.N) : nullptr;
    float* dU = (float*)(bws + bp.dU);
    float* dR = (float*)(bws + bp.dRes);
    float* dS = (float*)(bws + bp.dS);
    prof_before("bwd_recurrence_simt", s);
    if (p.dtype == TLA_BF16) {
        using Tb = __nv_bfloat16;
        auto kern = bwd_recurrence_kernel<Tb>;
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        kern<<<grid, 256, smem, s>>>((const Tb*)p.q, (const Tb*)p.k, (const Tb*)p.q2,
                                     (const Tb*)p.k2, G, p.beta, A, N, (const Tb*)dO, dht,
                                     dv, dh0, dU, dR, dS, p.T, p.H, p.dk, p.dv, p.E, tv,
                                     p.use_delta, p.out_dtype == TLA_FP32);
    } else {
        auto kern = bwd_recurrence_kernel<float>;
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        kern<<<grid, 256, smem, s>>>((const float*)p.q, (const float*)p.k, (const float*)p.q2,
                                     (const float*)p.k2, G, p.beta, A, N, (const float*)dO, dht,
                                     dv, dh0, dU, dR, dS, p.T, p.H, p.dk, p.dv, p.E, tv,
                                     p.use_delta, p.out_dtype == TLA_FP32);
    }
    prof_after(s);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Chunk-parallel gradients, one CTA per (b, h, chunk).  With S = S_[c] (chunk
// start), dS' = gradient at the chunk's end, U, Res, dU, dRes of the chunk:
//   Z_e = dO S_e^T, Y_e = -dRes S_e^T, X_e = U dS'_e^T         (C x dk each)
//   dQ  = sum_e diag(b_e) Z_e + (dA (.) R') K
//   dK  = sum_e diag(a_e) Y_e + sum_e diag(w_e) X_e + (dA (.) R')^T Q + (dKK + dKK^T) K
//   db_e = rowdot(Q, Z_e), da_e = rowdot(K, Y_e), dw_e = rowdot(K, X_e)
//   dgamma^C_e = <dS'_e, S_e>_F
//   dA  = dO U^T (lower incl. diagonal), dR' = dA (.) Q K^T
//   dT  = dU Res^T;  dN = dT diag(beta);  dbeta_s += sum_r dT_rs N_rs
//   dM  = -N^T dN N^T;  dL = strictly-lower part of dM
//   dbeta_r += sum_s dL_rs (K K^T)_rs R_rs;  dKK = dL (.) beta_r R;  dR = dL (.) beta_r K K^T
//   (sGLA: T = diag(beta), dbeta_r = dT_rr)
// then the second keys/queries and log-decays through R, R', a, b, w, gamma^C,
// and finally dg = reverse cumulative sum of dG within the chunk.
template <typename Tin>
__global__ void __launch_bounds__(256)
bwd_chunk_grads_kernel(const Tin* __restrict__ q, const Tin* __restrict__ k,
                       const Tin* __restrict__ v, const Tin* __restrict__ q2,
                       const Tin* __restrict__ k2, const float* __restrict__ G,
                       const float* __restrict__ beta, const float* __restrict__ Nmat,
                       const float* __restrict__ Sck, const float* __restrict__ Ubuf,
                       const float* __restrict__ Rbuf, const Tin* __restrict__ dO,
                       const float* __restrict__ dUbuf, const float* __restrict__ dRbuf,
                       const float* __restrict__ dSck, void* __restrict__ dq,
                       void* __restrict__ dk_out, void* __restrict__ dq2, void* __restrict__ dk2,
                       float* __restrict__ dbeta, float* __restrict__ dg, int T, int H, int dk,
                       int dv, int E, int use_delta, int out_f32) {
    const int c = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
    const int NT = gridDim.x;
    const int tid = threadIdx.x;
    const int t0 = c * kChunk;
    const int n = min(kChunk, T - t0);
    constexpr int MP = 65;
    extern __shared__ float sm[];
    float* B0 = sm;                      // N
    float* B1 = B0 + kChunk * MP;        // dN -> dR
    float* B2 = B1 + kChunk * MP;        // dT (.) N -> dR'
    float* B3 = B2 + kChunk * MP;        // F -> P
    float* B4 = B3 + kChunk * MP;        // dKK (strictly lower)
    float* B5 = B4 + kChunk * MP;        // row terms of dbeta
    float* t1 = B5 + kChunk * MP;        // [64][33] tiles
    float* t2 = t1 + kChunk * 33;
    float* t3 = t2 + kChunk * 33;
    float* t4 = t3 + kChunk * 33;
    float* t5 = t4 + kChunk * 33;        // [32][33]
    float* t6 = t5 + 32 * 33;
    float* Gs = t6 + 32 * 33;            // [64][E]
    float* k2s = Gs + kChunk * E;
    float* q2s = k2s + kChunk * E;
    float* dbq = q2s + kChunk * E;       // db_e  [64][E]
    float* dak = dbq + kChunk * E;       // da_e
    float* dwk = dak + kChunk * E;       // dw_e
    float* dk2a = dwk + kChunk * E;      // accumulators through R, R'
    float* dq2a = dk2a + kChunk * E;
    float* dGa = dq2a + kChunk * E;
    float* bs = dGa + kChunk * E;        // [64]
    float* dba = bs + kChunk;            // dbeta accumulator [64]
    float* dgc = dba + kChunk;           // [E] d gamma^C (Frobenius products)
    float* red = dgc + 32;               // [256]

    for (int i = tid; i < kChunk * E; i += blockDim.x) {
        int r = i / E, e = i % E;
        int rr = r < n ? r : n - 1;
        Gs[i] = G[tok_idx(b, t0 + rr, h, e, T, H, E)];
        k2s[i] = r < n ? to_f(k2[tok_idx(b, t0 + r, h, e, T, H, E)]) : 0.f;
        q2s[i] = r < n ? to_f(q2[tok_idx(b, t0 + r, h, e, T, H, E)]) : 0.f;
        dbq[i] = dak[i] = dwk[i] = 0.f;
    }
    for (int r = tid; r < kChunk; r += blockDim.x) {
        bs[r] = r < n ? (beta ? beta[(size_t(b) * T + t0 + r) * H + h] : 1.f) : 0.f;
        dba[r] = 0.f;
    }
    if (tid < 32) dgc[tid] = 0.f;
    const size_t mat = ((size_t(b) * H + h) * NT + c) * (kChunk * kChunk);
    if (use_delta)
        for (int i = tid; i < kChunk * kChunk; i += blockDim.x) B0[(i >> 6) * MP + (i & 63)] = Nmat[mat + i];

    // ---- phase A: C x C quantities; thread owns entries (r = tid/64 + 4j, s = tid%64)
    float dA[16], dT[16], QK[16], KK[16];
#pragma unroll
    for (int j = 0; j < 16; ++j) dA[j] = dT[j] = QK[j] = KK[j] = 0.f;
    const int s_own = tid & 63, r_base = tid >> 6;
    for (int n0 = 0; n0 < dv; n0 += 32) {
        __syncthreads();
        for (int i = tid; i < kChunk * 32; i += blockDim.x) {
            int r = i >> 5, nn = i & 31;
            bool ok = r < n && n0 + nn < dv;
            size_t off = tok_idx(b, t0 + r, h, n0 + nn, T, H, dv);
            t1[r * 33 + nn] = ok ? to_f(dO[off]) : 0.f;
            t2[r * 33 + nn] = ok ? Ubuf[off] : 0.f;
            t3[r * 33 + nn] = ok ? dUbuf[off] : 0.f;
            t4[r * 33 + nn] = ok ? (use_delta ? Rbuf[off] : to_f(v[off])) : 0.f;
        }
        __syncthreads();
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            int r = r_base + 4 * j;
            float a = dA[j], t = dT[j];
            for (int nn = 0; nn < 32; ++nn) {
                a = fmaf(t1[r * 33 + nn], t2[s_own * 33 + nn], a);
                t = fmaf(t3[r * 33 + nn], t4[s_own * 33 + nn], t);
            }
            dA[j] = a;
            dT[j] = t;
        }
    }
    for (int d0 = 0; d0 < dk; d0 += 32) {
        __syncthreads();
        for (int i = tid; i < kChunk * 32; i += blockDim.x) {
            int r = i >> 5, dd = i & 31;
            bool ok = r < n && d0 + dd < dk;
            size_t off = tok_idx(b, t0 + r, h, d0 + dd, T, H, dk);
            t1[r * 33 + dd] = ok ? to_f(q[off]) : 0.f;
            t2[r * 33 + dd] = ok ? to_f(k[off]) : 0.f;
        }
        __syncthreads();
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            int r = r_base + 4 * j;
            float a = QK[j], t = KK[j];
            for (int dd = 0; dd < 32; ++dd) {
                float ks = t2[s_own * 33 + dd];
                a = fmaf(t1[r * 33 + dd], ks, a);
                t = fmaf(t2[r * 33 + dd], ks, t);
            }
            QK[j] = a;
            KK[j] = t;
        }
    }
    // R, R' for the owned entries
    float Rv[16], Rq[16];
#pragma unroll
    for (int j = 0; j < 16; ++j) {
        int r = r_base + 4 * j, s = s_own;
        float R = 0.f, Q = 0.f;
        if (r >= s)
            for (int e = 0; e < E; ++e) {
                float gam = expf(Gs[r * E + e] - Gs[s * E + e]);
                float ks2 = k2s[s * E + e] * gam;
                R = fmaf(k2s[r * E + e], ks2, R);
                Q = fmaf(q2s[r * E + e], ks2, Q);
            }
        Rv[j] = R;
        Rq[j] = Q;
    }
    __syncthreads();
    if (use_delta) {
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            int r = r_base + 4 * j, s = s_own;
            float Nrs = B0[r * MP + s];
            B1[r * MP + s] = dT[j] * bs[s];      // dN
            B2[r * MP + s] = dT[j] * Nrs;        // column terms of dbeta
        }
        __syncthreads();
        if (tid < kChunk) {
            float acc = 0.f;
            for (int r = 0; r < kChunk; ++r) acc += B2[r * MP + tid];
            dba[tid] += acc;
        }
        // F = dN N^T
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            int r = r_base + 4 * j, s = s_own;
            float acc = 0.f;
            for (int x = 0; x < kChunk; ++x) acc = fmaf(B1[r * MP + x], B0[s * MP + x], acc);
            B3[r * MP + s] = acc;
        }
        __syncthreads();
        float dL[16];
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            int r = r_base + 4 * j, s = s_own;
            float acc = 0.f;
            for (int x = 0; x < kChunk; ++x) acc = fmaf(B0[x * MP + r], B3[x * MP + s], acc);
            dL[j] = (r > s) ? -acc : 0.f;
        }
        __syncthreads();
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            int r = r_base + 4 * j, s = s_own;
            B1[r * MP + s] = dL[j] * bs[r] * KK[j];   // dR (strictly lower)
            B4[r * MP + s] = dL[j] * bs[r] * Rv[j];   // dKK
            B5[r * MP + s] = dL[j] * KK[j] * Rv[j];   // row terms of dbeta
        }
    } else {
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            int r = r_base + 4 * j, s = s_own;
            B1[r * MP + s] = 0.f;
            B4[r * MP + s] = 0.f;
            B5[r * MP + s] = (r == s) ? dT[j] : 0.f;  // T = diag(beta): dbeta_r = dT_rr
        }
    }
#pragma unroll
    for (int j = 0; j < 16; ++j) {
        int r = r_base + 4 * j, s = s_own;
        bool low = r >= s;
        B2[r * MP + s] = low ? dA[j] * QK[j] : 0.f;   // dR'
        B3[r * MP + s] = low ? dA[j] * Rq[j] : 0.f;   // P = dA (.) R'
    }
    __syncthreads();
    if (tid < kChunk) {
        float acc = 0.f;
        for (int s = 0; s < kChunk; ++s) acc += B5[tid * MP + s];
        dba[tid] += acc;
    }
    // second keys / queries / log decays through R (dR in B1) and R' (dR' in B2)
    for (int i = tid; i < kChunk * E; i += blockDim.x) {
        int x = i / E, e = i % E;
        float gx = Gs[x * E + e], kx = k2s[x * E + e], qx = q2s[x * E + e];
        float dk2v = 0.f, dq2v = 0.f, dGv = 0.f;
        for (int s = 0; s <= x; ++s) {  // x as the row index r >= s
            float gam = expf(gx - Gs[s * E + e]);
            float ks = k2s[s * E + e];
            float dR = B1[x * MP + s], dRq = B2[x * MP + s];
            dk2v = fmaf(dR * ks, gam, dk2v);
            dq2v = fmaf(dRq * ks, gam, dq2v);
            dGv = fmaf((dR * kx + dRq * qx) * ks, gam, dGv);
        }
        for (int r = x; r < kChunk; ++r) {  // x as the column index s <= r
            float gam = expf(Gs[r * E + e] - gx);
            float dR = B1[r * MP + x], dRq = B2[r * MP + x];
            float t = (dR * k2s[r * E + e] + dRq * q2s[r * E + e]) * gam;
            dk2v = fmaf(t, 1.f, dk2v);
            dGv = fmaf(-t, kx, dGv);
        }
        dk2a[i] = dk2v;
        dq2a[i] = dq2v;
        dGa[i] = dGv;
    }

    // ---- phase B: E-fold products with the chunk-start state and the end-of-chunk gradient
    const size_t sbase = ((size_t(b) * H + h) * NT + c) * E;
    for (int d0 = 0; d0 < dk; d0 += 32) {
        __syncthreads();
        for (int i = tid; i < kChunk * 32; i += blockDim.x) {
            int r = i >> 5, dd = i & 31;
            bool ok = r < n && d0 + dd < dk;
            size_t off = tok_idx(b, t0 + r, h, d0 + dd, T, H, dk);
            t1[r * 33 + dd] = ok ? to_f(q[off]) : 0.f;
            t2[r * 33 + dd] = ok ? to_f(k[off]) : 0.f;
        }
        // thread owns (r = tid/32 + 8j, dd = tid%32), j < 8
        const int dd = tid & 31, rb = tid >> 5;
        float accq[8], acck[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) accq[j] = acck[j] = 0.f;
        for (int e = 0; e < E; ++e) {
            float zs[8], ys[8], xs[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) zs[j] = ys[j] = xs[j] = 0.f;
            float fro = 0.f;
            for (int n0 = 0; n0 < dv; n0 += 32) {
                __syncthreads();
                for (int i = tid; i < kChunk * 32; i += blockDim.x) {
                    int r = i >> 5, nn = i & 31;
                    bool ok = r < n && n0 + nn < dv;
                    size_t off = tok_idx(b, t0 + r, h, n0 + nn, T, H, dv);
                    t3[r * 33 + nn] = ok ? to_f(dO[off]) : 0.f;
                    t4[r * 33 + nn] = ok ? (use_delta ? dRbuf[off] : 0.f) : 0.f;
                    float uu = ok ? Ubuf[off] : 0.f;
                    // U goes into the first 64 rows of the two [32][33] tiles' neighbour:
                    // reuse B5 (free after phase A) as a [64][33] buffer
                    B5[r * 33 + nn] = uu;
                }
                for (int i = tid; i < 32 * 32; i += blockDim.x) {
                    int di = i >> 5, nn = i & 31;
                    bool ok = d0 + di < dk && n0 + nn < dv;
                    size_t off = ((sbase + e) * dk + d0 + di) * dv + n0 + nn;
                    t5[di * 33 + nn] = ok ? Sck[off] : 0.f;
                    t6[di * 33 + nn] = ok ? dSck[off] : 0.f;
                }
                __syncthreads();
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    int r = rb + 8 * j;
                    float z = zs[j], y = ys[j], x = xs[j];
                    for (int nn = 0; nn < 32; ++nn) {
                        float sv = t5[dd * 33 + nn], dsv = t6[dd * 33 + nn];
                        z = fmaf(t3[r * 33 + nn], sv, z);
                        y = fmaf(-t4[r * 33 + nn], sv, y);
                        x = fmaf(B5[r * 33 + nn], dsv, x);
                    }
                    zs[j] = z; ys[j] = y; xs[j] = x;
                }
                // Frobenius product <dS'_e, S_e> over this tile: thread covers 4 entries
                for (int i = tid; i < 32 * 32; i += blockDim.x) {
                    int di = i >> 5, nn = i & 31;
                    fro = fmaf(t6[di * 33 + nn], t5[di * 33 + nn], fro);
                }
            }
            // accumulate dQ, dK and the row dots db, da, dw (warp = one row r, lanes = dd)
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                int r = rb + 8 * j;
                float bq = 0.f, ak = 0.f, wk = 0.f;
                bq = q2s[r * E + e] * expf(Gs[r * E + e]);
                ak = k2s[r * E + e] * expf(Gs[r * E + e]);
                wk = k2s[r * E + e] * expf(Gs[(n - 1) * E + e] - Gs[r * E + e]);
                accq[j] = fmaf(bq, zs[j], accq[j]);
                acck[j] = fmaf(ak, ys[j], fmaf(wk, xs[j], acck[j]));
                float pb = t1[r * 33 + dd] * zs[j];
                float pa = t2[r * 33 + dd] * ys[j];
                float pw = t2[r * 33 + dd] * xs[j];
#pragma unroll
                for (int off = 16; off > 0; off >>= 1) {
                    pb += __shfl_xor_sync(0xffffffffu, pb, off);
                    pa += __shfl_xor_sync(0xffffffffu, pa, off);
                    pw += __shfl_xor_sync(0xffffffffu, pw, off);
                }
                if (dd == 0) {
                    dbq[r * E + e] += pb;
                    dak[r * E + e] += pa;
                    dwk[r * E + e] += pw;
                }
            }
            red[tid] = fro;
            __syncthreads();
            for (int st = 128; st > 0; st >>= 1) {
                if (tid < st) red[tid] += red[tid + st];
                __syncthreads();
            }
            if (tid == 0) dgc[e] += red[0];
        }
        // C x C contributions: dQ += P K, dK += P^T Q + (dKK + dKK^T) K
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            int r = rb + 8 * j;
            float aq = accq[j], ak = acck[j];
            for (int s = 0; s <= r; ++s) aq = fmaf(B3[r * MP + s], t2[s * 33 + dd], aq);
            for (int x = r; x < kChunk; ++x) ak = fmaf(B3[x * MP + r], t1[x * 33 + dd], ak);
            for (int s = 0; s < r; ++s) ak = fmaf(B4[r * MP + s], t2[s * 33 + dd], ak);
            for (int x = r + 1; x < kChunk; ++x) ak = fmaf(B4[x * MP + r], t2[x * 33 + dd], ak);
            if (r < n && d0 + dd < dk) {
                size_t off = tok_idx(b, t0 + r, h, d0 + dd, T, H, dk);
                store_out(dq, off, aq, out_f32);
                store_out(dk_out, off, ak, out_f32);
            }
        }
    }
    __syncthreads();
    // ---- phase C: assemble dq2, dk2, dG; gamma^C; reverse cumulative sum -> dg; dbeta
    for (int i = tid; i < kChunk * E; i += blockDim.x) {
        int e = i % E;
        float gam = expf(Gs[i]);
        float wdec = expf(Gs[(n - 1) * E + e] - Gs[i]);
        float a = k2s[i] * gam, bq = q2s[i] * gam, w = k2s[i] * wdec;
        dk2a[i] += dak[i] * gam + dwk[i] * wdec;
        dq2a[i] += dbq[i] * gam;
        dGa[i] += dak[i] * a + dbq[i] * bq - dwk[i] * w;
    }
    __syncthreads();
    if (tid < E) {
        const int e = tid;
        float dGC = 0.f;
        for (int r = 0; r < n; ++r) {
            float w = k2s[r * E + e] * expf(Gs[(n - 1) * E + e] - Gs[r * E + e]);
            dGC = fmaf(dwk[r * E + e], w, dGC);
        }
        dGC = fmaf(dgc[e], expf(Gs[(n - 1) * E + e]), dGC);
        dGa[(n - 1) * E + e] += dGC;
        float acc = 0.f;
        for (int r = n - 1; r >= 0; --r) {
            acc += dGa[r * E + e];
            dg[tok_idx(b, t0 + r, h, e, T, H, E)] = acc;
        }
    }
    for (int i = tid; i < n * E; i += blockDim.x) {
        int r = i / E, e = i % E;
        size_t off = tok_idx(b, t0 + r, h, e, T, H, E);
        store_out(dq2, off, dq2a[i], out_f32);
        store_out(dk2, off, dk2a[i], out_f32);
    }
    if (dbeta && tid < n) dbeta[(size_t(b) * T + t0 + tid) * H + h] = dba[tid];
}

// Gradient of a per-head gate: the sum over the slices of the per-slice gradient (fixed order).
__global__ void sum_slices_kernel(const float* __restrict__ src, float* __restrict__ dst,
                                  long long n, int E) {
    const long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x;
    if (i >= n) return;
    float acc = 0.f;
    for (int e = 0; e < E; ++e) acc += src[i * E + e];
    dst[i] = acc;
}

cudaError_t launch_sum_slices(const float* src, float* dst, long long n, int E, cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    const int threads = 256;
    prof_before("sum_slices", s);
    sum_slices_kernel<<<unsigned((n + threads - 1) / threads), threads, 0, s>>>(src, dst, n, E);
    prof_after(s);
    return cudaGetLastError();
}

static size_t grads_smem(const tla_problem& p) {
    return sizeof(float) * (6 * kChunk * 65 + 4 * kChunk * 33 + 2 * 32 * 33 + 9 * kChunk * p.E +
                            2 * kChunk + 32 + 256);
}

cudaError_t launch_bwd_chunk_grads(const tla_problem& p, const FwdPlan& fp, const char* fws,
                                   const BwdPlan& bp, const char* bws, const void* dO,
                                   void* dq, void* dk, void* dq2, void* dk2, float* dbeta,
                                   float* dg, cudaStream_t s) {
    int NT = (p.T + kChunk - 1) / kChunk;
    dim3 grid(NT, p.H, p.B);
    size_t smem = grads_smem(p);
    const float* G = (const float*)(fws + fp.G);
    const float* N = p.use_delta ? (const float*)(fws + fp.N) : nullptr;
    const float* S = (const float*)(fws + fp.S);
    const float* U = (const float*)(fws + fp.U);
    const float* R = p.use_delta ? (const float*)(fws + fp.Res) : nullptr;
    const float* dU = (const float*)(bws + bp.dU);
    const float* dR = (const float*)(bws + bp.dRes);
    const float* dS = (const float*)(bws + bp.dS);
    prof_before("bwd_chunk_grads_simt", s);
    if (p.dtype == TLA_BF16) {
        using Tb = __nv_bfloat16;
        auto kern = bwd_chunk_grads_kernel<Tb>;
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        kern<<<grid, 256, smem, s>>>((const Tb*)p.q, (const Tb*)p.k, (const Tb*)p.v,
                                     (const Tb*)p.q2, (const Tb*)p.k2, G, p.beta, N, S, U, R,
                                     (const Tb*)dO, dU, dR, dS, dq, dk, dq2, dk2, dbeta, dg, p.T,
                                     p.H, p.dk, p.dv, p.E, p.use_delta, p.out_dtype == TLA_FP32);
    } else {
        auto kern = bwd_chunk_grads_kernel<float>;
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        kern<<<grid, 256, smem, s>>>((const float*)p.q, (const float*)p.k, (const float*)p.v,
                                     (const float*)p.q2, (const float*)p.k2, G, p.beta, N, S, U,
                                     R, (const float*)dO, dU, dR, dS, dq, dk, dq2, dk2, dbeta, dg,
                                     p.T, p.H, p.dk, p.dv, p.E, p.use_delta,
                                     p.out_dtype == TLA_FP32);
    }
    prof_after(s);
    return cudaGetLastError();
}

}  // namespace tla
