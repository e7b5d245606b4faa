// Tensor-core (tcgen05) chunk-parallel gradients of the backward (Appendix A,
// Kernels: after the reverse recurrence, every chunk's remaining gradients are
// computed independently; fixed-order reductions, no floating-point atomics).
//
// One CTA of 8 warps per (b, h, chunk).  With S_e = chunk-start state, dS'_e =
// gradient of the state at the chunk's end, and U, Res, dU, dRes of the chunk:
//   dQ = sum_e diag(b_e) dO S_e^T + P K,                       P = dA (.) R'
//   dK = sum_e [diag(a_e) (-dRes) S_e^T + diag(w_e) U dS'_e^T] + (dKK + dKK^T) K + P^T Q
//   db_e = rowdot(dO, Q S_e), da_e = -rowdot(dRes, K S_e), dw_e = rowdot(U, K dS'_e)
//   dgamma^C_e = <dS'_e, S_e>_F
//   dA = dO U^T, dT = dU Res^T (sGLA: dU V^T), and the C x C algebra of the UT
//   transform (dN, F = dN N^T, dM = -N^T F, dL, dKK, dR, dR', dbeta).
// Tensor-core products (fp32 accumulation in TMEM, non-exact operands as bf16 hi/lo):
//   phase 0  [K;Q] K^T -> K K^T, Q K^T;  dO U^T -> dA;  dU Res^T -> dT   (M=64 for the last two)
//   phase 1  (CUDA cores) C x C algebra, then ACC = [[P, 0], [Kc, P^T]] [K; Q]
//   phase 2  per slice e:  ACC += [b_e dO ; -a_e dRes] S_e^T + [0 ; w_e U] dS'_e^T,
//            P_e = [K;Q] S_e, P'_e = [K;Q] dS'_e (the staged S tile is read K-major for
//            the first product and MN-major for the second)
//   phase 3  ACC rows 0-63 -> dq, rows 64-127 -> dk; second keys/queries, log gates, beta.
#include "common.cuh"
#include "internal.h"
#include "sm100.cuh"
#include "tc_common.cuh"
#include "tma_host.h"

namespace tla {
using namespace sm100;

namespace {

constexpr int kThreads = 256;
constexpr int kDk = 128;
constexpr int kBoxBytes = 64 * 64 * 2;
constexpr int MP = 65;                     // row stride of the fp32 C x C matrices
constexpr int kMatBytes = 64 * MP * 4;     // 16640

struct TcGradArgs {
    const __nv_bfloat16* q2;
    const __nv_bfloat16* k2;
    const __nv_bfloat16* v;
    const float* G;
    const float* beta;
    const float* Nmat;
    const float* Sck;
    const float* Ubuf;
    const float* Rbuf;
    const float* dUbuf;
    const float* dRbuf;
    const float* dSck;
    void* dq;
    void* dk;
    void* dq2;
    void* dk2;
    float* dbeta;
    float* dg;
    int* err;
    int T, H, dv, E, NT, use_delta, out_f32;
};

__device__ __forceinline__ void load_row8(const float* src, float* v) {
    const float4 a = reinterpret_cast<const float4*>(src)[0];
    const float4 c = reinterpret_cast<const float4*>(src)[1];
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = c.x; v[5] = c.y; v[6] = c.z; v[7] = c.w;
}

__device__ __forceinline__ void load_bf16x8(const uint8_t* src, float* v) {
    const uint4 u = *reinterpret_cast<const uint4*>(src);
    const __nv_bfloat162* p = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float2 f = __bfloat1622float2(p[i]);
        v[2 * i] = f.x;
        v[2 * i + 1] = f.y;
    }
}

__global__ void __launch_bounds__(kThreads, 1)
bwd_chunk_grads_tc_kernel(const __grid_constant__ CUtensorMap map_k,
                          const __grid_constant__ CUtensorMap map_q,
                          const __grid_constant__ CUtensorMap map_do, const TcGradArgs p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
    const int E = p.E, dv = p.dv, T = p.T, H = p.H, NT = p.NT;
    const int c = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
    const int t0 = c * 64, n = min(64, T - t0);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int T64 = 64 * dv * 2;               // bytes of a [64][dv] bf16 tile

    uint8_t* sKQ = sm;                         // [K rows | Q rows] x 2 blocks (TMA)
    uint8_t* sDO = sKQ + 4 * kBoxBytes;        // dO [64][dv] bf16 (TMA)
    uint8_t* sX = sDO + 2 * kBoxBytes;         // 64 KB work tiles
    uint8_t* sY = sX + 65536;                  // 64 KB work tiles
    float* Gs = reinterpret_cast<float*>(sY + 65536);
    float* k2s = Gs + 64 * E;
    float* q2s = k2s + 64 * E;
    float* dbq = q2s + 64 * E;
    float* dak = dbq + 64 * E;
    float* dwk = dak + 64 * E;
    float* dk2a = dwk + 64 * E;
    float* dq2a = dk2a + 64 * E;
    float* dGa = dq2a + 64 * E;
    float* bs = dGa + 64 * E;                  // [64]
    float* dba = bs + 64;                      // [64]
    float* dgc = dba + 64;                     // [16]
    float* red = dgc + 16;                     // [2][128] row-dot halves
    float* red2 = red + 256;                   // [256]

    __shared__ __align__(8) uint64_t bar_ld, bar_mma, bar_s, bar_d;
    __shared__ uint32_t tmem_slot;

    if (warp == 0) {
        tmem_alloc(&tmem_slot, 512);
        tmem_relinquish();
    }
    if (tid == 0) {
        mbar_init(&bar_ld, 1);
        mbar_init(&bar_mma, 1);
        mbar_init(&bar_s, 1);
        mbar_init(&bar_d, 1);
        fence_barrier_init();
        mbar_arrive_expect_tx(&bar_ld, 4 * kBoxBytes + (dv / 64) * kBoxBytes);
        for (int j = 0; j < 2; ++j) {
            tma_load_4d(sKQ + j * 2 * kBoxBytes, &map_k, &bar_ld, 64 * j, h, t0, b);
            tma_load_4d(sKQ + j * 2 * kBoxBytes + kBoxBytes, &map_q, &bar_ld, 64 * j, h, t0, b);
        }
        for (int j = 0; j < dv / 64; ++j) tma_load_4d(sDO + j * kBoxBytes, &map_do, &bar_ld, 64 * j, h, t0, b);
    }
    // small per-chunk arrays
    for (int i = tid; i < 64 * E; i += kThreads) {
        const int r = i / E, e = i - (i / E) * E;
        const int rr = r < n ? r : n - 1;
        Gs[i] = p.G[tok_idx(b, t0 + rr, h, e, T, H, E)];
        k2s[i] = r < n ? __bfloat162float(p.k2[tok_idx(b, t0 + r, h, e, T, H, E)]) : 0.f;
        q2s[i] = r < n ? __bfloat162float(p.q2[tok_idx(b, t0 + r, h, e, T, H, E)]) : 0.f;
        dbq[i] = dak[i] = dwk[i] = 0.f;
    }
    if (tid < 64) {
        bs[tid] = tid < n ? (p.beta ? p.beta[(size_t(b) * T + t0 + tid) * H + h] : 1.f) : 0.f;
        dba[tid] = 0.f;
    }
    if (tid < 16) dgc[tid] = 0.f;

    // ---- phase 0 staging: U -> sX (hi, lo); dU, Res (sGLA: V) -> sY (hi, lo, hi, lo)
    // (8-column chunks; consecutive threads take consecutive chunks of a row)
    for (int ci = tid; ci < 64 * (dv / 8); ci += kThreads) {
        const int r = ci / (dv / 8), cc = (ci % (dv / 8)) * 8;
        {
            float u[8], du[8], rs[8];
            if (r < n) {
                const size_t off = tok_idx(b, t0 + r, h, cc, T, H, dv);
                load_row8(p.Ubuf + off, u);
                load_row8(p.dUbuf + off, du);
                if (p.use_delta) {
                    load_row8(p.Rbuf + off, rs);
                } else {
                    for (int i = 0; i < 8; ++i) rs[i] = __bfloat162float(p.v[off + i]);
                }
            } else {
                for (int i = 0; i < 8; ++i) u[i] = du[i] = rs[i] = 0.f;
            }
            const uint32_t o = sw128_offset(r, cc, 64);
            st8_split(sX, sX + T64, o, u);
            st8_split(sY, sY + T64, o, du);
            st8_split(sY + 2 * T64, sY + 3 * T64, o, rs);
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;
    const uint32_t tACC = tmem, tP = tmem + 128, tP2 = tmem + 128 + dv;

    bool ok = mbar_wait(&bar_ld, 0);
    fence_proxy_async_smem();
    if (__syncthreads_or(!ok)) {
        if (tid == 0) record_device_error(p.err, TLA_ERR_TIMEOUT);
        __syncthreads();
        if (warp == 0) tmem_dealloc(tmem, 512);
        return;
    }
    uint32_t mph = 0;
    auto mma_wait = [&]() -> bool {
        const bool w = mbar_wait(&bar_mma, mph);
        mph ^= 1;
        return w;
    };

    // ---- phase 0 products
    if (tid == 0) {
        const uint32_t id_kq = idesc_bf16_f32(128, 64, 0, 0);
        for (int ks = 0; ks < kDk / 16; ++ks) {
            const uint64_t a = smem_desc(smem_u32(sKQ) + (ks >> 2) * 2 * kBoxBytes + (ks & 3) * 32, 16, 1024);
            umma_bf16(tmem + 128, a, a, id_kq, ks > 0 ? 1u : 0u);   // B = the key rows of the same tile
        }
        const uint32_t id64 = idesc_bf16_f32(64, 64, 0, 0);
        for (int ks = 0; ks < dv / 16; ++ks) {
            const uint32_t o = (ks >> 2) * kBoxBytes + (ks & 3) * 32;
            const uint64_t a = smem_desc(smem_u32(sDO) + o, 16, 1024);
            umma_bf16(tmem + 192, a, smem_desc(smem_u32(sX) + o, 16, 1024), id64, ks > 0 ? 1u : 0u);
            umma_bf16(tmem + 192, a, smem_desc(smem_u32(sX + T64) + o, 16, 1024), id64, 1u);
            const uint64_t uh = smem_desc(smem_u32(sY) + o, 16, 1024);
            const uint64_t ul = smem_desc(smem_u32(sY + T64) + o, 16, 1024);
            const uint64_t rh = smem_desc(smem_u32(sY + 2 * T64) + o, 16, 1024);
            const uint64_t rl = smem_desc(smem_u32(sY + 3 * T64) + o, 16, 1024);
            umma_bf16(tmem + 256, uh, rh, id64, ks > 0 ? 1u : 0u);
            umma_bf16(tmem + 256, uh, rl, id64, 1u);
            umma_bf16(tmem + 256, ul, rh, id64, 1u);
        }
        umma_commit(&bar_mma);
    }
    ok = mma_wait();
    if (__syncthreads_or(!ok)) {
        if (tid == 0) record_device_error(p.err, TLA_ERR_TIMEOUT);
        __syncthreads();
        if (warp == 0) tmem_dealloc(tmem, 512);
        return;
    }
    tc_fence_after();
    // TMEM -> fp32 C x C matrices (KK, QK in sX; dA, dT in sY)
    {
        float* MKK = reinterpret_cast<float*>(sX);
        float* MQK = reinterpret_cast<float*>(sX + kMatBytes);
        float* MdA = reinterpret_cast<float*>(sY);
        float* MdT = reinterpret_cast<float*>(sY + kMatBytes);
        const int wq = warp & 3, L = wq * 32 + lane;
        if (warp < 4) {
            float* dst = L < 64 ? MKK + L * MP : MQK + (L - 64) * MP;
            for (int j = 0; j < 64; j += 16) {
                float v[16];
                tmem_ld16(tmem_lane_addr(tmem + 128, warp, j), v);
                tmem_wait_ld();
                for (int i = 0; i < 16; ++i) dst[j + i] = v[i];
            }
        } else {
            const int r = 16 * wq + (lane & 15);
            for (int j = 0; j < 64; j += 16) {
                float va[16], vt[16];
                tmem_ld16(tmem_lane_addr(tmem + 192, warp, j), va);
                tmem_ld16(tmem_lane_addr(tmem + 256, warp, j), vt);
                tmem_wait_ld();
                if (lane < 16)
                    for (int i = 0; i < 16; ++i) {
                        MdA[r * MP + j + i] = va[i];
                        MdT[r * MP + j + i] = vt[i];
                    }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    const int s_own = tid & 63, r_base = tid >> 6;   // entries (r_base + 4j, s_own), j < 16
    float dA[16], dT[16], QK[16], KK[16];
    {
        const float* MKK = reinterpret_cast<const float*>(sX);
        const float* MQK = reinterpret_cast<const float*>(sX + kMatBytes);
        const float* MdA = reinterpret_cast<const float*>(sY);
        const float* MdT = reinterpret_cast<const float*>(sY + kMatBytes);
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            const int r = r_base + 4 * j;
            KK[j] = MKK[r * MP + s_own];
            QK[j] = MQK[r * MP + s_own];
            dA[j] = MdA[r * MP + s_own];
            dT[j] = MdT[r * MP + s_own];
        }
    }
    __syncthreads();

    // ---- phase 1: C x C algebra on CUDA cores
    float* B0 = reinterpret_cast<float*>(sX);
    float* B1 = reinterpret_cast<float*>(sX + kMatBytes);
    float* B2 = reinterpret_cast<float*>(sX + 2 * kMatBytes);
    float* B3 = reinterpret_cast<float*>(sY);
    float* B4 = reinterpret_cast<float*>(sY + kMatBytes);
    float* B5 = reinterpret_cast<float*>(sY + 2 * kMatBytes);
    const size_t mat = ((size_t(b) * H + h) * NT + c) * (64 * 64);
    if (p.use_delta)
        for (int i = tid; i < 64 * 64; i += kThreads) B0[(i >> 6) * MP + (i & 63)] = p.Nmat[mat + i];
    float Rv[16], Rq[16];
#pragma unroll
    for (int j = 0; j < 16; ++j) Rv[j] = Rq[j] = 0.f;
    for (int e = 0; e < E; ++e) {            // 16 independent entries per slice
        const float gs = Gs[s_own * E + e], ks = k2s[s_own * E + e];
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            const int r = r_base + 4 * j;
            // exp of a non-positive difference (entries above the diagonal are discarded)
            const float gam = expf(fminf(Gs[r * E + e] - gs, 0.f));
            const float ks2 = (r >= s_own) ? ks * gam : 0.f;
            Rv[j] = fmaf(k2s[r * E + e], ks2, Rv[j]);
            Rq[j] = fmaf(q2s[r * E + e], ks2, Rq[j]);
        }
    }
    __syncthreads();
    if (p.use_delta) {
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            const int r = r_base + 4 * j, s = s_own;
            B1[r * MP + s] = dT[j] * bs[s];              // dN
            B2[r * MP + s] = dT[j] * B0[r * MP + s];     // column terms of dbeta
        }
        __syncthreads();
        if (tid < 64) {
            float acc = 0.f;
            for (int r = 0; r < 64; ++r) acc += B2[r * MP + tid];
            dba[tid] += acc;
        }
        {                                               // F = dN N^T (16 independent sums)
            float acc[16];
#pragma unroll
            for (int j = 0; j < 16; ++j) acc[j] = 0.f;
#pragma unroll 4
            for (int x = 0; x < 64; ++x) {
                const float nsx = B0[s_own * MP + x];
#pragma unroll
                for (int j = 0; j < 16; ++j) acc[j] = fmaf(B1[(r_base + 4 * j) * MP + x], nsx, acc[j]);
            }
#pragma unroll
            for (int j = 0; j < 16; ++j) B3[(r_base + 4 * j) * MP + s_own] = acc[j];
        }
        __syncthreads();
        float dL[16];
        {                                               // dM = -N^T F, strictly lower part
#pragma unroll
            for (int j = 0; j < 16; ++j) dL[j] = 0.f;
#pragma unroll 4
            for (int x = 0; x < 64; ++x) {
                const float fxs = B3[x * MP + s_own];
#pragma unroll
                for (int j = 0; j < 16; ++j) dL[j] = fmaf(B0[x * MP + r_base + 4 * j], fxs, dL[j]);
            }
#pragma unroll
            for (int j = 0; j < 16; ++j) dL[j] = (r_base + 4 * j > s_own) ? -dL[j] : 0.f;
        }
        __syncthreads();
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            const int r = r_base + 4 * j, s = s_own;
            B1[r * MP + s] = dL[j] * bs[r] * KK[j];    // dR
            B4[r * MP + s] = dL[j] * bs[r] * Rv[j];    // dKK
            B5[r * MP + s] = dL[j] * KK[j] * Rv[j];    // row terms of dbeta
        }
    } else {
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            const int r = r_base + 4 * j, s = s_own;
            B1[r * MP + s] = 0.f;
            B4[r * MP + s] = 0.f;
            B5[r * MP + s] = (r == s) ? dT[j] : 0.f;   // T = diag(beta)
        }
    }
#pragma unroll
    for (int j = 0; j < 16; ++j) {
        const int r = r_base + 4 * j, s = s_own;
        const bool low = r >= s;
        B2[r * MP + s] = low ? dA[j] * QK[j] : 0.f;    // dR'
        B3[r * MP + s] = low ? dA[j] * Rq[j] : 0.f;    // P = dA (.) R'
    }
    __syncthreads();
    if (tid < 64) {
        float acc = 0.f;
        for (int s = 0; s < 64; ++s) acc += B5[tid * MP + s];
        dba[tid] += acc;
    }
    for (int i = tid; i < 64 * E; i += kThreads) {      // through R (dR in B1) and R' (dR' in B2)
        const int x = i / E, e = i - (i / E) * E;
        const float gx = Gs[x * E + e], kx = k2s[x * E + e], qx = q2s[x * E + e];
        float dk2v = 0.f, dq2v = 0.f, dGv = 0.f;
        for (int s = 0; s <= x; ++s) {
            const float gam = expf(gx - Gs[s * E + e]);
            const float ks = k2s[s * E + e];
            const float dR = B1[x * MP + s], dRq = B2[x * MP + s];
            dk2v = fmaf(dR * ks, gam, dk2v);
            dq2v = fmaf(dRq * ks, gam, dq2v);
            dGv = fmaf((dR * kx + dRq * qx) * ks, gam, dGv);
        }
        for (int r = x; r < 64; ++r) {
            const float gam = expf(Gs[r * E + e] - gx);
            const float dR = B1[r * MP + x], dRq = B2[r * MP + x];
            const float t = (dR * k2s[r * E + e] + dRq * q2s[r * E + e]) * gam;
            dk2v += t;
            dGv = fmaf(-t, kx, dGv);
        }
        dk2a[i] = dk2v;
        dq2a[i] = dq2v;
        dGa[i] = dGv;
    }
    __syncthreads();
    // A3 = [[P, 0], [dKK + dKK^T, P^T]] (128 x 128) as bf16 hi/lo into sX (P in B3, dKK in B4)
    {
        const int i = tid >> 1, jh = tid & 1;
        for (int j0 = jh * 64; j0 < jh * 64 + 64; j0 += 8) {
            float v[8];
            for (int u = 0; u < 8; ++u) {
                const int j = j0 + u;
                float x;
                if (i < 64) x = (j < 64) ? B3[i * MP + j] : 0.f;
                else {
                    const int r = i - 64;
                    x = (j < 64) ? B4[r * MP + j] + B4[j * MP + r] : B3[(j - 64) * MP + r];
                }
                v[u] = x;
            }
            st8_split(sX, sX + 32768, sw128_offset(i, j0, 128), v);
        }
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (tid == 0) {
        const uint32_t id = idesc_bf16_f32(128, kDk, 0, 1);
        for (int ks = 0; ks < 8; ++ks) {
            const uint32_t o = (ks >> 2) * 16384 + (ks & 3) * 32;
            const uint64_t bq = smem_desc(smem_u32(sKQ) + ks * 2048, 2 * kBoxBytes, 1024);
            umma_bf16(tACC, smem_desc(smem_u32(sX) + o, 16, 1024), bq, id, ks > 0 ? 1u : 0u);
            umma_bf16(tACC, smem_desc(smem_u32(sX + 32768) + o, 16, 1024), bq, id, 1u);
        }
        umma_commit(&bar_mma);
    }
    ok = mma_wait();
    if (__syncthreads_or(!ok)) {
        if (tid == 0) record_device_error(p.err, TLA_ERR_TIMEOUT);
        __syncthreads();
        if (warp == 0) tmem_dealloc(tmem, 512);
        return;
    }
    tc_fence_after();

    // ---- phase 2: per slice.  The checkpoint tiles (bf16 hi/lo, operand layout) arrive by
    // bulk copy: S_e into sX, then dS'_e into sY once the first products have consumed A1.
    const size_t sbase = ((size_t(b) * H + h) * NT + c) * E;
    const uint32_t slab_bytes = uint32_t(kDk) * dv * 4;   // hi tile + lo tile
    const uint32_t LO = uint32_t(kDk) * dv * 2;           // lo tile offset of a checkpoint slab
    const int wq = warp & 3, L = wq * 32 + lane, half = warp >> 2;
    const int cpr = dv / 8;   // 8-column chunks per row
    uint32_t sph = 0, dph = 0;
    if (tid == 0) {
        mbar_arrive_expect_tx(&bar_s, slab_bytes);
        bulk_load(sX, reinterpret_cast<const uint8_t*>(p.Sck) + sbase * kDk * dv * 4, slab_bytes, &bar_s);
    }
    bool failed = false;
    for (int e = 0; e < E && !failed; ++e) {
        // A1_e = [b_e dO ; -a_e dRes] -> sY
        for (int ci = tid; ci < 128 * cpr; ci += kThreads) {
            const int i = ci / cpr, cc = (ci % cpr) * 8;
            float v[8];
            if (i < 64) {
                const float bq = q2s[i * E + e] * expf(Gs[i * E + e]);
                load_bf16x8(sDO + sw128_offset(i, cc, 64), v);
                for (int u = 0; u < 8; ++u) v[u] *= bq;
            } else {
                const int r = i - 64;
                if (p.use_delta && r < n) {
                    const float a = -k2s[r * E + e] * expf(Gs[r * E + e]);
                    load_row8(p.dRbuf + tok_idx(b, t0 + r, h, cc, T, H, dv), v);
                    for (int u = 0; u < 8; ++u) v[u] *= a;
                } else {
                    for (int u = 0; u < 8; ++u) v[u] = 0.f;
                }
            }
            st8_split(sY, sY + 32768, sw128_offset(i, cc, 128), v);
        }
        bool ok = mbar_wait(&bar_s, sph);
        sph ^= 1;
        fence_proxy_async_smem();
        tc_fence_before();
        if (__syncthreads_or(!ok)) { failed = true; break; }
        tc_fence_after();
        if (tid == 0) {
            const uint32_t idA = idesc_bf16_f32(128, kDk, 0, 0);
            for (int ks = 0; ks < dv / 16; ++ks) {
                const uint32_t o = (ks >> 2) * 16384 + (ks & 3) * 32;
                const uint64_t ah = smem_desc(smem_u32(sY) + o, 16, 1024);
                const uint64_t al = smem_desc(smem_u32(sY + 32768) + o, 16, 1024);
                const uint64_t bh = smem_desc(smem_u32(sX) + o, 16, 1024);
                const uint64_t bl = smem_desc(smem_u32(sX + LO) + o, 16, 1024);
                umma_bf16(tACC, ah, bh, idA, 1u);
                umma_bf16(tACC, ah, bl, idA, 1u);
                umma_bf16(tACC, al, bh, idA, 1u);
            }
            const uint32_t idP = idesc_bf16_f32(128, dv, 0, 1);
            for (int ks = 0; ks < kDk / 16; ++ks) {
                const uint64_t a = smem_desc(smem_u32(sKQ) + (ks >> 2) * 2 * kBoxBytes + (ks & 3) * 32, 16, 1024);
                umma_bf16(tP, a, smem_desc(smem_u32(sX) + ks * 2048, 16384, 1024), idP, ks > 0 ? 1u : 0u);
                umma_bf16(tP, a, smem_desc(smem_u32(sX + LO) + ks * 2048, 16384, 1024), idP, 1u);
            }
            umma_commit(&bar_mma);
        }
        ok = mma_wait();
        if (__syncthreads_or(!ok)) { failed = true; break; }
        tc_fence_after();
        if (tid == 0) {   // A1 consumed: dS'_e into sY
            mbar_arrive_expect_tx(&bar_d, slab_bytes);
            bulk_load(sY, reinterpret_cast<const uint8_t*>(p.dSck) + (sbase + e) * kDk * dv * 4,
                      slab_bytes, &bar_d);
        }
        // row dots of P_e = [K;Q] S_e while dS'_e is in flight
        {
            float acc = 0.f;
            const int cw = dv / 2;
            for (int j = half * cw; j < half * cw + cw; j += 16) {
                float pv[16];
                tmem_ld16(tmem_lane_addr(tP, warp, j), pv);
                tmem_wait_ld();
                float x[16];
                if (L < 64) {
                    if (L < n && p.use_delta) {
                        load_row8(p.dRbuf + tok_idx(b, t0 + L, h, j, T, H, dv), x);
                        load_row8(p.dRbuf + tok_idx(b, t0 + L, h, j + 8, T, H, dv), x + 8);
                    } else {
                        for (int u = 0; u < 16; ++u) x[u] = 0.f;
                    }
                } else {
                    load_bf16x8(sDO + sw128_offset(L - 64, j, 64), x);
                    load_bf16x8(sDO + sw128_offset(L - 64, j + 8, 64), x + 8);
                }
                for (int u = 0; u < 16; ++u) acc = fmaf(x[u], pv[u], acc);
            }
            red[half * 128 + L] = acc;
        }
        ok = mbar_wait(&bar_d, dph);
        dph ^= 1;
        // <dS'_e, S_e> from the hi/lo tiles (hi + lo reproduces each value to ~2^-16)
        {
            float fro = 0.f;
            for (int ci = tid; ci < 128 * cpr; ci += kThreads) {
                const uint32_t o = sw128_offset(ci / cpr, (ci % cpr) * 8, 128);
                float sh[8], sl[8], dh[8], dl[8];
                load_bf16x8(sX + o, sh);
                load_bf16x8(sX + LO + o, sl);
                load_bf16x8(sY + o, dh);
                load_bf16x8(sY + LO + o, dl);
                for (int u = 0; u < 8; ++u) fro = fmaf(dh[u] + dl[u], sh[u] + sl[u], fro);
            }
            red2[tid] = fro;
        }
        if (__syncthreads_or(!ok)) { failed = true; break; }
        if (tid < 128) {
            const float v = red[tid] + red[128 + tid];
            if (tid < 64) dak[tid * E + e] = -v;
            else dbq[(tid - 64) * E + e] = v;
        }
        if (tid == 0) {
            float f = 0.f;
            for (int i = 0; i < kThreads; ++i) f += red2[i];
            dgc[e] = f;
        }
        // A2_e = [0 ; w_e U] -> sX (S_e consumed)
        for (int ci = tid; ci < 128 * cpr; ci += kThreads) {
            const int i = ci / cpr, cc = (ci % cpr) * 8;
            float v[8];
            const int r = i - 64;
            if (i >= 64 && r < n) {
                const float w = k2s[r * E + e] * expf(Gs[(n - 1) * E + e] - Gs[r * E + e]);
                load_row8(p.Ubuf + tok_idx(b, t0 + r, h, cc, T, H, dv), v);
                for (int u = 0; u < 8; ++u) v[u] *= w;
            } else {
                for (int u = 0; u < 8; ++u) v[u] = 0.f;
            }
            st8_split(sX, sX + 32768, sw128_offset(i, cc, 128), v);
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        tc_fence_after();
        if (tid == 0) {
            const uint32_t idA = idesc_bf16_f32(128, kDk, 0, 0);
            for (int ks = 0; ks < dv / 16; ++ks) {
                const uint32_t o = (ks >> 2) * 16384 + (ks & 3) * 32;
                const uint64_t ah = smem_desc(smem_u32(sX) + o, 16, 1024);
                const uint64_t al = smem_desc(smem_u32(sX + 32768) + o, 16, 1024);
                const uint64_t bh = smem_desc(smem_u32(sY) + o, 16, 1024);
                const uint64_t bl = smem_desc(smem_u32(sY + LO) + o, 16, 1024);
                umma_bf16(tACC, ah, bh, idA, 1u);
                umma_bf16(tACC, ah, bl, idA, 1u);
                umma_bf16(tACC, al, bh, idA, 1u);
            }
            const uint32_t idP = idesc_bf16_f32(128, dv, 0, 1);
            for (int ks = 0; ks < kDk / 16; ++ks) {
                const uint64_t a = smem_desc(smem_u32(sKQ) + (ks >> 2) * 2 * kBoxBytes + (ks & 3) * 32, 16, 1024);
                umma_bf16(tP2, a, smem_desc(smem_u32(sY) + ks * 2048, 16384, 1024), idP, ks > 0 ? 1u : 0u);
                umma_bf16(tP2, a, smem_desc(smem_u32(sY + LO) + ks * 2048, 16384, 1024), idP, 1u);
            }
            umma_commit(&bar_mma);
        }
        ok = mma_wait();
        if (__syncthreads_or(!ok)) { failed = true; break; }
        tc_fence_after();
        if (tid == 0 && e + 1 < E) {   // A2 consumed: S_{e+1} into sX
            mbar_arrive_expect_tx(&bar_s, slab_bytes);
            bulk_load(sX, reinterpret_cast<const uint8_t*>(p.Sck) + (sbase + e + 1) * kDk * dv * 4,
                      slab_bytes, &bar_s);
        }
        // row dots of P'_e = [K;Q] dS'_e (key rows)
        {
            float acc = 0.f;
            const int cw = dv / 2;
            for (int j = half * cw; j < half * cw + cw; j += 16) {
                float pv[16];
                tmem_ld16(tmem_lane_addr(tP2, warp, j), pv);
                tmem_wait_ld();
                if (L < n) {
                    float x[16];
                    load_row8(p.Ubuf + tok_idx(b, t0 + L, h, j, T, H, dv), x);
                    load_row8(p.Ubuf + tok_idx(b, t0 + L, h, j + 8, T, H, dv), x + 8);
                    for (int u = 0; u < 16; ++u) acc = fmaf(x[u], pv[u], acc);
                }
            }
            red[half * 128 + L] = acc;
        }
        __syncthreads();
        if (tid < 64) dwk[tid * E + e] = red[tid] + red[128 + tid];
        tc_fence_before();
        __syncthreads();
        tc_fence_after();
    }
    if (failed) {
        if (tid == 0) record_device_error(p.err, TLA_ERR_TIMEOUT);
        tc_fence_before();
        __syncthreads();
        if (warp == 0) tmem_dealloc(tmem, 512);
        return;
    }

    // ---- phase 3: dq (ACC rows 0-63), dk (rows 64-127)
    {
        const int row = L < 64 ? L : L - 64;
        void* dst = L < 64 ? p.dq : p.dk;
        for (int j = half * 64; j < half * 64 + 64; j += 16) {
            float v[16];
            tmem_ld16(tmem_lane_addr(tACC, warp, j), v);
            tmem_wait_ld();
            if (row < n) store_row(dst, tok_idx(b, t0 + row, h, j, T, H, kDk), v, 16, p.out_f32);
        }
    }
    for (int i = tid; i < 64 * E; i += kThreads) {
        const int e = i - (i / E) * E;
        const float gam = expf(Gs[i]);
        const float wdec = expf(Gs[(n - 1) * E + e] - Gs[i]);
        const float a = k2s[i] * gam, bq = q2s[i] * gam, w = k2s[i] * wdec;
        dk2a[i] += dak[i] * gam + dwk[i] * wdec;
        dq2a[i] += dbq[i] * gam;
        dGa[i] += dak[i] * a + dbq[i] * bq - dwk[i] * w;
    }
    __syncthreads();
    if (tid < E) {
        const int e = tid;
        float dGC = 0.f;
        for (int r = 0; r < n; ++r) {
            const float w = k2s[r * E + e] * expf(Gs[(n - 1) * E + e] - Gs[r * E + e]);
            dGC = fmaf(dwk[r * E + e], w, dGC);
        }
        dGC = fmaf(dgc[e], expf(Gs[(n - 1) * E + e]), dGC);
        dGa[(n - 1) * E + e] += dGC;
        float acc = 0.f;
        for (int r = n - 1; r >= 0; --r) {
            acc += dGa[r * E + e];
            p.dg[tok_idx(b, t0 + r, h, e, T, H, E)] = acc;
        }
    }
    for (int i = tid; i < n * E; i += kThreads) {
        const int r = i / E, e = i - (i / E) * E;
        const size_t off = tok_idx(b, t0 + r, h, e, T, H, E);
        store_out(p.dq2, off, dq2a[i], p.out_f32);
        store_out(p.dk2, off, dk2a[i], p.out_f32);
    }
    if (p.dbeta && tid < n) p.dbeta[(size_t(b) * T + t0 + tid) * H + h] = dba[tid];
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tmem_dealloc(tmem, 512);
}

size_t grads_tc_smem(int E) {
    return 1024 + 6 * kBoxBytes + 2 * 65536 + (9 * 64 * E + 64 + 64 + 16 + 256 + 256) * 4;
}

}  // namespace

int tc_grads_shape_ok(const tla_problem& p) {
    return p.dk == kDk && p.dv % 64 == 0 && p.dv <= 128 && p.E <= 8 &&
           grads_tc_smem(p.E) <= 227 * 1024;
}

int tc_grads_ok(const tla_problem& p, const FwdPlan& fp) { return fp.ck_tiles && tc_grads_shape_ok(p); }

cudaError_t launch_bwd_chunk_grads_tc(const tla_problem& p, const FwdPlan& fp, const char* fws,
                                      const BwdPlan& bp, const char* bws, const void* dO,
                                      void* dq, void* dk, void* dq2, void* dk2, float* dbeta,
                                      float* dg, int* err, cudaStream_t s) {
    CUtensorMap mk, mq, mo;
    if (!make_token_map(&mk, p.k, p.B, p.T, p.H, kDk, 64, 64, true) ||
        !make_token_map(&mq, p.q, p.B, p.T, p.H, kDk, 64, 64, true) ||
        !make_token_map(&mo, dO, p.B, p.T, p.H, p.dv, 64, 64, true))
        return cudaErrorInvalidValue;
    TcGradArgs a;
    a.q2 = (const __nv_bfloat16*)p.q2;
    a.k2 = (const __nv_bfloat16*)p.k2;
    a.v = (const __nv_bfloat16*)p.v;
    a.G = (const float*)(fws + fp.G);
    a.beta = p.beta;
    a.Nmat = p.use_delta ? (const float*)(fws + fp.N) : nullptr;
    a.Sck = (const float*)(fws + fp.S);
    a.Ubuf = (const float*)(fws + fp.U);
    a.Rbuf = p.use_delta ? (const float*)(fws + fp.Res) : nullptr;
    a.dUbuf = (const float*)(bws + bp.dU);
    a.dRbuf = (const float*)(bws + bp.dRes);
    a.dSck = (const float*)(bws + bp.dS);
    a.dq = dq; a.dk = dk; a.dq2 = dq2; a.dk2 = dk2; a.dbeta = dbeta; a.dg = dg;
    a.err = err;
    a.T = p.T; a.H = p.H; a.dv = p.dv; a.E = p.E; a.NT = fp.NT;
    a.use_delta = p.use_delta; a.out_f32 = p.out_dtype == TLA_FP32;
    const size_t smem = grads_tc_smem(p.E);
    cudaFuncSetAttribute(bwd_chunk_grads_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         (int)smem);
    dim3 grid(fp.NT, p.H, p.B);
    prof_before("bwd_chunk_grads_tc", s);
    bwd_chunk_grads_tc_kernel<<<grid, kThreads, smem, s>>>(mk, mq, mo, a);
    prof_after(s);
    return cudaGetLastError();
}

}  // namespace tla
