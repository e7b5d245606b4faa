// Per-chunk preparation for the tensor-core path (bf16 inputs, d_k = 128, or 64 with the
// key/query boxes zero-filled past it).
// One CTA of 8 warps per (b, h, chunk) computes, Appendix A:
//   K K^T and Q K^T                  one UMMA [K; Q] K^T on the TMA key/query tile
//   R, R' element by element         exp of non-positive log-decay differences (Eq. joint-gram)
//   A = Q K^T (.) R' (lower incl. diagonal), L = tril(diag(beta)(K K^T (.) R), -1)
//   N = (I + L)^{-1}                 blocked: the four 16 x 16 diagonal blocks by forward
//                                    substitution (one warp each, registers only), then the
//                                    off-diagonal blocks in two levels (Eq. joint-solve):
//                                    blocks (1,0) and (3,2), then the lower-left 32 x 32
//                                    block from the two 32 x 32 diagonal blocks
//   T = N diag(beta) (sGLA: diag(beta)), A T
// and writes A and N (fp32), the bf16 hi/lo tiles [T; A T] (forward recurrence) and
// [A; T] (backward recurrence, which reads them as the MN-major operands A^T and T^T), and
// the per-row coefficient block
// [k'_e gamma_e | q'_e gamma_e | k'_e gamma^C_e / gamma_e | gamma^C_e] (slice-major).
#include "common.cuh"
#include "internal.h"
#include "sm100.cuh"
#include "tma_host.h"

namespace tla {
using namespace sm100;

namespace {

constexpr int kThreads = 256;
constexpr int kDk = 128;
constexpr int kBoxBytes = 64 * 64 * 2;
constexpr int MP = 68;                        // row stride (floats) of the C x C matrices
constexpr int kSlot = 64 * MP;                // floats per matrix slot (17408 bytes)
constexpr int XS = 20;                        // row stride of the transposed 16 x 16 diagonal blocks

struct TcPrepArgs {
    const __nv_bfloat16* q2;
    const __nv_bfloat16* k2;
    const float* G;
    const float* beta;
    float* Aout;
    float* Nout;
    __nv_bfloat16* A2out;
    __nv_bfloat16* BTout;
    float* coef;
    int* err;
    const int2* ctab;    // packed documents: (first token, rows) of each chunk; else NULL
    int T, H, E, NT, use_delta;
    int dk;              // key dimension: 128, or 64 (the key/query boxes past it are zero)
};

__device__ __forceinline__ void ld4(const float* src, float* v) {
    const float4 x = *reinterpret_cast<const float4*>(src);
    v[0] = x.x; v[1] = x.y; v[2] = x.z; v[3] = x.w;
}
__device__ __forceinline__ void st4(float* dst, float v0, float v1, float v2, float v3) {
    *reinterpret_cast<float4*>(dst) = make_float4(v0, v1, v2, v3);
}
// Four consecutive values as bf16 hi/lo pairs (8 bytes into each of two global arrays).
__device__ __forceinline__ void put4(__nv_bfloat16* hi, __nv_bfloat16* lo, float v0, float v1,
                                     float v2, float v3) {
    const __nv_bfloat162 h0 = __floats2bfloat162_rn(v0, v1), h1 = __floats2bfloat162_rn(v2, v3);
    const float2 f0 = __bfloat1622float2(h0), f1 = __bfloat1622float2(h1);
    const __nv_bfloat162 l0 = __floats2bfloat162_rn(v0 - f0.x, v1 - f0.y);
    const __nv_bfloat162 l1 = __floats2bfloat162_rn(v2 - f1.x, v3 - f1.y);
    *reinterpret_cast<uint2*>(hi) =
        make_uint2(*reinterpret_cast<const uint32_t*>(&h0), *reinterpret_cast<const uint32_t*>(&h1));
    *reinterpret_cast<uint2*>(lo) =
        make_uint2(*reinterpret_cast<const uint32_t*>(&l0), *reinterpret_cast<const uint32_t*>(&l1));
}

__global__ void __launch_bounds__(kThreads, 2)
chunk_prep_tc_kernel(const __grid_constant__ CUtensorMap map_k,
                     const __grid_constant__ CUtensorMap map_q, const TcPrepArgs p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
    const int E = p.E, T = p.T, H = p.H, NT = p.NT;
    const int c = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
    int t0 = c * 64, n = min(64, T - t0);
    if (p.ctab) {
        const int2 cr = p.ctab[c];
        t0 = cr.x;
        n = cr.y;
    }
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    // five matrix slots; the TMA key/query tile overlays slots 3-4 until the products are read
    float* slot = reinterpret_cast<float*>(sm);
    float* LT = slot;                 // L^T (K K^T first)
    float* MX = slot + kSlot;         // N = (I + L)^{-1} (Q K^T first)
    float* MAT = slot + 2 * kSlot;    // A^T
    float* MW = slot + 3 * kSlot;     // off-diagonal block products, then T
    float* XT = slot + 4 * kSlot;     // transposed 16 x 16 diagonal blocks of N, 4 x [16][XS]
    uint8_t* sKQ = sm + 3 * kSlot * 4;   // 1024-aligned (3 x 17408 = 51 x 1024)
    float* Gs = slot + 5 * kSlot;
    float* k2s = Gs + 64 * E;
    float* q2s = k2s + 64 * E;
    float* bs = q2s + 64 * E;

    __shared__ __align__(8) uint64_t bar_ld, bar_mma;
    __shared__ uint32_t tmem_slot;
    if (warp == 0) {
        tmem_alloc(&tmem_slot, 64);
        tmem_relinquish();
    }
    if (tid == 0) {
        mbar_init(&bar_ld, 1);
        mbar_init(&bar_mma, 1);
        fence_barrier_init();
        mbar_arrive_expect_tx(&bar_ld, 4 * kBoxBytes);
        for (int j = 0; j < 2; ++j) {
            tma_load_4d(sKQ + j * 2 * kBoxBytes, &map_k, &bar_ld, 64 * j, h, t0, b);
            tma_load_4d(sKQ + j * 2 * kBoxBytes + kBoxBytes, &map_q, &bar_ld, 64 * j, h, t0, b);
        }
    }
    // the chunk's log decays, second keys and queries and beta: loaded into registers now
    // (token-major, E values of a token side by side), so that their latency overlaps the
    // key/query copies and the Gram product; stored slice-major ([E][64]) after it
    // (raw register copies, nothing computed from them until the product has been issued, so
    // no instruction waits for the loads here)
    float gv[4], bv = 1.f;
    unsigned short kv[4], qv[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {   // 64 E <= 1024 values: at most four per thread
        const int i = tid + u * kThreads;
        gv[u] = 0.f;
        kv[u] = qv[u] = 0;   // bf16 zero
        if (i < 64 * E) {
            const int r = i / E, e = i - (i / E) * E;
            const int rr = r < n ? r : n - 1;
            gv[u] = p.G[tok_idx(b, t0 + rr, h, e, T, H, E)];
            if (r < n) {
                kv[u] = __bfloat16_as_ushort(p.k2[tok_idx(b, t0 + r, h, e, T, H, E)]);
                qv[u] = __bfloat16_as_ushort(p.q2[tok_idx(b, t0 + r, h, e, T, H, E)]);
            }
        }
    }
    if (tid < n && p.beta) bv = p.beta[(size_t(b) * T + t0 + tid) * H + h];
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;
    bool ok = mbar_wait(&bar_ld, 0);
    if (__syncthreads_or(!ok)) {
        if (tid == 0) {
            record_device_error(p.err, TLA_ERR_TIMEOUT);
            mbar_wait(&bar_ld, 0);   // bounded: the copies still in flight
        }
        __syncthreads();
        if (warp == 0) tmem_dealloc(tmem, 64);
        return;
    }
    if (tid == 0) {
        const uint32_t id = idesc_bf16_f32(128, 64, 0, 0);
        for (int ks = 0; ks < kDk / 16; ++ks) {
            if (ks * 16 >= p.dk) break;   // zero key columns past d_k
            const uint64_t a = smem_desc(smem_u32(sKQ) + (ks >> 2) * 2 * kBoxBytes + (ks & 3) * 32, 16, 1024);
            umma_bf16(tmem, a, a, id, ks > 0 ? 1u : 0u);
        }
        umma_commit(&bar_mma);
    }
    ok = mbar_wait(&bar_mma, 0);
    if (__syncthreads_or(!ok)) {
        if (tid == 0) {
            record_device_error(p.err, TLA_ERR_TIMEOUT);
            mbar_wait(&bar_mma, 0);
        }
        __syncthreads();
        if (warp == 0) tmem_dealloc(tmem, 64);
        return;
    }
    tc_fence_after();
    if (warp < 4) {   // rows 0-63: K K^T -> slot 0, rows 64-127: Q K^T -> slot 1
        const int L = warp * 32 + lane;
        float* dst = (L < 64 ? LT : MX) + (L & 63) * MP;
        for (int j = 0; j < 64; j += 16) {
            float v[16];
            tmem_ld16(tmem_lane_addr(tmem, warp, j), v);
            tmem_wait_ld();
#pragma unroll
            for (int q = 0; q < 4; ++q) st4(dst + j + 4 * q, v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
        }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        const int i = tid + u * kThreads;
        if (i < 64 * E) {
            const int r = i / E, e = i - (i / E) * E;
            Gs[e * 64 + r] = gv[u];
            k2s[e * 64 + r] = __bfloat162float(__ushort_as_bfloat16(kv[u]));
            q2s[e * 64 + r] = __bfloat162float(__ushort_as_bfloat16(qv[u]));
        }
    }
    if (tid < 64) bs[tid] = tid < n ? bv : 0.f;   // beta, 1 without one, 0 past the chunk's rows
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tmem_dealloc(tmem, 64);

    // ---- A and L on 4 x 4 blocks: thread owns rows R0..R0+3, columns S0..S0+3
    const int R0 = 4 * (tid >> 4), S0 = 4 * (tid & 15);
    const bool live = R0 + 3 >= S0;   // blocks entirely above the diagonal are zero
    float KK[4][4], Av[4][4], Lv[4][4];
#pragma unroll
    for (int a = 0; a < 4; ++a) {
        ld4(LT + (R0 + a) * MP + S0, KK[a]);
        ld4(MX + (R0 + a) * MP + S0, Av[a]);   // Q K^T for now
    }
    __syncthreads();
    if (live) {
        float R[4][4], Rq[4][4];
#pragma unroll
        for (int a = 0; a < 4; ++a)
#pragma unroll
            for (int c2 = 0; c2 < 4; ++c2) R[a][c2] = Rq[a][c2] = 0.f;
        for (int e = 0; e < E; ++e) {
            float gs[4], ks[4], grv[4], krv[4], qrv[4];
            ld4(Gs + e * 64 + S0, gs);
            ld4(k2s + e * 64 + S0, ks);
            ld4(Gs + e * 64 + R0, grv);
            ld4(k2s + e * 64 + R0, krv);
            ld4(q2s + e * 64 + R0, qrv);
#pragma unroll
            for (int a = 0; a < 4; ++a) {
                const float gr = grv[a], kr = krv[a], qr = qrv[a];
#pragma unroll
                for (int c2 = 0; c2 < 4; ++c2) {
                    // exp of a non-positive log-decay difference (Eq. joint-gram); the
                    // clamp only matters above the diagonal, where the entry is discarded
                    const float ks2 = ks[c2] * __expf(fminf(gr - gs[c2], 0.f));
                    R[a][c2] = fmaf(kr, ks2, R[a][c2]);
                    Rq[a][c2] = fmaf(qr, ks2, Rq[a][c2]);
                }
            }
        }
#pragma unroll
        for (int a = 0; a < 4; ++a)
#pragma unroll
            for (int c2 = 0; c2 < 4; ++c2) {
                const int r = R0 + a, s2 = S0 + c2;
                Av[a][c2] = (r >= s2) ? Av[a][c2] * Rq[a][c2] : 0.f;
                Lv[a][c2] = (r > s2) ? bs[r] * KK[a][c2] * R[a][c2] : 0.f;
            }
    } else {
#pragma unroll
        for (int a = 0; a < 4; ++a)
#pragma unroll
            for (int c2 = 0; c2 < 4; ++c2) Av[a][c2] = Lv[a][c2] = 0.f;
    }
    const size_t mat = ((size_t(b) * H + h) * NT + c) * (64 * 64);
#pragma unroll
    for (int a = 0; a < 4; ++a) {
        if (p.Aout)
            *reinterpret_cast<float4*>(p.Aout + mat + (R0 + a) * 64 + S0) = make_float4(Av[a][0], Av[a][1], Av[a][2], Av[a][3]);
    }
#pragma unroll
    for (int c2 = 0; c2 < 4; ++c2) {
        st4(MAT + (S0 + c2) * MP + R0, Av[0][c2], Av[1][c2], Av[2][c2], Av[3][c2]);
        st4(LT + (S0 + c2) * MP + R0, Lv[0][c2], Lv[1][c2], Lv[2][c2], Lv[3][c2]);
    }
    __syncthreads();

    // ---- N = (I + L)^{-1} (Eq. joint-solve): the four 16 x 16 diagonal blocks by forward
    // substitution (warps 0-3, lane = column), then the off-diagonal blocks in two levels
    if (p.use_delta) {
        if (warp < 4 && lane < 16) {
            // column s2 of the block's inverse: x_r = delta_{r,s2} - sum_{j<r} L_rj x_j, each
            // x_r applied to the later rows as soon as it is final (the same terms in the same
            // order as row-by-row substitution, but a dependent chain of 16 steps, not 120)
            const int o = 16 * warp, s2 = lane;
            float x[16], acc[16];
#pragma unroll
            for (int k = 0; k < 16; ++k) acc[k] = (k == s2) ? 1.f : 0.f;
#pragma unroll
            for (int r = 0; r < 16; ++r) {
                x[r] = acc[r];
#pragma unroll
                for (int k = r + 1; k < 16; ++k) acc[k] = fmaf(-LT[(o + r) * MP + o + k], x[r], acc[k]);
            }
#pragma unroll
            for (int r = 0; r < 16; ++r) {
                MX[(o + r) * MP + o + s2] = x[r];
                XT[warp * 16 * XS + s2 * XS + r] = x[r];
            }
        }
        for (int i = tid; i < 64 * 64; i += kThreads) {   // zero the strictly upper blocks
            const int r = i >> 6, s2 = i & 63;
            if ((s2 >> 4) > (r >> 4)) MX[r * MP + s2] = 0.f;
        }
        __syncthreads();
        // Off-diagonal blocks in two levels (2 x 2 register blocks, each entry's sum in order):
        // level 1 the 16 x 16 blocks (1,0) and (3,2), X_ij = -X_ii (L_ij X_jj) (128 threads);
        // level 2 the lower-left 32 x 32 block, N21 = -N22 (L21 N11), N11 and N22 the 32 x 32
        // diagonal blocks, complete after level 1 (256 threads) -- a dependent depth of 96
        // multiply-adds instead of 144 by distance.
        {
            const int bi = 1 + 2 * (tid >> 6), bj = bi - 1;
            const int r0 = 16 * bi + 2 * ((tid >> 3) & 7), s0 = 16 * bj + 2 * (tid & 7);
            if (tid < 128) {   // W = L_ij X_jj
                float w[2][2] = {{0.f, 0.f}, {0.f, 0.f}};
#pragma unroll 4
                for (int x = 16 * bj; x < 16 * bi; ++x) {
                    const float2 l = *reinterpret_cast<const float2*>(LT + x * MP + r0);
                    const float2 xv = *reinterpret_cast<const float2*>(MX + x * MP + s0);
                    w[0][0] = fmaf(l.x, xv.x, w[0][0]);
                    w[0][1] = fmaf(l.x, xv.y, w[0][1]);
                    w[1][0] = fmaf(l.y, xv.x, w[1][0]);
                    w[1][1] = fmaf(l.y, xv.y, w[1][1]);
                }
#pragma unroll
                for (int a = 0; a < 2; ++a)
                    *reinterpret_cast<float2*>(MW + (r0 + a) * MP + s0) = make_float2(w[a][0], w[a][1]);
            }
            __syncthreads();
            if (tid < 128) {   // X_ij = -X_ii W
                float xo[2][2] = {{0.f, 0.f}, {0.f, 0.f}};
                const float* xt = XT + bi * 16 * XS;
#pragma unroll 4
                for (int x = 0; x < 16; ++x) {
                    const float2 xi = *reinterpret_cast<const float2*>(xt + x * XS + (r0 - 16 * bi));
                    const float2 wv = *reinterpret_cast<const float2*>(MW + (16 * bi + x) * MP + s0);
                    xo[0][0] = fmaf(xi.x, wv.x, xo[0][0]);
                    xo[0][1] = fmaf(xi.x, wv.y, xo[0][1]);
                    xo[1][0] = fmaf(xi.y, wv.x, xo[1][0]);
                    xo[1][1] = fmaf(xi.y, wv.y, xo[1][1]);
                }
#pragma unroll
                for (int a = 0; a < 2; ++a)
                    *reinterpret_cast<float2*>(MX + (r0 + a) * MP + s0) = make_float2(-xo[a][0], -xo[a][1]);
            }
            __syncthreads();
        }
        {
            const int i0 = 2 * (tid >> 4), j0 = 2 * (tid & 15);   // rows 32 + i0.., columns j0..
            float w[2][2] = {{0.f, 0.f}, {0.f, 0.f}};
#pragma unroll 4
            for (int k = j0; k < 32; ++k) {   // W = L21 N11 (N11 lower triangular)
                const float2 l = *reinterpret_cast<const float2*>(LT + k * MP + 32 + i0);
                const float2 nv = *reinterpret_cast<const float2*>(MX + k * MP + j0);
                w[0][0] = fmaf(l.x, nv.x, w[0][0]);
                w[0][1] = fmaf(l.x, nv.y, w[0][1]);
                w[1][0] = fmaf(l.y, nv.x, w[1][0]);
                w[1][1] = fmaf(l.y, nv.y, w[1][1]);
            }
#pragma unroll
            for (int a = 0; a < 2; ++a)
                *reinterpret_cast<float2*>(MW + (32 + i0 + a) * MP + j0) = make_float2(w[a][0], w[a][1]);
            __syncthreads();
            float xo[2][2] = {{0.f, 0.f}, {0.f, 0.f}};
#pragma unroll 4
            for (int k = 0; k <= i0 + 1; ++k) {   // N21 = -N22 W (N22 lower triangular)
                const float n0 = MX[(32 + i0) * MP + 32 + k], n1 = MX[(33 + i0) * MP + 32 + k];
                const float2 wv = *reinterpret_cast<const float2*>(MW + (32 + k) * MP + j0);
                xo[0][0] = fmaf(n0, wv.x, xo[0][0]);
                xo[0][1] = fmaf(n0, wv.y, xo[0][1]);
                xo[1][0] = fmaf(n1, wv.x, xo[1][0]);
                xo[1][1] = fmaf(n1, wv.y, xo[1][1]);
            }
#pragma unroll
            for (int a = 0; a < 2; ++a)
                *reinterpret_cast<float2*>(MX + (32 + i0 + a) * MP + j0) = make_float2(-xo[a][0], -xo[a][1]);
            __syncthreads();
        }
        for (int i = tid; i < 64 * 16; i += kThreads) {
            const int r = i >> 4, c4 = (i & 15) * 4;
            *reinterpret_cast<float4*>(p.Nout + mat + r * 64 + c4) = *reinterpret_cast<const float4*>(MX + r * MP + c4);
        }
    }
    // ---- T = N diag(beta) (sGLA: diag(beta)), then A T; bf16 hi/lo tiles
    float Tv[4][4];
#pragma unroll
    for (int a = 0; a < 4; ++a) {
        float nr[4];
        if (p.use_delta) ld4(MX + (R0 + a) * MP + S0, nr);
#pragma unroll
        for (int c2 = 0; c2 < 4; ++c2) {
            const int r = R0 + a, s2 = S0 + c2;
            const float nv = p.use_delta ? nr[c2] : (r == s2 ? 1.f : 0.f);
            Tv[a][c2] = (r >= s2) ? nv * bs[s2] : 0.f;
        }
    }
#pragma unroll
    for (int a = 0; a < 4; ++a) st4(MW + (R0 + a) * MP + S0, Tv[a][0], Tv[a][1], Tv[a][2], Tv[a][3]);
    __syncthreads();
    float ATv[4][4];   // (A T)[r][s] = sum_{j=s}^{r} A[r][j] T[j][s]
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int c2 = 0; c2 < 4; ++c2) ATv[a][c2] = 0.f;
    if (live) {
#pragma unroll 4
        for (int j = S0; j < R0 + 4; ++j) {
            float av[4], tv[4];
            ld4(MAT + j * MP + R0, av);
            ld4(MW + j * MP + S0, tv);
#pragma unroll
            for (int a = 0; a < 4; ++a)
#pragma unroll
                for (int c2 = 0; c2 < 4; ++c2) ATv[a][c2] = fmaf(av[a], tv[c2], ATv[a][c2]);
        }
    }
    __syncthreads();   // every matrix slot is free from here
    // images of the two tile blocks in their global layout (bf16 row-major 64-wide rows):
    // [T; A T] hi (128 x 64) then lo, and [A hi, A lo, T hi, T lo] (64 x 64 each), built in
    // slots 0-3 (each thread writes its rows: no transposed stores) and written by two bulk
    // copies
    __nv_bfloat16* stA2 = reinterpret_cast<__nv_bfloat16*>(sm);
    __nv_bfloat16* stBT = stA2 + 4 * 64 * 64;
#pragma unroll
    for (int a = 0; a < 4; ++a) {
        const int o = (R0 + a) * 64 + S0;
        put4(stA2 + o, stA2 + 8192 + o, Tv[a][0], Tv[a][1], Tv[a][2], Tv[a][3]);
        put4(stA2 + 4096 + o, stA2 + 12288 + o, ATv[a][0], ATv[a][1], ATv[a][2], ATv[a][3]);
    }
    if (p.BTout) {
#pragma unroll
        for (int a = 0; a < 4; ++a) {
            const int o = (R0 + a) * 64 + S0;
            put4(stBT + o, stBT + 4096 + o, Av[a][0], Av[a][1], Av[a][2], Av[a][3]);
            put4(stBT + 8192 + o, stBT + 12288 + o, Tv[a][0], Tv[a][1], Tv[a][2], Tv[a][3]);
        }
    }
    fence_proxy_async_smem();
    __syncthreads();
    const size_t m2 = ((size_t(b) * H + h) * NT + c) * (4 * 64 * 64);
    if (tid == 0) {
        bulk_store(p.A2out + m2, stA2, 4 * 64 * 64 * 2);
        if (p.BTout) bulk_store(p.BTout + m2, stBT, 4 * 64 * 64 * 2);
        bulk_commit();
    }
    // coefficient block, slice-major: [a | b | w] each [E][64 rows], then gamma^C_e
    float* cf = p.coef + ((size_t(b) * H + h) * NT + c) * (3 * 64 * E + 16);
    for (int i = tid; i < 64 * E; i += kThreads) {
        const int e = i >> 6;
        const float Gr = Gs[i], GC = Gs[e * 64 + n - 1];
        const float gam = __expf(Gr);
        cf[i] = k2s[i] * gam;
        cf[64 * E + i] = q2s[i] * gam;
        cf[128 * E + i] = k2s[i] * __expf(GC - Gr);
    }
    if (tid < 16) cf[192 * E + tid] = tid < E ? __expf(Gs[tid * 64 + n - 1]) : 0.f;
    if (tid == 0) bulk_wait_read_all();   // the images stay in shared memory until read
}

size_t prep_tc_smem(int E) { return 1024 + size_t(5) * kSlot * 4 + (3 * 64 * E + 64) * 4; }

}  // namespace

cudaError_t launch_chunk_prep_tc(const tla_problem& p, const FwdPlan& fp, char* ws, int* err,
                                 cudaStream_t s) {
    CUtensorMap mk, mq;
    if (!make_token_map(&mk, p.k, p.B, p.T, p.H, p.dk, 64, 64, true) ||
        !make_token_map(&mq, p.q, p.B, p.T, p.H, p.dk, 64, 64, true))
        return cudaErrorInvalidValue;
    TcPrepArgs a;
    a.q2 = (const __nv_bfloat16*)p.q2;
    a.k2 = (const __nv_bfloat16*)p.k2;
    a.G = (const float*)(ws + fp.G);
    a.beta = p.beta;
    a.Aout = fp.need_A ? (float*)(ws + fp.A) : nullptr;   // read only by the CUDA-core backward
    a.Nout = p.use_delta ? (float*)(ws + fp.N) : nullptr;
    a.A2out = (__nv_bfloat16*)(ws + fp.A2);
    a.BTout = fp.tcb ? (__nv_bfloat16*)(ws + fp.BT) : nullptr;
    a.coef = (float*)(ws + fp.coef);
    a.err = err;
    a.ctab = p.cu_seqlens ? (const int2*)(ws + fp.ctab) : nullptr;
    a.T = p.T; a.H = p.H; a.E = p.E; a.NT = fp.NT; a.use_delta = p.use_delta; a.dk = p.dk;
    const size_t smem = prep_tc_smem(p.E);
    cudaFuncSetAttribute(chunk_prep_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    dim3 grid(fp.NT, p.H, p.B);
    prof_before("chunk_prep_tc", s);
    chunk_prep_tc_kernel<<<grid, kThreads, smem, s>>>(mk, mq, a);
    prof_after(s);
    return cudaGetLastError();
}

}  // namespace tla
