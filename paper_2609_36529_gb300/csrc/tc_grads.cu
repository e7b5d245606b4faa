// Tensor-core (tcgen05) chunk-parallel gradients of the backward (Appendix A,
// Kernels: after the reverse recurrence, every chunk's remaining gradients are
// computed independently; fixed-order reductions, no floating-point atomics).
//
// One CTA of 8 warps per (b, h, chunk).  With S_e = chunk-start state, dS'_e =
// gradient of the state at the chunk's end, and U, Res, dU, dRes of the chunk:
//   dQ = sum_e diag(b_e) dO S_e^T + P K,                       P = dA (.) R'
//   dK = sum_e [diag(a_e) (-dRes) S_e^T + diag(w_e) U dS'_e^T] + (dKK + dKK^T) K + P^T Q
//   db_e = rowdot(Q, dO S_e^T), da_e = rowdot(K, -dRes S_e^T), dw_e = rowdot(K, U dS'_e^T)
//   dgamma^C_e = <dS'_e, S_e>_F
//   dA = dO U^T, dT = dU Res^T (sGLA: dU V^T), and the C x C algebra of the UT
//   transform (dN, F = dN N^T, dM = -N^T F, dL, dKK, dR, dR', dbeta).
// Tensor-core products (fp32 accumulation in TMEM, non-exact operands as bf16 hi/lo):
//   phase 0  [K;Q] K^T -> K K^T, Q K^T;  dO U^T -> dA;  dU Res^T -> dT   (M=64 for the last two)
//   phase 1  (CUDA cores) C x C algebra, then ACC^T = [K; Q]^T [[P, 0], [Kc, P^T]]^T
//   phase 2  per slice e, transposed so that TMEM lanes index the key dimension d:
//              D1 = S_e [dO ; -dRes]^T   (128 x 128: query tokens, then key tokens)
//              D2 = dS'_e U^T            (128 x 64)
//            The slice's row scalings b_e, a_e, w_e are applied to D1/D2 in registers
//            (one thread per (d, 32 tokens)), and the row dots come from the same values
//            against the thread's column of Q or K, summed across the 128 lanes.  The
//            unscaled operands [dO ; -dRes] and U are staged once for all slices.
//   phase 3  dq = registers + ACC^T[:, 0:64]^T, dk = registers + ACC^T[:, 64:128]^T;
//            second keys/queries, log gates, beta.
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
constexpr int kBoxBytes = 64 * 64 * 2;     // one TMA box: 64 rows x 64 bf16
constexpr int kNBytes = 64 * 64 * 4;       // one C x C fp32 matrix in global memory
constexpr int MP = 68;                     // row stride (floats) of the shared C x C matrices
constexpr int kMat = 64 * MP;              // floats per shared C x C matrix
constexpr uint32_t kWorkBytes = 131072;    // [K;Q] tiles + phase 0/1 scratch; later two slabs
constexpr int GP = 68;                     // slice stride of the per-token arrays [E][GP] (float4
                                           // aligned, and slices fall on different banks)

struct TcGradArgs {
    const __nv_bfloat16* q2;
    const __nv_bfloat16* k2;
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
    const int2* ctab;    // packed documents: (first token, rows) of each chunk; else NULL
    float* scratch;      // E > 8: per chunk [3][64][E] fp32 partials (dk', dq', dG) in global
                         // memory, leaving the shared memory to the operands
    int T, H, dv, E, NT, use_delta, out_f32;
    int kdim;            // key dimension: 128, or 64 padded to 128 by zero rows (TMA fill)
};

// Copies of data this kernel reads once (the state and state-gradient slabs, the token
// tiles), with their L2 lines marked evict-first: streaming them then does not push out the
// next slice's slabs, which are prefetched into L2 one slice ahead.
__device__ __forceinline__ void tma_load_4d_once(void* dst, const CUtensorMap* map, uint64_t* bar,
                                                 int x, int y, int z, int w) {
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%0], [%1, {%2, %3, %4, %5}], [%6], %7;" ::"r"(smem_u32(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(w), "r"(smem_u32(bar)), "l"(pol)
        : "memory");
}
__device__ __forceinline__ void bulk_load_once(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%0], [%1], %2, [%3], %4;" ::"r"(smem_u32(dst)),
        "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(smem_u32(bar)), "l"(pol)
        : "memory");
}

// 4 x 4 block (rows R0.., columns S0..) of a shared row-major matrix.
__device__ __forceinline__ void ld4x4(const float* M, int R0, int S0, float (&v)[4][4]) {
#pragma unroll
    for (int a = 0; a < 4; ++a) {
        const float4 x = *reinterpret_cast<const float4*>(M + (R0 + a) * MP + S0);
        v[a][0] = x.x; v[a][1] = x.y; v[a][2] = x.z; v[a][3] = x.w;
    }
}

// out[a][c] = sum_x A[x][R0 + a] B[x][S0 + c]  (both operands stored with x as the row).
__device__ __forceinline__ void mm4x4(const float* A, const float* B, int R0, int S0, float (&out)[4][4]) {
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int c = 0; c < 4; ++c) out[a][c] = 0.f;
#pragma unroll 4
    for (int x = 0; x < 64; ++x) {
        const float4 u = *reinterpret_cast<const float4*>(A + x * MP + R0);
        const float4 w = *reinterpret_cast<const float4*>(B + x * MP + S0);
        const float ua[4] = {u.x, u.y, u.z, u.w}, wb[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
        for (int a = 0; a < 4; ++a)
#pragma unroll
            for (int c = 0; c < 4; ++c) out[a][c] = fmaf(ua[a], wb[c], out[a][c]);
    }
}

// Four consecutive values as bf16 hi/lo (8 bytes into each tile).
__device__ __forceinline__ void st4_split(uint8_t* hi, uint8_t* lo, uint32_t off, float v0, float v1,
                                          float v2, float v3) {
    const __nv_bfloat162 h0 = __floats2bfloat162_rn(v0, v1), h1 = __floats2bfloat162_rn(v2, v3);
    const float2 f0 = __bfloat1622float2(h0), f1 = __bfloat1622float2(h1);
    const __nv_bfloat162 l0 = __floats2bfloat162_rn(v0 - f0.x, v1 - f0.y);
    const __nv_bfloat162 l1 = __floats2bfloat162_rn(v2 - f1.x, v3 - f1.y);
    *reinterpret_cast<uint2*>(hi + off) =
        make_uint2(*reinterpret_cast<const uint32_t*>(&h0), *reinterpret_cast<const uint32_t*>(&h1));
    *reinterpret_cast<uint2*>(lo + off) =
        make_uint2(*reinterpret_cast<const uint32_t*>(&l0), *reinterpret_cast<const uint32_t*>(&l1));
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

// Four consecutive bf16 values (8-byte aligned) as fp32.
__device__ __forceinline__ void load_bf16x4(const __nv_bfloat16* src, float* v) {
    const uint2 u = *reinterpret_cast<const uint2*>(src);
    const float2 lo = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.x));
    const float2 hi = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.y));
    v[0] = lo.x; v[1] = lo.y; v[2] = hi.x; v[3] = hi.y;
}

// One halving step of a warp transpose-reduction over 2S values per lane.
template <int S>
__device__ __forceinline__ void xreduce_step(float* v, int lane) {
    const bool up = (lane & S) != 0;
#pragma unroll
    for (int k = 0; k < S; ++k) {
        const float send = up ? v[k] : v[k + S];
        const float keep = up ? v[k + S] : v[k];
        v[k] = keep + __shfl_xor_sync(0xffffffffu, send, S);
    }
}
// v[0..31] per lane -> the return value of lane l is the sum over the warp's lanes of v[l].
__device__ __forceinline__ float xreduce32(float* v, int lane) {
    xreduce_step<16>(v, lane);
    xreduce_step<8>(v, lane);
    xreduce_step<4>(v, lane);
    xreduce_step<2>(v, lane);
    xreduce_step<1>(v, lane);
    return v[0];
}

// Element j (0..31) of a thread's column of packed bf16 pairs, as fp32.
__device__ __forceinline__ float unpack_bf16(const uint32_t* pk, int j) {
    const uint32_t w = pk[j >> 1];
    return __uint_as_float((j & 1) ? (w & 0xffff0000u) : (w << 16));
}

// BIG: more than 8 slices, whose per-token partial sums of dk', dq' and dG live in a per-chunk
// global scratch (read and written a few times per element, L2-resident) instead of shared
// memory.
template <int OUT_F32, bool PACKED, bool BIG>
__global__ void __launch_bounds__(kThreads, 1)
bwd_chunk_grads_tc_kernel(const __grid_constant__ CUtensorMap map_k,
                          const __grid_constant__ CUtensorMap map_q,
                          const __grid_constant__ CUtensorMap map_do,
                          const __grid_constant__ CUtensorMap map_s,
                          const __grid_constant__ CUtensorMap map_ds, const TcGradArgs p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
    const int E = p.E, dv = p.dv, T = p.T, H = p.H, NT = p.NT;
    const int c = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
    // first token and rows of this chunk (packed documents: from the chunk table; a separate
    // instance, so that the regular one keeps t0 a compile-time multiple of 64)
    int t0 = c * 64, n = min(64, T - t0);
    if (PACKED) {
        const int2 cr = p.ctab[c];
        t0 = cr.x;
        n = cr.y;
    }
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const uint32_t T64 = 64u * dv * 2;         // bytes of a [64][dv] bf16 tile
    const int nb = dv / 64;                    // 64-column blocks of a value row

    // persistent operands (SW128 K-major over the value dimension)
    uint8_t* sB = sm;                          // [dO ; -dRes hi]: 128 rows, 16 KB per block
    uint8_t* sRlo = sB + 2 * T64;              // -dRes lo: 64 rows
    uint8_t* sUh = sRlo + T64;                 // U hi
    uint8_t* sUl = sUh + T64;                  // U lo
    uint8_t* W = sUl + T64;                    // 128 KB work region
    uint8_t* sKQ = W;                          // [K rows | Q rows] per 64-column block (TMA)
    uint8_t* scr = W + 4 * kBoxBytes;          // 96 KB: phase 0 staging, six C x C matrices, A3
    // per-token log decays, second keys and queries of the chunk, slice-major [E][GP]
    float* Gs = reinterpret_cast<float*>(W + kWorkBytes);
    __nv_bfloat16* k2s = reinterpret_cast<__nv_bfloat16*>(Gs + GP * E);
    __nv_bfloat16* q2s = k2s + GP * E;
    float* dwk = reinterpret_cast<float*>(q2s + GP * E);   // [64][E]
    float* bs = dwk + 64 * E;                  // [64]
    float* dba = bs + 64;                      // [64]
    float* dgc = dba + 64;                     // [16]
    float* scl = dgc + 16;                     // [2][3][64]: b_e, a_e, w_e (slice parity)
    float* red = scl + 384;                    // [3][4][64] row-dot partials per lane quarter
    float* frw = red + 768;                    // [2][8] Frobenius partials per warp (slice parity)
    // [64][E] partial sums of dk', dq', dG: shared memory, or this chunk's global scratch
    float* dk2a = BIG ? p.scratch + ((size_t(b) * H + h) * NT + c) * (3 * 64 * E) : frw + 16;
    float* dq2a = dk2a + 64 * E;
    float* dGa = dq2a + 64 * E;

    __shared__ __align__(8) uint64_t bar_ld, bar_mma, bar_q[4], bar_mh[2], bar_fh[2];
    __shared__ uint32_t tmem_slot;

    const size_t sbase = ((size_t(b) * H + h) * NT + c) * E;   // this chunk's first slab
    const uint32_t slab_bytes = uint32_t(kDk) * dv * 4;        // hi tile + lo tile
    const uint8_t* gS = reinterpret_cast<const uint8_t*>(p.Sck);
    const uint8_t* gD = reinterpret_cast<const uint8_t*>(p.dSck);

    if (warp == 0) {
        tmem_alloc(&tmem_slot, 512);
        tmem_relinquish();
    }
    if (tid == 0) {
        mbar_init(&bar_ld, 1);
        mbar_init(&bar_mma, 1);
        for (int q = 0; q < 4; ++q) mbar_init(&bar_q[q], 1);
        for (int j = 0; j < 2; ++j) {
            mbar_init(&bar_mh[j], 1);
            mbar_init(&bar_fh[j], kThreads / 32 - 1);   // one arrival per warp 1..7
        }
        fence_barrier_init();
        const size_t ci = (size_t(b) * H + h) * NT + c;
        const uint32_t tt = 2 * T64;   // one token tile: hi then lo
        // one arrival per phase (the barrier counts a single arrival): every byte of the
        // tensor loads and the token-tile copies is announced here, before any copy starts
        mbar_arrive_expect_tx(&bar_ld, 4 * kBoxBytes + nb * kBoxBytes + 3 * tt + (p.use_delta ? tt : 0));
        for (int j = 0; j < 2; ++j) {
            tma_load_4d_once(sKQ + j * 2 * kBoxBytes, &map_k, &bar_ld, 64 * j, h, t0, b);
            tma_load_4d_once(sKQ + j * 2 * kBoxBytes + kBoxBytes, &map_q, &bar_ld, 64 * j, h, t0, b);
        }
        for (int j = 0; j < nb; ++j) tma_load_4d_once(sB + j * 2 * kBoxBytes, &map_do, &bar_ld, 64 * j, h, t0, b);
        bulk_load_once(sUh, reinterpret_cast<const uint8_t*>(p.Ubuf) + ci * tt, tt, &bar_ld);
        bulk_load_once(scr, reinterpret_cast<const uint8_t*>(p.dUbuf) + ci * tt, tt, &bar_ld);
        bulk_load_once(scr + tt, reinterpret_cast<const uint8_t*>(p.Rbuf) + ci * tt, tt, &bar_ld);
        if (p.use_delta) {
            const uint8_t* g = reinterpret_cast<const uint8_t*>(p.dRbuf) + ci * tt;
            for (int j = 0; j < nb; ++j) bulk_load_once(sB + j * 16384 + 8192, g + j * 8192, 8192, &bar_ld);
            bulk_load_once(sRlo, g + T64, T64, &bar_ld);
        }
        bulk_prefetch_l2(gS + sbase * slab_bytes, slab_bytes);
        if (p.use_delta) bulk_prefetch_l2(p.Nmat + ((size_t(b) * H + h) * NT + c) * (64 * 64), kNBytes);
        bulk_prefetch_l2(gD + sbase * slab_bytes, slab_bytes);
    }
    for (int i = tid; i < 64 * E; i += kThreads) {
        const int r = i / E, e = i - (i / E) * E;
        const int rr = r < n ? r : n - 1;
        Gs[e * GP + r] = p.G[tok_idx(b, t0 + rr, h, e, T, H, E)];
        k2s[e * GP + r] = r < n ? p.k2[tok_idx(b, t0 + r, h, e, T, H, E)] : __float2bfloat16_rn(0.f);
        q2s[e * GP + r] = r < n ? p.q2[tok_idx(b, t0 + r, h, e, T, H, E)] : __float2bfloat16_rn(0.f);
    }
    if (tid < 64) {
        bs[tid] = tid < n ? (p.beta ? p.beta[(size_t(b) * T + t0 + tid) * H + h] : 1.f) : 0.f;
        dba[tid] = 0.f;
    }
    if (tid < 16) dgc[tid] = 0.f;

    // ---- staging: the token tiles arrive by bulk copy (U -> sUh/sUl; dU, Res -> scratch for
    //      dT; -dRes -> sB rows 64..127 (hi) and sRlo (lo)); sGLA has no -dRes operand
    uint8_t* sdUh = scr;
    uint8_t* sdUl = scr + T64;
    uint8_t* sRh = scr + 2 * T64;
    uint8_t* sRl = scr + 3 * T64;
    if (!p.use_delta)
        for (int i = tid; i < nb * 512; i += kThreads)
            *reinterpret_cast<uint4*>(sB + (i >> 9) * 16384 + 8192 + (i & 511) * 16) = make_uint4(0, 0, 0, 0);
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;
    const uint32_t tACC = tmem;   // phase 2: D1/D2 at columns 128/256 (even slices), 320/448 (odd)

    uint32_t mph = 0;
    // Failure exit: record the timeout, wait (bounded) for this CTA's copies and
    // products still in flight, free TMEM.
    auto bail = [&](uint64_t* pend_a, uint32_t pa, uint64_t* pend_b, uint32_t pb, bool mma) {
        if (tid == 0) {
            record_device_error(p.err, TLA_ERR_TIMEOUT);
            if (pend_a) mbar_wait(pend_a, pa);
            if (pend_b) mbar_wait(pend_b, pb);
            if (mma) mbar_wait(&bar_mma, mph);
        }
        tc_fence_before();
        __syncthreads();
        if (warp == 0) tmem_dealloc(tmem, 512);
    };

    bool ok = mbar_wait(&bar_ld, 0);
    if (__syncthreads_or(!ok)) {
        bail(&bar_ld, 0, nullptr, 0, false);
        return;
    }

    // ---- phase 0 products
    if (tid == 0) {
        const uint32_t id_kq = idesc_bf16_f32(128, 64, 0, 0);
        for (int ks = 0; ks < kDk / 16; ++ks) {
            if (ks * 16 >= p.kdim) break;   // zero key columns past d_k
            const uint64_t a = smem_desc(smem_u32(sKQ) + (ks >> 2) * 2 * kBoxBytes + (ks & 3) * 32, 16, 1024);
            umma_bf16(tmem + 128, a, a, id_kq, ks > 0 ? 1u : 0u);   // B = the key rows of the same tile
        }
        const uint32_t id64 = idesc_bf16_f32(64, 64, 0, 0);
        for (int ks = 0; ks < dv / 16; ++ks) {
            const uint32_t k32 = (ks & 3) * 32;
            const uint32_t o = (ks >> 2) * kBoxBytes + k32;
            const uint64_t a = smem_desc(smem_u32(sB) + (ks >> 2) * 2 * kBoxBytes + k32, 16, 1024);
            umma_bf16(tmem + 192, a, smem_desc(smem_u32(sUh) + o, 16, 1024), id64, ks > 0 ? 1u : 0u);
            umma_bf16(tmem + 192, a, smem_desc(smem_u32(sUl) + o, 16, 1024), id64, 1u);
            const uint64_t uh = smem_desc(smem_u32(sdUh) + o, 16, 1024);
            const uint64_t ul = smem_desc(smem_u32(sdUl) + o, 16, 1024);
            const uint64_t rh = smem_desc(smem_u32(sRh) + o, 16, 1024);
            const uint64_t rl = smem_desc(smem_u32(sRl) + o, 16, 1024);
            umma_bf16(tmem + 256, uh, rh, id64, ks > 0 ? 1u : 0u);
            umma_bf16(tmem + 256, uh, rl, id64, 1u);
            umma_bf16(tmem + 256, ul, rh, id64, 1u);
        }
        umma_commit(&bar_mma);
    }
    // N (the chunk's (I + L)^-1, row-major) into registers while the products run
    const size_t mat = ((size_t(b) * H + h) * NT + c) * (64 * 64);
    float nv[16];
#pragma unroll
    for (int k = 0; k < 16; ++k) nv[k] = p.use_delta ? p.Nmat[mat + tid + k * kThreads] : 0.f;
    ok = mbar_wait(&bar_mma, mph);
    if (__syncthreads_or(!ok)) {
        bail(nullptr, 0, nullptr, 0, true);
        return;
    }
    mph ^= 1;
    tc_fence_after();

    // fp32 C x C matrices in the scratch area: row-major, row stride MP (float4-aligned rows)
    float* Mkk = reinterpret_cast<float*>(scr);
    float* Mqk = Mkk + kMat;
    float* MdA = Mqk + kMat;
    float* MdT = MdA + kMat;
    // TMEM -> KK, QK (M = 128: rows are lanes), dA, dT (M = 64: rows 16 per lane quarter)
    {
        const int wq = warp & 3, L = wq * 32 + lane;
        if (warp < 4) {
            float* dst = (L < 64 ? Mkk : Mqk) + (L & 63) * MP;
            for (int j = 0; j < 64; j += 16) {
                float v[16];
                tmem_ld16(tmem_lane_addr(tmem + 128, warp, j), v);
                tmem_wait_ld();
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    *reinterpret_cast<float4*>(dst + j + 4 * q) =
                        make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
            }
        } else {
            const int r = 16 * wq + (lane & 15);
            for (int j = 0; j < 64; j += 16) {
                float va[16], vt[16];
                tmem_ld16(tmem_lane_addr(tmem + 192, warp, j), va);
                tmem_ld16(tmem_lane_addr(tmem + 256, warp, j), vt);
                tmem_wait_ld();
                if (lane < 16)
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        *reinterpret_cast<float4*>(MdA + r * MP + j + 4 * q) =
                            make_float4(va[4 * q], va[4 * q + 1], va[4 * q + 2], va[4 * q + 3]);
                        *reinterpret_cast<float4*>(MdT + r * MP + j + 4 * q) =
                            make_float4(vt[4 * q], vt[4 * q + 1], vt[4 * q + 2], vt[4 * q + 3]);
                    }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    // ---- phase 1: C x C algebra on CUDA cores; each thread owns the 4 x 4 block of
    // rows R0..R0+3 and columns S0..S0+3.
    const int R0 = 4 * (tid >> 4), S0 = 4 * (tid & 15);
    float KK[4][4], QK[4][4], dA[4][4], dT[4][4];
    ld4x4(Mkk, R0, S0, KK);
    ld4x4(Mqk, R0, S0, QK);
    ld4x4(MdA, R0, S0, dA);
    ld4x4(MdT, R0, S0, dT);
    __syncthreads();
    float* Nm = reinterpret_cast<float*>(scr);   // N
    float* NmT = Nm + kMat;                       // N^T
    float* dNT = NmT + kMat;                       // dN^T, then dR
    float* Fm = dNT + kMat;                       // F, then dR'
    float* dKKm = Fm + kMat;                      // dKK
    if (p.use_delta)
#pragma unroll
        for (int k = 0; k < 16; ++k) {
            const int i = tid + k * kThreads, x = i >> 6, s = i & 63;
            Nm[x * MP + s] = nv[k];
            NmT[s * MP + x] = nv[k];
        }
    float Rv[4][4], Rq[4][4];   // sum_e k2_e(r) k2_e(s) exp(G_e(r) - G_e(s)), same with q2_e(r), r >= s
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int c2 = 0; c2 < 4; ++c2) Rv[a][c2] = Rq[a][c2] = 0.f;
    for (int e = 0; e < E; ++e) {
        float gs[4], ksv[4], grv[4], krv[4], qrv[4];
        {   // four consecutive tokens of slice e: one 16-byte / 8-byte load each
            const float4 g4 = *reinterpret_cast<const float4*>(Gs + e * GP + S0);
            const float4 h4 = *reinterpret_cast<const float4*>(Gs + e * GP + R0);
            gs[0] = g4.x; gs[1] = g4.y; gs[2] = g4.z; gs[3] = g4.w;
            grv[0] = h4.x; grv[1] = h4.y; grv[2] = h4.z; grv[3] = h4.w;
            load_bf16x4(k2s + e * GP + S0, ksv);
            load_bf16x4(k2s + e * GP + R0, krv);
            load_bf16x4(q2s + e * GP + R0, qrv);
        }
        // the block's 16 exponentials first (independent), then the sums
        float ks2[4][4];
#pragma unroll
        for (int a = 0; a < 4; ++a)
#pragma unroll
            for (int c2 = 0; c2 < 4; ++c2)   // exp of a non-positive difference
                ks2[a][c2] = __expf(fminf(grv[a] - gs[c2], 0.f));
#pragma unroll
        for (int a = 0; a < 4; ++a)
#pragma unroll
            for (int c2 = 0; c2 < 4; ++c2) {
                // entries above the diagonal are discarded
                const float kg = (R0 + a >= S0 + c2) ? ksv[c2] * ks2[a][c2] : 0.f;
                Rv[a][c2] = fmaf(krv[a], kg, Rv[a][c2]);
                Rq[a][c2] = fmaf(qrv[a], kg, Rq[a][c2]);
            }
    }
    __syncthreads();
    float dKK[4][4], rp[4];
    if (p.use_delta) {
        {   // dN = dT diag(beta) (stored transposed); column terms of dbeta: sum_r dT (.) N
            float cp[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
            for (int a = 0; a < 4; ++a) {
                const float4 nr = *reinterpret_cast<const float4*>(Nm + (R0 + a) * MP + S0);
                cp[0] = fmaf(dT[a][0], nr.x, cp[0]);
                cp[1] = fmaf(dT[a][1], nr.y, cp[1]);
                cp[2] = fmaf(dT[a][2], nr.z, cp[2]);
                cp[3] = fmaf(dT[a][3], nr.w, cp[3]);
            }
#pragma unroll
            for (int c2 = 0; c2 < 4; ++c2) {
                const float bsv = bs[S0 + c2];
                *reinterpret_cast<float4*>(dNT + (S0 + c2) * MP + R0) =
                    make_float4(dT[0][c2] * bsv, dT[1][c2] * bsv, dT[2][c2] * bsv, dT[3][c2] * bsv);
                cp[c2] += __shfl_xor_sync(0xffffffffu, cp[c2], 16);
            }
            if (lane < 16)
#pragma unroll
                for (int c2 = 0; c2 < 4; ++c2) red[warp * 64 + S0 + c2] = cp[c2];
        }
        __syncthreads();
        if (tid < 64) {
            float acc = 0.f;
#pragma unroll
            for (int w = 0; w < kThreads / 32; ++w) acc += red[w * 64 + tid];
            dba[tid] += acc;
        }
        {   // F = dN N^T
            float F[4][4];
            mm4x4(dNT, NmT, R0, S0, F);
#pragma unroll
            for (int a = 0; a < 4; ++a)
                *reinterpret_cast<float4*>(Fm + (R0 + a) * MP + S0) = make_float4(F[a][0], F[a][1], F[a][2], F[a][3]);
        }
        __syncthreads();
        float dL[4][4];   // dM = -N^T F, strictly lower part
        mm4x4(Nm, Fm, R0, S0, dL);
#pragma unroll
        for (int a = 0; a < 4; ++a)
#pragma unroll
            for (int c2 = 0; c2 < 4; ++c2) dL[a][c2] = (R0 + a > S0 + c2) ? -dL[a][c2] : 0.f;
        __syncthreads();
#pragma unroll
        for (int a = 0; a < 4; ++a) {
            const float br = bs[R0 + a];
            float dR[4];
            rp[a] = 0.f;
#pragma unroll
            for (int c2 = 0; c2 < 4; ++c2) {
                dR[c2] = dL[a][c2] * br * KK[a][c2];
                dKK[a][c2] = dL[a][c2] * br * Rv[a][c2];
                rp[a] = fmaf(dL[a][c2] * KK[a][c2], Rv[a][c2], rp[a]);   // row terms of dbeta
            }
            *reinterpret_cast<float4*>(dNT + (R0 + a) * MP + S0) = make_float4(dR[0], dR[1], dR[2], dR[3]);
            *reinterpret_cast<float4*>(dKKm + (R0 + a) * MP + S0) =
                make_float4(dKK[a][0], dKK[a][1], dKK[a][2], dKK[a][3]);
        }
    } else {
#pragma unroll
        for (int a = 0; a < 4; ++a) {
            rp[a] = 0.f;
#pragma unroll
            for (int c2 = 0; c2 < 4; ++c2) {
                dKK[a][c2] = 0.f;
                if (R0 + a == S0 + c2) rp[a] = dT[a][c2];   // T = diag(beta)
            }
            *reinterpret_cast<float4*>(dNT + (R0 + a) * MP + S0) = make_float4(0.f, 0.f, 0.f, 0.f);
            *reinterpret_cast<float4*>(dKKm + (R0 + a) * MP + S0) = make_float4(0.f, 0.f, 0.f, 0.f);
        }
    }
    // row sums of dbeta's row terms over the 16 threads of a half-warp (one half-warp per row block)
#pragma unroll
    for (int a = 0; a < 4; ++a) {
#pragma unroll
        for (int s = 1; s < 16; s <<= 1) rp[a] += __shfl_xor_sync(0xffffffffu, rp[a], s);
    }
    if ((tid & 15) == 0)
#pragma unroll
        for (int a = 0; a < 4; ++a) dba[R0 + a] += rp[a];
    float Pv[4][4];   // P = dA (.) R'
#pragma unroll
    for (int a = 0; a < 4; ++a) {
        float dRq[4];
#pragma unroll
        for (int c2 = 0; c2 < 4; ++c2) {
            const bool low = R0 + a >= S0 + c2;
            dRq[c2] = low ? dA[a][c2] * QK[a][c2] : 0.f;
            Pv[a][c2] = low ? dA[a][c2] * Rq[a][c2] : 0.f;
        }
        *reinterpret_cast<float4*>(Fm + (R0 + a) * MP + S0) = make_float4(dRq[0], dRq[1], dRq[2], dRq[3]);
    }
    __syncthreads();
    {   // through R (dR) and R' (dR'): one (token, slice) pair per thread
        const float* dRm = dNT;
        const float* dRqm = Fm;
        for (int i = tid; i < 64 * E; i += kThreads) {
            const int x = i / E, e = i - (i / E) * E;
            const float gx = Gs[e * GP + x];
            const float kx = __bfloat162float(k2s[e * GP + x]), qx = __bfloat162float(q2s[e * GP + x]);
            float dk2v = 0.f, dq2v = 0.f, dGv = 0.f;
#pragma unroll 4
            for (int s = 0; s <= x; ++s) {
                const float gam = __expf(gx - Gs[e * GP + s]);
                const float ks = __bfloat162float(k2s[e * GP + s]);
                const float dR = dRm[x * MP + s], dRq = dRqm[x * MP + s];
                dk2v = fmaf(dR * ks, gam, dk2v);
                dq2v = fmaf(dRq * ks, gam, dq2v);
                dGv = fmaf((dR * kx + dRq * qx) * ks, gam, dGv);
            }
#pragma unroll 4
            for (int r = x; r < 64; ++r) {
                const float gam = __expf(Gs[e * GP + r] - gx);
                const float dR = dRm[r * MP + x], dRq = dRqm[r * MP + x];
                const float t = (dR * __bfloat162float(k2s[e * GP + r]) +
                                 dRq * __bfloat162float(q2s[e * GP + r])) * gam;
                dk2v += t;
                dGv = fmaf(-t, kx, dGv);
            }
            dk2a[i] = dk2v;
            dq2a[i] = dq2v;
            dGa[i] = dGv;
        }
    }
    __syncthreads();
    // B operands of the last products, bf16 hi/lo (K-major, 64 rows):
    //   Pt  = P                        (64 x 64)   -> dq rows
    //   KPt = [dKK + dKK^T | P^T]      (64 x 128)  -> dk rows
    uint8_t* Pth = scr;
    uint8_t* Ptl = scr + 8192;
    uint8_t* KPh = scr + 16384;
    uint8_t* KPl = scr + 32768;
#pragma unroll
    for (int a = 0; a < 4; ++a) {
        st4_split(Pth, Ptl, sw128_offset(R0 + a, S0, 64), Pv[a][0], Pv[a][1], Pv[a][2], Pv[a][3]);
        float kc4[4];
#pragma unroll
        for (int c2 = 0; c2 < 4; ++c2) kc4[c2] = dKK[a][c2] + dKKm[(S0 + c2) * MP + R0 + a];
        st4_split(KPh, KPl, sw128_offset(R0 + a, S0, 64), kc4[0], kc4[1], kc4[2], kc4[3]);
    }
#pragma unroll
    for (int c2 = 0; c2 < 4; ++c2)
        st4_split(KPh, KPl, sw128_offset(S0 + c2, 64 + R0, 64), Pv[0][c2], Pv[1][c2], Pv[2][c2], Pv[3][c2]);
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    // ACC^T (lanes = key dimension d, columns = output rows): [K]^T Pt^T, then [K;Q]^T KPt^T
    if (tid == 0) {
        const uint32_t id = idesc_bf16_f32(128, 64, 1, 0);
        for (int ks = 0; ks < 4; ++ks) {
            const uint64_t a = smem_desc(smem_u32(sKQ) + ks * 2048, 2 * kBoxBytes, 1024);
            umma_bf16(tACC, a, smem_desc(smem_u32(Pth) + ks * 32, 16, 1024), id, ks > 0 ? 1u : 0u);
            umma_bf16(tACC, a, smem_desc(smem_u32(Ptl) + ks * 32, 16, 1024), id, 1u);
        }
        for (int ks = 0; ks < 8; ++ks) {
            const uint64_t a = smem_desc(smem_u32(sKQ) + ks * 2048, 2 * kBoxBytes, 1024);
            const uint32_t o = (ks >> 2) * 8192 + (ks & 3) * 32;
            umma_bf16(tACC + 64, a, smem_desc(smem_u32(KPh) + o, 16, 1024), id, ks > 0 ? 1u : 0u);
            umma_bf16(tACC + 64, a, smem_desc(smem_u32(KPl) + o, 16, 1024), id, 1u);
        }
        umma_commit(&bar_mma);
    }
    // this thread's key dimension d and token block, and its columns of K and Q (bf16 pairs)
    const int wq = warp & 3, tb = 32 * (warp >> 2), d = wq * 32 + lane;
    uint32_t kc[16], qc[16];
    {
        const uint8_t* kb = sKQ + (d >> 6) * 2 * kBoxBytes;
#pragma unroll
        for (int m = 0; m < 16; ++m) {
            const int t = tb + 2 * m;
            const uint32_t o0 = sw128_offset(t, d & 63, 64), o1 = sw128_offset(t + 1, d & 63, 64);
            kc[m] = uint32_t(*reinterpret_cast<const uint16_t*>(kb + o0)) |
                    (uint32_t(*reinterpret_cast<const uint16_t*>(kb + o1)) << 16);
            qc[m] = uint32_t(*reinterpret_cast<const uint16_t*>(kb + kBoxBytes + o0)) |
                    (uint32_t(*reinterpret_cast<const uint16_t*>(kb + kBoxBytes + o1)) << 16);
        }
    }
    ok = mbar_wait(&bar_mma, mph);
    if (__syncthreads_or(!ok)) {
        bail(nullptr, 0, nullptr, 0, true);
        return;
    }
    mph ^= 1;
    tc_fence_after();

    // ---- phase 2: per slice.  S_e and dS'_e (bf16 hi/lo, row-major checkpoints) arrive by TMA
    // in the operand layout, one 64-column half of each per quarter of the work region, with a
    // barrier per quarter.  The slice is pipelined by halves: thread 0 issues half j's products
    // as soon as its quarters land (committed to bar_mh[j]); warps 1-7 take half j's part of the
    // Frobenius sum (bar_fh[j]); once both are done the half's quarters take the next slice's
    // copies, while the other half is still being multiplied.  Slice e-1's epilogue runs on all
    // warps meanwhile (D1/D2 double-buffered in TMEM).  Every barrier of this phase completes
    // once per slice, so the parity of slice e is e & 1.
    uint32_t pend = 0, mpend = 0;   // thread 0: quarters with copies in flight, halves with products
    int pend_slice = 0;             // thread 0: the slice those copies belong to
    auto quarter = [&](int which, int j) { return W + (2 * j + which) * 32768; };   // 0: S, 1: dS'
    auto issue_half = [&](int e, int j) {
        for (int which = 0; which < 2; ++which) {
            uint64_t* bar = &bar_q[2 * j + which];
            mbar_arrive_expect_tx(bar, 32768);   // [hi | lo][128][64 columns]
            tma_load_4d_once(quarter(which, j), which ? &map_ds : &map_s, bar, 64 * j, 0, int(sbase + e), 0);
            pend |= 1u << (2 * j + which);
        }
        pend_slice = e;
        if (j == 0 && e + 1 < E) {
            bulk_prefetch_l2(gS + (sbase + e + 1) * slab_bytes, slab_bytes);
            bulk_prefetch_l2(gD + (sbase + e + 1) * slab_bytes, slab_bytes);
        }
    };
    auto fail = [&](int e) {   // timeout: record it, drain this CTA's copies and products
        if (tid == 0) {
            record_device_error(p.err, TLA_ERR_TIMEOUT);
            for (int q = 0; q < 4; ++q)
                if ((pend >> q) & 1) mbar_wait(&bar_q[q], pend_slice & 1);
            for (int j = 0; j < 2; ++j)
                if ((mpend >> j) & 1) mbar_wait(&bar_mh[j], e & 1);
        }
        tc_fence_before();
        __syncthreads();
        if (warp == 0) tmem_dealloc(tmem, 512);
    };
    if (tid == 0)
        for (int j = 0; j < nb; ++j) issue_half(0, j);
    float acq[32], ack[32];
#pragma unroll
    for (int j = 0; j < 32; ++j) acq[j] = ack[j] = 0.f;
    for (int e = 0; e <= E; ++e) {   // e == E only finishes slice E-1
        const bool act = e < E;
        const int pb = e & 1;
        const uint32_t par = e & 1;
        bool ok = true;
        // the row-dot partials of slice e-2 have been read (end of the last iteration)
        tc_fence_before();
        __syncthreads();
        tc_fence_after();
        if (act) {
            if (tid < 192) {   // b_e, a_e, w_e of the 64 tokens
                const int r = tid & 63, i = e * GP + r;
                float sv;
                if (tid < 64) sv = __bfloat162float(q2s[i]) * __expf(Gs[i]);
                else if (tid < 128) sv = __bfloat162float(k2s[i]) * __expf(Gs[i]);
                else sv = __bfloat162float(k2s[i]) * __expf(Gs[e * GP + n - 1] - Gs[i]);
                scl[pb * 192 + tid] = sv;
            }
            if (warp == 0) {
                if (lane == 0) {   // D1 = S_e [dO; -dRes]^T, D2 = dS'_e U^T, by halves of K = dv
                    const uint32_t d1 = pb ? tmem + 320 : tmem + 128, d2 = pb ? tmem + 448 : tmem + 256;
                    const uint32_t id128 = idesc_bf16_f32(128, 128, 0, 0);
                    const uint32_t id64 = idesc_bf16_f32(128, 64, 0, 0);
                    for (int j = 0; j < nb && ok; ++j) {
                        ok = mbar_wait(&bar_q[2 * j], par) && mbar_wait(&bar_q[2 * j + 1], par);
                        if (!ok) break;
                        pend &= ~(3u << (2 * j));
                        const uint32_t qs = smem_u32(quarter(0, j)), qd = smem_u32(quarter(1, j));
                        for (int kk = 0; kk < 4; ++kk) {
                            const uint32_t k32 = kk * 32, acc = (j > 0 || kk > 0) ? 1u : 0u;
                            const uint64_t sh = smem_desc(qs + k32, 16, 1024);
                            const uint64_t sl = smem_desc(qs + 16384 + k32, 16, 1024);
                            const uint64_t bh = smem_desc(smem_u32(sB) + j * 16384 + k32, 16, 1024);
                            umma_bf16(d1, sh, bh, id128, acc);
                            umma_bf16(d1, sl, bh, id128, 1u);
                            if (p.use_delta)
                                umma_bf16(d1 + 64, sh, smem_desc(smem_u32(sRlo) + j * 8192 + k32, 16, 1024), id64, 1u);
                            const uint64_t dh = smem_desc(qd + k32, 16, 1024);
                            const uint64_t dl = smem_desc(qd + 16384 + k32, 16, 1024);
                            const uint64_t uh = smem_desc(smem_u32(sUh) + j * 8192 + k32, 16, 1024);
                            const uint64_t ul = smem_desc(smem_u32(sUl) + j * 8192 + k32, 16, 1024);
                            umma_bf16(d2, dh, uh, id64, acc);
                            umma_bf16(d2, dl, uh, id64, 1u);
                            umma_bf16(d2, dh, ul, id64, 1u);
                        }
                        umma_commit(&bar_mh[j]);
                        mpend |= 1u << j;
                    }
                    // a half's quarters are free once its products and Frobenius part have read them
                    for (int j = 0; j < nb && ok; ++j) {
                        ok = mbar_wait(&bar_mh[j], par) && mbar_wait(&bar_fh[j], par);
                        if (!ok) break;
                        mpend &= ~(1u << j);
                        if (e + 1 < E) issue_half(e + 1, j);
                    }
                }
                __syncwarp();
            } else {   // <dS'_e, S_e> (hi + lo reproduces each value to ~2^-16), warps 1..7
                float fro = 0.f;
                for (int j = 0; j < nb; ++j) {
                    ok = ok && mbar_wait(&bar_q[2 * j], par) && mbar_wait(&bar_q[2 * j + 1], par);
                    if (ok) {
                        const uint8_t* qsb = quarter(0, j);
                        const uint8_t* qdb = quarter(1, j);
                        for (uint32_t o = (tid - 32) * 16; o < 16384; o += (kThreads - 32) * 16) {
                            float sh[8], sl[8], dh[8], dl[8];
                            load_bf16x8(qsb + o, sh);
                            load_bf16x8(qsb + 16384 + o, sl);
                            load_bf16x8(qdb + o, dh);
                            load_bf16x8(qdb + 16384 + o, dl);
#pragma unroll
                            for (int u = 0; u < 8; ++u) fro = fmaf(dh[u] + dl[u], sh[u] + sl[u], fro);
                        }
                    }
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&bar_fh[j]);   // also on failure: thread 0's wait stays bounded
                }
#pragma unroll
                for (int sft = 16; sft >= 1; sft >>= 1) fro += __shfl_xor_sync(0xffffffffu, fro, sft);
                if (lane == 0) frw[pb * 8 + warp] = fro;
            }
        }
        if (e > 0) {   // epilogue of slice e-1 (its D1/D2 and scales)
            const int ep = (e - 1) & 1;
            const uint32_t d1 = ep ? tmem + 320 : tmem + 128, d2 = ep ? tmem + 448 : tmem + 256;
            const float* sc = scl + ep * 192;
            float z[32];
            // D1 query columns: dq += b_e (dO S_e^T); db_e = rowdot(Q, dO S_e^T)
            tmem_ld16(tmem_lane_addr(d1, warp, tb), z);
            tmem_ld16(tmem_lane_addr(d1, warp, tb + 16), z + 16);
            tmem_wait_ld();
#pragma unroll
            for (int jj = 0; jj < 32; ++jj) {
                acq[jj] = fmaf(sc[tb + jj], z[jj], acq[jj]);
                z[jj] *= unpack_bf16(qc, jj);
            }
            red[(0 * 4 + wq) * 64 + tb + lane] = xreduce32(z, lane);
            // D1 key columns: dk += a_e (-dRes S_e^T); da_e = rowdot(K, -dRes S_e^T)
            tmem_ld16(tmem_lane_addr(d1, warp, 64 + tb), z);
            tmem_ld16(tmem_lane_addr(d1, warp, 64 + tb + 16), z + 16);
            tmem_wait_ld();
#pragma unroll
            for (int jj = 0; jj < 32; ++jj) {
                ack[jj] = fmaf(sc[64 + tb + jj], z[jj], ack[jj]);
                z[jj] *= unpack_bf16(kc, jj);
            }
            red[(1 * 4 + wq) * 64 + tb + lane] = xreduce32(z, lane);
            // D2: dk += w_e (U dS'_e^T); dw_e = rowdot(K, U dS'_e^T)
            tmem_ld16(tmem_lane_addr(d2, warp, tb), z);
            tmem_ld16(tmem_lane_addr(d2, warp, tb + 16), z + 16);
            tmem_wait_ld();
#pragma unroll
            for (int jj = 0; jj < 32; ++jj) {
                ack[jj] = fmaf(sc[128 + tb + jj], z[jj], ack[jj]);
                z[jj] *= unpack_bf16(kc, jj);
            }
            red[(2 * 4 + wq) * 64 + tb + lane] = xreduce32(z, lane);
        }
        tc_fence_before();
        if (__syncthreads_or(!ok)) {
            fail(e);
            return;
        }
        tc_fence_after();
        if (e > 0) {   // slice e-1's row dots -> dq2, dk2, dG (a_e = k2 gamma, b_e = q2 gamma, w_e)
            const int es = e - 1;
            if (tid < 64) {
                const int i = tid * E + es, ig = es * GP + tid;
                float db = 0.f, da = 0.f, dw = 0.f;
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    db += red[(0 * 4 + q) * 64 + tid];
                    da += red[(1 * 4 + q) * 64 + tid];
                    dw += red[(2 * 4 + q) * 64 + tid];
                }
                const float gam = __expf(Gs[ig]);
                const float wdec = __expf(Gs[es * GP + n - 1] - Gs[ig]);
                const float k2v = __bfloat162float(k2s[ig]), q2v = __bfloat162float(q2s[ig]);
                dk2a[i] += da * gam + dw * wdec;
                dq2a[i] += db * gam;
                dGa[i] += da * (k2v * gam) + db * (q2v * gam) - dw * (k2v * wdec);
                dwk[i] = dw;
            } else if (tid == 64) {
                float f = 0.f;
                for (int w = 1; w < kThreads / 32; ++w) f += frw[(es & 1) * 8 + w];
                dgc[es] = f;
            }
        }
    }

    // ---- phase 3: dq, dk = register sums + ACC^T, staged as [64 tokens][128] fp32 tiles in the
    // (now idle) work region and written as whole rows
    {
        float* dqs = reinterpret_cast<float*>(W);
        float* dks = dqs + 64 * kDk;
        float v[32];
        tmem_ld16(tmem_lane_addr(tACC, warp, tb), v);
        tmem_ld16(tmem_lane_addr(tACC, warp, tb + 16), v + 16);
        tmem_wait_ld();
#pragma unroll
        for (int j = 0; j < 32; ++j) dqs[(tb + j) * kDk + d] = acq[j] + v[j];
        tmem_ld16(tmem_lane_addr(tACC, warp, 64 + tb), v);
        tmem_ld16(tmem_lane_addr(tACC, warp, 64 + tb + 16), v + 16);
        tmem_wait_ld();
#pragma unroll
        for (int j = 0; j < 32; ++j) dks[(tb + j) * kDk + d] = ack[j] + v[j];
        __syncthreads();
        for (int i = tid; i < 2 * 64 * (kDk / 4); i += kThreads) {
            const int m = i >= 64 * (kDk / 4), j = i - m * 64 * (kDk / 4);
            const int t = j / (kDk / 4), c4 = (j % (kDk / 4)) * 4;
            if (t >= n || c4 >= p.kdim) continue;   // padded key columns are not outputs
            const float4 x = *reinterpret_cast<const float4*>((m ? dks : dqs) + t * kDk + c4);
            const size_t off = tok_idx(b, t0 + t, h, c4, T, H, p.kdim);
            void* dst = m ? p.dk : p.dq;
            if (OUT_F32) {
                *reinterpret_cast<float4*>(static_cast<float*>(dst) + off) = x;
            } else {
                const __nv_bfloat162 lo = __floats2bfloat162_rn(x.x, x.y), hi = __floats2bfloat162_rn(x.z, x.w);
                *reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(dst) + off) =
                    make_uint2(*reinterpret_cast<const uint32_t*>(&lo), *reinterpret_cast<const uint32_t*>(&hi));
            }
        }
    }
    __syncthreads();
    for (int e = warp; e < E; e += kThreads / 32) {   // a warp per slice: dgamma^C, then the
                                                      // reverse cumulative sum of dG
        const float gl = Gs[e * GP + n - 1];
        float dGC = 0.f;
        for (int r = lane; r < n; r += 32)
            dGC = fmaf(dwk[r * E + e], __bfloat162float(k2s[e * GP + r]) * __expf(gl - Gs[e * GP + r]), dGC);
#pragma unroll
        for (int s = 16; s >= 1; s >>= 1) dGC += __shfl_xor_sync(0xffffffffu, dGC, s);
        dGC = fmaf(dgc[e], __expf(gl), dGC);
        const int r0 = 2 * lane, r1 = r0 + 1;
        const float a0 = r0 < n ? dGa[r0 * E + e] + (r0 == n - 1 ? dGC : 0.f) : 0.f;
        const float a1 = r1 < n ? dGa[r1 * E + e] + (r1 == n - 1 ? dGC : 0.f) : 0.f;
        const float pair = a0 + a1;
        float suf = pair;   // inclusive suffix sum over lanes
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const float v = __shfl_down_sync(0xffffffffu, suf, off);
            if (lane + off < 32) suf += v;
        }
        float above = __shfl_down_sync(0xffffffffu, suf, 1);   // sum over the lanes above
        if (lane == 31) above = 0.f;
        const float s1 = a1 + above;
        if (r0 < n) p.dg[tok_idx(b, t0 + r0, h, e, T, H, E)] = a0 + s1;
        if (r1 < n) p.dg[tok_idx(b, t0 + r1, h, e, T, H, E)] = s1;
    }
    for (int i = tid; i < n * E; i += kThreads) {
        const int r = i / E, e = i - (i / E) * E;
        const size_t off = tok_idx(b, t0 + r, h, e, T, H, E);
        store_out(p.dq2, off, dq2a[i], OUT_F32);
        store_out(p.dk2, off, dk2a[i], OUT_F32);
    }
    if (p.dbeta && tid < n) p.dbeta[(size_t(b) * T + t0 + tid) * H + h] = dba[tid];
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tmem_dealloc(tmem, 512);
}

size_t grads_tc_smem(int E, int dv) {
    const size_t T64 = size_t(64) * dv * 2;
    // Gs, k2s, q2s, dwk, bs, dba, dgc, scl, red, frw, and dk2a, dq2a, dGa unless E > 8
    const size_t small = size_t(GP) * E * (4 + 2 + 2) + size_t(64) * E * 4 * (E > 8 ? 1 : 4) +
                         (64 + 64 + 16 + 384 + 768 + 16) * 4;
    return 1024 + 5 * T64 + kWorkBytes + small;
}

}  // namespace

int tc_grads_shape_ok(const tla_problem& p) {
    return (p.dk == kDk || p.dk == 64) && p.dv % 64 == 0 && p.dv <= 128 && p.E <= 16 &&
           grads_tc_smem(p.E, p.dv) <= 227 * 1024;
}

int tc_grads_ok(const tla_problem& p, const FwdPlan& fp) { return fp.ck_tiles && tc_grads_shape_ok(p); }

cudaError_t launch_bwd_chunk_grads_tc(const tla_problem& p, const FwdPlan& fp, const char* fws,
                                      const BwdPlan& bp, char* bws, const void* dO,
                                      void* dq, void* dk, void* dq2, void* dk2, float* dbeta,
                                      float* dg, int* err, cudaStream_t s) {
    CUtensorMap mk, mq, mo, ms, md;
    const long long nslab = (long long)p.B * p.H * fp.NT * p.E;
    if (!make_token_map(&mk, p.k, p.B, p.T, p.H, p.dk, 64, 64, true) ||
        !make_token_map(&mq, p.q, p.B, p.T, p.H, p.dk, 64, 64, true) ||
        !make_token_map(&mo, dO, p.B, p.T, p.H, p.dv, 64, 64, true) ||
        !make_ckpt_map(&ms, fws + fp.S, nslab, p.dv, 64, 1, 128) ||
        !make_ckpt_map(&md, bws + bp.dS, nslab, p.dv, 64, 1, 128))
        return cudaErrorInvalidValue;
    TcGradArgs a;
    a.q2 = (const __nv_bfloat16*)p.q2;
    a.k2 = (const __nv_bfloat16*)p.k2;
    a.G = (const float*)(fws + fp.G);
    a.beta = p.beta;
    a.Nmat = p.use_delta ? (const float*)(fws + fp.N) : nullptr;
    a.Sck = (const float*)(fws + fp.S);
    a.Ubuf = (const float*)(fws + fp.U);
    a.Rbuf = (const float*)(fws + fp.Res);
    a.dUbuf = (const float*)(bws + bp.dU);
    a.dRbuf = (const float*)(bws + bp.dRes);
    a.dSck = (const float*)(bws + bp.dS);
    a.dq = dq; a.dk = dk; a.dq2 = dq2; a.dk2 = dk2; a.dbeta = dbeta; a.dg = dg;
    a.err = err;
    a.ctab = p.cu_seqlens ? (const int2*)(fws + fp.ctab) : nullptr;
    const bool big = p.E > 8;
    a.scratch = big ? (float*)(bws + bp.gscr) : nullptr;
    a.T = p.T; a.H = p.H; a.dv = p.dv; a.E = p.E; a.NT = fp.NT;
    a.use_delta = p.use_delta; a.out_f32 = p.out_dtype == TLA_FP32; a.kdim = p.dk;
    const size_t smem = grads_tc_smem(p.E, p.dv);
    auto kern = big ? (a.ctab ? (a.out_f32 ? bwd_chunk_grads_tc_kernel<1, true, true>
                                           : bwd_chunk_grads_tc_kernel<0, true, true>)
                              : (a.out_f32 ? bwd_chunk_grads_tc_kernel<1, false, true>
                                           : bwd_chunk_grads_tc_kernel<0, false, true>))
                    : (a.ctab ? (a.out_f32 ? bwd_chunk_grads_tc_kernel<1, true, false>
                                           : bwd_chunk_grads_tc_kernel<0, true, false>)
                              : (a.out_f32 ? bwd_chunk_grads_tc_kernel<1, false, false>
                                           : bwd_chunk_grads_tc_kernel<0, false, false>));
    cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    dim3 grid(fp.NT, p.H, p.B);
    prof_before("bwd_chunk_grads_tc", s);
    kern<<<grid, kThreads, smem, s>>>(mk, mq, mo, ms, md, a);
    prof_after(s);
    return cudaGetLastError();
}

}  // namespace tla
