// Per-chunk preparation for the tensor-core path (bf16 inputs, dk = 128).
// One CTA of 8 warps per (b, h, chunk) computes, Appendix A:
//   K K^T and Q K^T                  one UMMA [K; Q] K^T on the TMA key/query tile
//   R, R' element by element         exp of non-positive log-decay differences (Eq. joint-gram)
//   A = Q K^T (.) R' (lower incl. diagonal), L = tril(diag(beta)(K K^T (.) R), -1)
//   N = (I + L)^{-1}                 blocked: the four 16 x 16 diagonal blocks by forward
//                                    substitution (one warp each, registers only), then the
//                                    off-diagonal blocks by distance (Eq. joint-solve)
//   T = N diag(beta) (sGLA: diag(beta)), A T
// and writes A and N (fp32), the bf16 hi/lo tiles [T; A T] (forward recurrence) and
// [A^T; T^T] (backward recurrence), and the per-row coefficient block
// [k'_e gamma_e | q'_e gamma_e | k'_e gamma^C_e / gamma_e | gamma^C_e].
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
constexpr int MP = 65;

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
    int T, H, E, NT, use_delta;
};

__device__ __forceinline__ void put_pair(__nv_bfloat16* hi, __nv_bfloat16* lo, float x) {
    const __nv_bfloat16 h = __float2bfloat16_rn(x);
    *hi = h;
    *lo = __float2bfloat16_rn(x - __bfloat162float(h));
}

__global__ void __launch_bounds__(kThreads, 2)
chunk_prep_tc_kernel(const __grid_constant__ CUtensorMap map_k,
                     const __grid_constant__ CUtensorMap map_q, const TcPrepArgs p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
    const int E = p.E, T = p.T, H = p.H, NT = p.NT;
    const int c = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
    const int t0 = c * 64, n = min(64, T - t0);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    uint8_t* sKQ = sm;
    float* ML = reinterpret_cast<float*>(sm + 4 * kBoxBytes);   // K K^T -> L
    float* MA = ML + 64 * MP;                                   // Q K^T -> A
    float* MX = MA + 64 * MP;                                   // N = (I + L)^{-1}
    float* MW = MX + 64 * MP;                                   // block products
    float* Gs = MW + 64 * MP;
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
    for (int i = tid; i < 64 * E; i += kThreads) {
        const int r = i / E, e = i - (i / E) * E;
        const int rr = r < n ? r : n - 1;
        Gs[i] = p.G[tok_idx(b, t0 + rr, h, e, T, H, E)];
        k2s[i] = r < n ? __bfloat162float(p.k2[tok_idx(b, t0 + r, h, e, T, H, E)]) : 0.f;
        q2s[i] = r < n ? __bfloat162float(p.q2[tok_idx(b, t0 + r, h, e, T, H, E)]) : 0.f;
    }
    if (tid < 64) bs[tid] = tid < n ? (p.beta ? p.beta[(size_t(b) * T + t0 + tid) * H + h] : 1.f) : 0.f;
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;
    bool ok = mbar_wait(&bar_ld, 0);
    if (__syncthreads_or(!ok)) {
        if (tid == 0) record_device_error(p.err, TLA_ERR_TIMEOUT);
        __syncthreads();
        if (warp == 0) tmem_dealloc(tmem, 64);
        return;
    }
    if (tid == 0) {
        const uint32_t id = idesc_bf16_f32(128, 64, 0, 0);
        for (int ks = 0; ks < kDk / 16; ++ks) {
            const uint64_t a = smem_desc(smem_u32(sKQ) + (ks >> 2) * 2 * kBoxBytes + (ks & 3) * 32, 16, 1024);
            umma_bf16(tmem, a, a, id, ks > 0 ? 1u : 0u);
        }
        umma_commit(&bar_mma);
    }
    ok = mbar_wait(&bar_mma, 0);
    if (__syncthreads_or(!ok)) {
        if (tid == 0) record_device_error(p.err, TLA_ERR_TIMEOUT);
        __syncthreads();
        if (warp == 0) tmem_dealloc(tmem, 64);
        return;
    }
    tc_fence_after();
    if (warp < 4) {   // rows 0-63: K K^T, rows 64-127: Q K^T
        const int L = warp * 32 + lane;
        float* dst = L < 64 ? ML + L * MP : MA + (L - 64) * MP;
        for (int j = 0; j < 64; j += 16) {
            float v[16];
            tmem_ld16(tmem_lane_addr(tmem, warp, j), v);
            tmem_wait_ld();
            for (int i = 0; i < 16; ++i) dst[j + i] = v[i];
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tmem_dealloc(tmem, 64);

    // A and L in place
    const size_t mat = ((size_t(b) * H + h) * NT + c) * (64 * 64);
    for (int i = tid; i < 64 * 64; i += kThreads) {
        const int r = i >> 6, s = i & 63;
        float a = 0.f, l = 0.f;
        if (r >= s) {
            float R = 0.f, Rq = 0.f;
            for (int e = 0; e < E; ++e) {
                const float gam = expf(Gs[r * E + e] - Gs[s * E + e]);
                const float ks2 = k2s[s * E + e] * gam;
                R = fmaf(k2s[r * E + e], ks2, R);
                Rq = fmaf(q2s[r * E + e], ks2, Rq);
            }
            a = MA[r * MP + s] * Rq;
            if (r > s) l = bs[r] * ML[r * MP + s] * R;
        }
        MA[r * MP + s] = a;
        ML[r * MP + s] = l;
        p.Aout[mat + i] = a;
    }
    __syncthreads();

    // N = (I + L)^{-1}: diagonal 16 x 16 blocks (warps 0-3, lane = column), then the rest
    if (p.use_delta) {
        if (warp < 4 && lane < 16) {
            const int o = 16 * warp, s = lane;
            float x[16];
#pragma unroll
            for (int r = 0; r < 16; ++r) {
                float acc = (r == s) ? 1.f : 0.f;
#pragma unroll
                for (int j = 0; j < r; ++j) acc = fmaf(-ML[(o + r) * MP + o + j], x[j], acc);
                x[r] = acc;
            }
#pragma unroll
            for (int r = 0; r < 16; ++r) MX[(o + r) * MP + o + s] = x[r];
        }
        // zero the strictly upper blocks
        for (int i = tid; i < 64 * 64; i += kThreads) {
            const int r = i >> 6, s = i & 63;
            if ((s >> 4) > (r >> 4)) MX[r * MP + s] = 0.f;
        }
        __syncthreads();
        for (int dist = 1; dist < 4; ++dist) {
            const int nblk = 4 - dist;   // blocks (i, i - dist), i = dist..3
            // W_ij = sum_{k=j}^{i-1} L_ik X_kj
            for (int idx = tid; idx < nblk * 256; idx += kThreads) {
                const int bi = dist + idx / 256, bj = bi - dist, e2 = idx & 255;
                const int r = 16 * bi + (e2 >> 4), s = 16 * bj + (e2 & 15);
                float acc = 0.f;
                for (int x = 16 * bj; x < 16 * bi; ++x) acc = fmaf(ML[r * MP + x], MX[x * MP + s], acc);
                MW[r * MP + s] = acc;
            }
            __syncthreads();
            // X_ij = -X_ii W_ij
            for (int idx = tid; idx < nblk * 256; idx += kThreads) {
                const int bi = dist + idx / 256, bj = bi - dist, e2 = idx & 255;
                const int r = 16 * bi + (e2 >> 4), s = 16 * bj + (e2 & 15);
                float acc = 0.f;
                for (int x = 16 * bi; x <= r; ++x) acc = fmaf(MX[r * MP + x], MW[x * MP + s], acc);
                MX[r * MP + s] = -acc;
            }
            __syncthreads();
        }
        for (int i = tid; i < 64 * 64; i += kThreads) p.Nout[mat + i] = MX[(i >> 6) * MP + (i & 63)];
    } else {
        for (int i = tid; i < 64 * 64; i += kThreads) MX[(i >> 6) * MP + (i & 63)] = ((i >> 6) == (i & 63)) ? 1.f : 0.f;
        __syncthreads();
    }
    // T = N diag(beta) into MW; then A T, and the bf16 pairs
    for (int i = tid; i < 64 * 64; i += kThreads) {
        const int r = i >> 6, s = i & 63;
        MW[r * MP + s] = (r >= s) ? MX[r * MP + s] * bs[s] : 0.f;
    }
    __syncthreads();
    const size_t m2 = ((size_t(b) * H + h) * NT + c) * (4 * 64 * 64);
    for (int i = tid; i < 64 * 64; i += kThreads) {
        const int r = i >> 6, s = i & 63;
        float at = 0.f;
        for (int j = s; j <= r; ++j) at = fmaf(MA[r * MP + j], MW[j * MP + s], at);
        const float t = MW[r * MP + s];
        put_pair(p.A2out + m2 + i, p.A2out + m2 + 2 * 4096 + i, t);
        put_pair(p.A2out + m2 + 4096 + i, p.A2out + m2 + 3 * 4096 + i, at);
        if (p.BTout) {   // element (r, s) of A^T and T^T
            put_pair(p.BTout + m2 + i, p.BTout + m2 + 4096 + i, MA[s * MP + r]);
            put_pair(p.BTout + m2 + 2 * 4096 + i, p.BTout + m2 + 3 * 4096 + i, MW[s * MP + r]);
        }
    }
    // coefficient block
    float* cf = p.coef + ((size_t(b) * H + h) * NT + c) * (3 * 64 * E + 16);
    for (int i = tid; i < 64 * E; i += kThreads) {
        const int e = i - (i / E) * E;
        const float Gr = Gs[i], GC = Gs[(n - 1) * E + e];
        const float gam = expf(Gr);
        cf[i] = k2s[i] * gam;
        cf[64 * E + i] = q2s[i] * gam;
        cf[128 * E + i] = k2s[i] * expf(GC - Gr);
    }
    if (tid < 16) cf[192 * E + tid] = tid < E ? expf(Gs[(n - 1) * E + tid]) : 0.f;
}

size_t prep_tc_smem(int E) { return 1024 + 4 * kBoxBytes + 4 * 64 * MP * 4 + (3 * 64 * E + 64) * 4; }

}  // namespace

cudaError_t launch_chunk_prep_tc(const tla_problem& p, const FwdPlan& fp, char* ws, int* err,
                                 cudaStream_t s) {
    CUtensorMap mk, mq;
    if (!make_token_map(&mk, p.k, p.B, p.T, p.H, kDk, 64, 64, true) ||
        !make_token_map(&mq, p.q, p.B, p.T, p.H, kDk, 64, 64, true))
        return cudaErrorInvalidValue;
    TcPrepArgs a;
    a.q2 = (const __nv_bfloat16*)p.q2;
    a.k2 = (const __nv_bfloat16*)p.k2;
    a.G = (const float*)(ws + fp.G);
    a.beta = p.beta;
    a.Aout = (float*)(ws + fp.A);
    a.Nout = p.use_delta ? (float*)(ws + fp.N) : nullptr;
    a.A2out = (__nv_bfloat16*)(ws + fp.A2);
    a.BTout = fp.tcb ? (__nv_bfloat16*)(ws + fp.BT) : nullptr;
    a.coef = (float*)(ws + fp.coef);
    a.err = err;
    a.T = p.T; a.H = p.H; a.E = p.E; a.NT = fp.NT; a.use_delta = p.use_delta;
    const size_t smem = prep_tc_smem(p.E);
    cudaFuncSetAttribute(chunk_prep_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    dim3 grid(fp.NT, p.H, p.B);
    prof_before("chunk_prep_tc", s);
    chunk_prep_tc_kernel<<<grid, kThreads, smem, s>>>(mk, mq, a);
    prof_after(s);
    return cudaGetLastError();
}

}  // namespace tla
