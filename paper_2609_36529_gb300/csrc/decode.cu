// Single-token decode step (Algorithm 2, one iteration), HBM-bound.
//
// Per (b, h) and block of 16 value columns one CTA reads its E x dk x 16 slab of the
// fp32 state once from HBM and writes the updated slab back once:
//   Shat_e = alpha_e S_e                                   (Eq. forget3)
//   r      = sum_e k'_e Shat_e^T k,  u = beta (v - r)      (Eq. gdn3; sGLA: u = beta v)
//   S_e    = Shat_e + k'_e k u^T                           (triadic write)
//   o      = sum_e q'_e S_e^T q = p + (q'.k')(q.k) u,  p = sum_e q'_e Shat_e^T q
// The last identity lets o come from the same single read of the slab.
// Reductions over (e, d) use warp shuffles then a fixed-order pass over warps,
// so results are deterministic.
//
// decode_smem_kernel (slabs of at most 1024 rows of 16 columns, the usual case): the slab
// arrives by one TMA tensor load into shared memory, is updated there in place and leaves
// by one TMA tensor store.  It needs few registers, so three CTAs -- three slabs in flight
// -- share an SM; with the slab held in registers (decode_step_kernel, which takes every
// other supported shape) only two fit, and HBM idles while they reduce.
#include <cstring>

#include "common.cuh"
#include "internal.h"
#include "sm100.cuh"
#include "tma_host.h"

namespace tla {

constexpr int kDecThreads = 256;

namespace {

// fp32 recurrent state [B*H*E][dk][dv] viewed as 3-D (dv, dk, B*H*E); box (box_c, dk, box_e):
// the box_e x dk x box_c slab of one (b, h) and block of value columns, unswizzled.
bool make_state_map(CUtensorMap* m, const void* base, long long nslice, int dk, int dv, int box_c,
                    int box_e) {
    auto enc = tensor_map_encoder();
    if (!enc) return false;
    cuuint64_t dims[3] = {(cuuint64_t)dv, (cuuint64_t)dk, (cuuint64_t)nslice};
    cuuint64_t strides[2] = {(cuuint64_t)dv * 4, (cuuint64_t)dk * dv * 4};
    cuuint32_t box[3] = {(cuuint32_t)box_c, (cuuint32_t)dk, (cuuint32_t)box_e};
    cuuint32_t es[3] = {1, 1, 1};
    CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, const_cast<void*>(base), dims, strides,
                     box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

// TMA tensor store shared -> global of the box at (x, y, z) of a 3-d tensor map, in the
// issuing thread's current bulk async-group (x * element size a multiple of 16 bytes).
__device__ __forceinline__ void tma_store_3d(const CUtensorMap* map, const void* src, int x, int y,
                                             int z) {
    asm volatile("cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%1, %2, %3}], [%4];" ::"l"(
                     reinterpret_cast<uint64_t>(map)),
                 "r"(x), "r"(y), "r"(z), "r"(sm100::smem_u32(src))
                 : "memory");
}

}  // namespace

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

// One slab per CTA in shared memory: one TMA tensor load, in-place update, one TMA tensor
// store; few registers, so three CTAs (three slabs in flight) share an SM.  The CTA waits
// only until the store has read its shared memory (the store's global writes complete
// after it exits, before the launch completes).
template <typename Tin>
__global__ void __launch_bounds__(kDecThreads, 3)
decode_smem_kernel(const __grid_constant__ CUtensorMap map_s, const Tin* __restrict__ q,
                   const Tin* __restrict__ k, const Tin* __restrict__ v, const Tin* __restrict__ q2,
                   const Tin* __restrict__ k2, const float* __restrict__ g,
                   const float* __restrict__ beta, Tin* __restrict__ o, int* err, int dk, int dv,
                   int E, int use_delta) {
    using namespace sm100;
    extern __shared__ uint8_t smem_raw[];
    float* S = reinterpret_cast<float*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    constexpr int NW = kDecThreads / 32;
    __shared__ __align__(8) uint64_t full;
    __shared__ float qs[128], ks[128], q2s[32], k2s[32], al[32];
    __shared__ float4 red_r[NW][4], red_p[NW][4];
    __shared__ __align__(16) float us[16];
    __shared__ float dots[2];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int quad = tid & 3, row0 = tid >> 2;
    const int nb = blockIdx.x, bh = blockIdx.y, n0 = nb * 16;
    const int rows = E * dk, passes = rows / 64;
    if (tid == 0) {
        mbar_init(&full, 1);
        fence_barrier_init();
        mbar_arrive_expect_tx(&full, uint32_t(rows) * 64);
        tma_load_3d(S, &map_s, &full, n0, 0, bh * E);
    }
    if (tid < dk) {
        qs[tid] = to_f(q[size_t(bh) * dk + tid]);
        ks[tid] = to_f(k[size_t(bh) * dk + tid]);
    } else if (tid >= 128 && tid < 128 + E) {
        const int e = tid - 128;
        q2s[e] = to_f(q2[size_t(bh) * E + e]);
        k2s[e] = to_f(k2[size_t(bh) * E + e]);
        al[e] = expf(g[size_t(bh) * E + e]);
    }
    __syncthreads();
    if (warp == 0) {
        float x = 0.f, y = 0.f;
        for (int i = lane; i < dk; i += 32) x = fmaf(qs[i], ks[i], x);
        if (lane < E) y = q2s[lane] * k2s[lane];
#pragma unroll
        for (int off = 16; off >= 1; off >>= 1) {
            x += __shfl_xor_sync(0xffffffffu, x, off);
            y += __shfl_xor_sync(0xffffffffu, y, off);
        }
        if (lane == 0) { dots[0] = x; dots[1] = y; }
    }
    const bool ok = mbar_wait(&full, 0);
    if (__syncthreads_or(!ok)) {
        if (tid == 0) {
            record_device_error(err, TLA_ERR_TIMEOUT);
            mbar_wait(&full, 0);   // bounded drain of the load
        }
        return;
    }
    float4 pr = make_float4(0.f, 0.f, 0.f, 0.f), pp = pr;
#pragma unroll 4
    for (int pass = 0; pass < passes; ++pass) {
        const int row = row0 + pass * 64, e = row / dk, d = row - e * dk;
        float4 sv = reinterpret_cast<const float4*>(S)[row * 4 + quad];
        const float a = al[e];
        sv.x *= a; sv.y *= a; sv.z *= a; sv.w *= a;
        const float ck = k2s[e] * ks[d], cq = q2s[e] * qs[d];
        pr.x = fmaf(ck, sv.x, pr.x); pr.y = fmaf(ck, sv.y, pr.y);
        pr.z = fmaf(ck, sv.z, pr.z); pr.w = fmaf(ck, sv.w, pr.w);
        pp.x = fmaf(cq, sv.x, pp.x); pp.y = fmaf(cq, sv.y, pp.y);
        pp.z = fmaf(cq, sv.z, pp.z); pp.w = fmaf(cq, sv.w, pp.w);
    }
#pragma unroll
    for (int off = 4; off < 32; off <<= 1) {
        pr.x += __shfl_xor_sync(0xffffffffu, pr.x, off);
        pr.y += __shfl_xor_sync(0xffffffffu, pr.y, off);
        pr.z += __shfl_xor_sync(0xffffffffu, pr.z, off);
        pr.w += __shfl_xor_sync(0xffffffffu, pr.w, off);
        pp.x += __shfl_xor_sync(0xffffffffu, pp.x, off);
        pp.y += __shfl_xor_sync(0xffffffffu, pp.y, off);
        pp.z += __shfl_xor_sync(0xffffffffu, pp.z, off);
        pp.w += __shfl_xor_sync(0xffffffffu, pp.w, off);
    }
    if (lane < 4) {
        red_r[warp][lane] = pr;
        red_p[warp][lane] = pp;
    }
    __syncthreads();
    if (tid < 16) {
        const int qd = tid >> 2, comp = tid & 3;
        float r = 0.f, pq = 0.f;
        for (int w = 0; w < NW; ++w) {
            r += reinterpret_cast<const float*>(&red_r[w][qd])[comp];
            pq += reinterpret_cast<const float*>(&red_p[w][qd])[comp];
        }
        const float vv = to_f(v[size_t(bh) * dv + n0 + tid]);
        const float bt = beta ? beta[bh] : 1.f;
        const float u = use_delta ? bt * (vv - r) : bt * vv;
        us[tid] = u;
        o[size_t(bh) * dv + n0 + tid] = from_f<Tin>(fmaf(dots[1] * dots[0], u, pq));
    }
    __syncthreads();
    const float4 u4 = reinterpret_cast<const float4*>(us)[quad];
#pragma unroll 4
    for (int pass = 0; pass < passes; ++pass) {
        const int row = row0 + pass * 64, e = row / dk, d = row - e * dk;
        float4* p4 = reinterpret_cast<float4*>(S) + row * 4 + quad;
        float4 sv = *p4;
        const float a = al[e], c = k2s[e] * ks[d];
        sv.x = fmaf(a, sv.x, c * u4.x); sv.y = fmaf(a, sv.y, c * u4.y);
        sv.z = fmaf(a, sv.z, c * u4.z); sv.w = fmaf(a, sv.w, c * u4.w);
        *p4 = sv;
    }
    fence_proxy_async_smem();
    __syncthreads();
    if (tid == 0) {
        tma_store_3d(&map_s, S, n0, 0, bh * E);
        bulk_commit();
        bulk_wait_read_all();   // the CTA's shared memory must outlive the store's read
    }
}

cudaError_t launch_decode_step(int B, int H, int dk, int dv, int E, int use_delta, int dtype,
                               const void* q, const void* k, const void* v, const void* q2,
                               const void* k2, const float* g, const float* beta,
                               float* state, void* o, int* err, cudaStream_t s) {
    if (dv % 16 == 0 && dk <= 128 && E <= 32 && (E * dk) % 64 == 0 && E * dk <= 1024) {
        CUtensorMap map;
        memset(&map, 0, sizeof(map));
        if (!make_state_map(&map, state, (long long)B * H * E, dk, dv, 16, E)) return cudaErrorInvalidValue;
        const size_t smem = 1024 + size_t(E) * dk * 64;
        dim3 grid(dv / 16, B * H);
        prof_before("decode_step", s);
        if (dtype == TLA_BF16) {
            using Tb = __nv_bfloat16;
            auto kern = decode_smem_kernel<Tb>;
            cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            kern<<<grid, kDecThreads, smem, s>>>(map, (const Tb*)q, (const Tb*)k, (const Tb*)v,
                                                 (const Tb*)q2, (const Tb*)k2, g, beta, (Tb*)o, err,
                                                 dk, dv, E, use_delta);
        } else {
            auto kern = decode_smem_kernel<float>;
            cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            kern<<<grid, kDecThreads, smem, s>>>(map, (const float*)q, (const float*)k, (const float*)v,
                                                 (const float*)q2, (const float*)k2, g, beta, (float*)o,
                                                 err, dk, dv, E, use_delta);
        }
        prof_after(s);
        return cudaGetLastError();
    }
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
