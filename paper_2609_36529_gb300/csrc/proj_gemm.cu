// Input projection of the layer (Appendix A, Input projections; Algorithm 2): one GEMM
// produces the q, k, v, q', k' channels of every head,
//   P[t, h, c] = sum_i u[t, i] W[h C + c, i]      (C = 2 dk + dv + 2 E, channels [q|k|v|q'|k'])
// on tcgen05 tensor cores, and its epilogue runs the rest of the input path on the
// accumulator tile, so P need not make a round trip through HBM:
//   causal depthwise convolution of width K (tokens before the sequence start are zero),
//   SiLU on q, k, v and softplus on q', k', L2 normalisation of q, k, q', k'
//   (x / sqrt(|x|^2 + eps)), and for each token the log gates
//   -exp(A_log) softplus(gate_in + gate_bias) and beta = sigmoid(beta_in).
// Optionally P itself is written (bf16), for the backward of the input path.
//
// Tiling.  One CTA per (sequence, block of 125 tokens, head, channel group): the M = 128
// accumulator rows are tokens t0 - 3 .. t0 + 124, so the three rows before the block give
// the convolution window of its first tokens (2.3 % of the products recomputed).  Channel
// group 0 is [q | k] (N = 2 dk), group 1 is [v | q' | k'] (N = dv + 2 E rounded up to 16;
// the rows past the head's channels are computed and discarded).  The K dimension (model
// width) streams through a two-stage TMA pipeline of 64-wide bf16 blocks in the 128-byte
// swizzled K-major layout both operands use.  Warp 0 issues the copies, warp 1 the UMMAs
// (fp32 accumulation in TMEM), warps 2-5 run the epilogue: the tile goes from TMEM to
// shared memory (one thread per token row, fp32, odd row stride), the convolution and
// activation run one thread per channel down the tokens (a sliding window of raw values in
// registers), and the normalisation and the bf16 stores run one thread per token again.
// Every mbarrier wait is bounded; on expiry the CTA records TLA_ERR_TIMEOUT and leaves.
#include <cuda_bf16.h>

#include "act.cuh"
#include "common.cuh"
#include "internal.h"
#include "sm100.cuh"
#include "tma_host.h"

namespace tla {

int* device_error_word();

namespace {
using namespace sm100;

constexpr int kThreads = 192;       // warp 0 TMA, warp 1 MMA, warps 2-5 epilogue
constexpr int kRowsOut = 125;       // tokens written per CTA (M = 128 minus the 3-row halo)
constexpr int kHalo = 3;
constexpr int kStages = 2;
constexpr uint32_t kABytes = 128 * 128;       // A block: 128 rows x 64 bf16
constexpr uint32_t kBMax = 256 * 128;         // B block: up to 256 rows x 64 bf16
constexpr uint32_t kStageBytes = kABytes + kBMax;

struct ProjArgs {
    const float* conv_w;      // [H, C, K]
    const float* gate_in;     // [B, T, H, E]
    const float* gate_bias;   // [H, E]
    const float* A_log;       // [H, E]
    const float* beta_in;     // [B, T, H] or NULL
    __nv_bfloat16 *q, *k, *v, *q2, *k2;
    float* g;
    float* beta;
    __nv_bfloat16* P;         // [B, T, H, C] or NULL
    int* err;
    int B, T, H, dk, dv, E, K, Dm, n1;   // n1: UMMA N of channel group 1
    float eps;
};

__device__ __forceinline__ void epi_sync() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

__device__ __forceinline__ float silu(float x) { return x * sigm(x); }

// n values of a row, L2-normalised (x / sqrt(|x|^2 + eps)) when norm, as bf16 (16-byte stores
// when n is a multiple of 8).
__device__ __forceinline__ void put_row(__nv_bfloat16* dst, const float* src, int n, bool norm, float eps) {
    float r = 1.f;
    if (norm) {   // four partial sums: four loads and FMA chains in flight
        float s4[4] = {0.f, 0.f, 0.f, 0.f};
        int i = 0;
#pragma unroll 4
        for (; i + 4 <= n; i += 4)
#pragma unroll
            for (int u = 0; u < 4; ++u) s4[u] = fmaf(src[i + u], src[i + u], s4[u]);
        for (; i < n; ++i) s4[0] = fmaf(src[i], src[i], s4[0]);
        r = rsqrtf((s4[0] + s4[1]) + (s4[2] + s4[3]) + eps);
    }
    if (n % 8 == 0) {
#pragma unroll 4
        for (int i = 0; i < n; i += 8) {
            uint32_t w4[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const __nv_bfloat162 pr = __floats2bfloat162_rn(src[i + 2 * u] * r, src[i + 2 * u + 1] * r);
                w4[u] = *reinterpret_cast<const uint32_t*>(&pr);
            }
            *reinterpret_cast<uint4*>(dst + i) = make_uint4(w4[0], w4[1], w4[2], w4[3]);
        }
    } else {
        for (int i = 0; i < n; ++i) dst[i] = __float2bfloat16_rn(src[i] * r);
    }
}

__global__ void __launch_bounds__(kThreads, 2)
proj_gemm_kernel(const __grid_constant__ CUtensorMap map_u, const __grid_constant__ CUtensorMap map_w0,
                 const __grid_constant__ CUtensorMap map_w1, const ProjArgs p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
    __shared__ __align__(8) uint64_t full[kStages], empty[kStages], acc_full;
    __shared__ uint32_t tmem_slot;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int grp = blockIdx.x & 1, h = blockIdx.x >> 1;
    const int t0 = blockIdx.y * kRowsOut, b = blockIdx.z;
    const int dk = p.dk, dv = p.dv, E = p.E, K = p.K, T = p.T, H = p.H;
    const int C = 2 * dk + dv + 2 * E;
    const int N = grp == 0 ? 2 * dk : p.n1;
    const int nkb = p.Dm / 64;
    const uint32_t bbytes = uint32_t(N) * 128;

    if (warp == 1) {
        tmem_alloc(&tmem_slot, 256);
        tmem_relinquish();
    }
    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_init(&acc_full, 1);
        fence_barrier_init();
        tma_prefetch_desc(&map_u);
        tma_prefetch_desc(grp == 0 ? &map_w0 : &map_w1);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;

    if (warp == 0) {
        // ---- producer: A = 128 token rows from t0 - 3 (rows before the batch read as zero),
        // B = this group's weight rows
        if (lane == 0) {
            const int arow = b * T + t0 - kHalo;
            const int wrow = h * C + (grp == 0 ? 0 : 2 * dk);
            const CUtensorMap* mw = grp == 0 ? &map_w0 : &map_w1;
            for (int kb = 0; kb < nkb; ++kb) {
                const int s = kb % kStages;
                if (kb >= kStages && !mbar_wait(&empty[s], ((kb / kStages) - 1) & 1)) {
                    record_device_error(p.err, TLA_ERR_TIMEOUT);
                    break;
                }
                uint8_t* st = sm + s * kStageBytes;
                mbar_arrive_expect_tx(&full[s], kABytes + bbytes);
                tma_load_2d(st, &map_u, &full[s], kb * 64, arow);
                tma_load_2d(st + kABytes, mw, &full[s], kb * 64, wrow);
            }
        }
    } else if (warp == 1) {
        // ---- MMA issuer: D[128 x N] += A_kb B_kb^T over the K blocks
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16_f32(128, N, 0, 0);
            bool ok = true;
            for (int kb = 0; kb < nkb && ok; ++kb) {
                const int s = kb % kStages;
                ok = mbar_wait(&full[s], (kb / kStages) & 1);
                if (!ok) break;
                tc_fence_after();
                const uint32_t a0 = smem_u32(sm + s * kStageBytes), b0 = a0 + kABytes;
#pragma unroll
                for (int k = 0; k < 4; ++k)
                    umma_bf16(tmem, smem_desc(a0 + k * 32, 16, 1024), smem_desc(b0 + k * 32, 16, 1024), idesc,
                              (kb | k) ? 1u : 0u);
                umma_commit(&empty[s]);
            }
            if (!ok) record_device_error(p.err, TLA_ERR_TIMEOUT);
            umma_commit(&acc_full);   // arrives once every issued product has completed
        }
    } else {
        // ---- epilogue (warps 2-5): TMEM lane quadrant warp % 4 holds rows 32 (warp % 4) ..
        const int et = tid - 64;                       // 0..127
        const int row = 32 * (warp & 3) + lane;        // accumulator row of this thread
        const int trow = t0 - kHalo + row;             // its token
        const bool out_row = row >= kHalo && trow < T && row < kHalo + kRowsOut;
        const bool ok = mbar_wait(&acc_full, 0);
        tc_fence_after();
        if (!ok) {
            if (et == 0) record_device_error(p.err, TLA_ERR_TIMEOUT);
        } else {
            float* S = reinterpret_cast<float*>(sm);   // [128][ld] fp32 (the stage buffers are idle)
            const size_t tok = (size_t(b) * T + (trow < 0 ? 0 : trow)) * H + h;   // (b, t, h) index
            // group 0 in two passes (q, then k), group 1 in one ([v | q' | k'])
            const int npass = grp == 0 ? 2 : 1;
            for (int pass = 0; pass < npass; ++pass) {
                const int tc0 = pass * dk;                         // first TMEM column of the pass
                const int nc = grp == 0 ? dk : dv + 2 * E;         // channels of the pass
                const int c0 = (grp == 0 ? 0 : 2 * dk) + tc0;     // their first channel in the head
                const int ld = nc + 1;                             // odd stride: no bank conflicts
                // TMEM -> shared memory (and the raw projection, when requested), 32 columns
                // per wait (the accumulator's 256 columns cover the second load)
                for (int j = 0; j < nc; j += 32) {
                    float v[32];
                    tmem_ld16(tmem_lane_addr(tmem, warp, tc0 + j), v);
                    tmem_ld16(tmem_lane_addr(tmem, warp, tc0 + j + 16), v + 16);
                    tmem_wait_ld();
                    const int cnt = nc - j < 32 ? nc - j : 32;
#pragma unroll
                    for (int u = 0; u < 32; ++u)
                        if (u < cnt) S[row * ld + j + u] = v[u];
                    if (p.P && out_row)
#pragma unroll
                        for (int u = 0; u < 32; ++u)
                            if (u < cnt) p.P[tok * C + c0 + j + u] = __float2bfloat16_rn(v[u]);
                }
                epi_sync();
                // causal depthwise convolution and activation, one thread per channel down the rows
                for (int c = et; c < nc; c += 128) {
                    const int cg = c0 + c;                 // channel within the head
                    const bool soft = cg >= 2 * dk + dv;   // q', k': softplus; q, k, v: SiLU
                    float w[4];   // taps padded on the left to four
#pragma unroll
                    for (int j = 0; j < 4; ++j)
                        w[j] = j >= 4 - K ? p.conv_w[(size_t(h) * C + cg) * K + j - (4 - K)] : 0.f;
                    float* col = S + c;
                    // eight rows at a time: their raw values are read before any of them is
                    // overwritten, so the eight loads are in flight together; the activation is
                    // chosen once per channel, outside the loop, so that the eight rows'
                    // activations interleave
                    auto conv_rows = [&](auto act) {
                        float x0 = 0.f, x1 = 0.f, x2 = 0.f;   // raw values of the three previous rows
                        for (int r0 = 0; r0 < 128; r0 += 8) {
                            float xr[8], y[8];
#pragma unroll
                            for (int i = 0; i < 8; ++i) xr[i] = t0 - kHalo + r0 + i >= 0 ? col[(r0 + i) * ld] : 0.f;
#pragma unroll
                            for (int i = 0; i < 8; ++i) {
                                const float a = fmaf(w[0], x0, fmaf(w[1], x1, fmaf(w[2], x2, w[3] * xr[i])));
                                y[i] = act(a);
                                x0 = x1; x1 = x2; x2 = xr[i];
                            }
#pragma unroll
                            for (int i = 0; i < 8; ++i)
                                if (r0 + i >= kHalo) col[(r0 + i) * ld] = y[i];
                        }
                    };
                    if (soft) conv_rows([](float a) { return softplus(a); });
                    else conv_rows([](float a) { return silu(a); });
                }
                epi_sync();
                // normalisation and stores, one thread per token row
                if (out_row) {
                    const float* y = S + row * ld;
                    if (grp == 0) {
                        put_row(pass == 0 ? p.q + tok * dk : p.k + tok * dk, y, dk, true, p.eps);
                    } else {
                        put_row(p.v + tok * dv, y, dv, false, p.eps);
                        put_row(p.q2 + tok * E, y + dv, E, true, p.eps);
                        put_row(p.k2 + tok * E, y + dv + E, E, true, p.eps);
                        // log forget gates and beta of this token (no convolution)
                        for (int e = 0; e < E; ++e) {
                            const float x = p.gate_in[tok * E + e] + p.gate_bias[h * E + e];
                            p.g[tok * E + e] = -__expf(p.A_log[h * E + e]) * softplus(x);
                        }
                        if (p.beta_in) p.beta[tok] = sigm(p.beta_in[tok]);
                    }
                }
                epi_sync();   // the next pass rewrites the buffer
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tmem, 256);
}

}  // namespace

}  // namespace tla

using namespace tla;

static tla_status check_projection(const tla_projection_args* a) {
    if (!a) return TLA_ERR_INVALID_ARG;
    if (a->B < 1 || a->T < 1 || a->H < 1 || a->E < 1 || a->Dm < 64) return TLA_ERR_INVALID_ARG;
    if (a->K < 1 || a->K > 4 || !(a->eps > 0.f)) return TLA_ERR_INVALID_ARG;
    if (!a->u || !a->W || !a->conv_w || !a->gate_in || !a->gate_bias || !a->A_log || !a->q ||
        !a->k || !a->v || !a->q2 || !a->k2 || !a->g)
        return TLA_ERR_INVALID_ARG;
    if ((a->beta_in != nullptr) != (a->beta != nullptr)) return TLA_ERR_INVALID_ARG;
    if ((a->dk != 64 && a->dk != 128) || (a->dv != 64 && a->dv != 128)) return TLA_ERR_UNSUPPORTED;
    if (a->E > 16 || a->Dm % 64 != 0) return TLA_ERR_UNSUPPORTED;
    if ((long long)a->H * 2 > 65535 || a->B > 65535) return TLA_ERR_UNSUPPORTED;
    const void* ptrs[] = {a->u, a->W, a->conv_w, a->gate_in, a->gate_bias, a->A_log, a->beta_in,
                          a->q, a->k, a->v, a->q2, a->k2, a->g, a->beta, a->P};
    for (const void* x : ptrs)
        if (((uintptr_t)x & 15) != 0) return TLA_ERR_INVALID_ARG;
    return TLA_OK;
}

extern "C" tla_status tla_layer_projection(const tla_projection_args* a, void* stream) {
    const tla_status st0 = check_projection(a);
    if (st0 != TLA_OK) return st0;
    const int C = 2 * a->dk + a->dv + 2 * a->E;
    const int n1 = ((a->dv + 2 * a->E) + 15) / 16 * 16;
    CUtensorMap mu, mw0, mw1;
    if (!make_matrix_map(&mu, a->u, (long long)a->B * a->T, a->Dm, 64, 128) ||
        !make_matrix_map(&mw0, a->W, (long long)a->H * C, a->Dm, 64, 2 * a->dk) ||
        !make_matrix_map(&mw1, a->W, (long long)a->H * C, a->Dm, 64, n1))
        return TLA_ERR_CUDA;
    int* err = device_error_word();
    if (!err) return TLA_ERR_CUDA;
    ProjArgs p;
    p.conv_w = a->conv_w; p.gate_in = a->gate_in; p.gate_bias = a->gate_bias; p.A_log = a->A_log;
    p.beta_in = a->beta_in;
    p.q = (__nv_bfloat16*)a->q; p.k = (__nv_bfloat16*)a->k; p.v = (__nv_bfloat16*)a->v;
    p.q2 = (__nv_bfloat16*)a->q2; p.k2 = (__nv_bfloat16*)a->k2;
    p.g = a->g; p.beta = a->beta; p.P = (__nv_bfloat16*)a->P; p.err = err;
    p.B = a->B; p.T = a->T; p.H = a->H; p.dk = a->dk; p.dv = a->dv; p.E = a->E; p.K = a->K;
    p.Dm = a->Dm; p.n1 = n1; p.eps = a->eps;
    const size_t smem = 1024 + size_t(kStages) * kStageBytes;
    cudaStream_t s = (cudaStream_t)stream;
    cudaFuncSetAttribute(proj_gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    dim3 grid(2 * a->H, (a->T + kRowsOut - 1) / kRowsOut, a->B);
    prof_before("proj_gemm", s);
    proj_gemm_kernel<<<grid, kThreads, smem, s>>>(mu, mw0, mw1, p);
    prof_after(s);
    return cudaGetLastError() == cudaSuccess ? TLA_OK : TLA_ERR_CUDA;
}
