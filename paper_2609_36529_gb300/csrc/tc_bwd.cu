// Tensor-core (tcgen05) backward recurrence over chunks (Appendix A, Kernels: a
// reverse pass over the chunks yields the gradient of every state slice at
// each chunk boundary; the remaining gradients follow chunk-parallel).
//
// Differentiating the chunk step of Eq. joint-chunk (see tc_fwd.cu) gives, per
// chunk c walked backwards, with dS' the gradient of the state at the chunk's end:
//   dU   = A^T dO + sum_e diag(w_e) K dS'_e
//   dRes = T^T dU                                   (= dV)
//   dS_e = gamma^C_e dS'_e + Q^T diag(b_e) dO - K^T diag(a_e) dRes
// One CTA of 8 warps per (b, h, block of TV value columns) keeps dS for its
// value columns in TMEM.  Per chunk:
//   MMA-A'  P' = K dS'_all              (M=64, N=NE, K=dk; dS' MN-major hi/lo, the two halves
//                                        side by side, N = 2 NE, when that fits one instruction;
//                                        at E = 16 in two halves of the slices, one after the
//                                        other, so that P', Y and the slab fit 512 columns)
//   MMA-0   Y  = A^T dO                 (M=64, N=TV, K=64; A^T hi/lo read MN-major from the
//                                        row-major A tiles, dO exact bf16, MN-major as the
//                                        TMA loads it)
//   epi     dU = Y + sum_e w_e (.) P'_e  -> dU hi/lo operand, dU to the workspace
//   MMA-B'  dRes = T^T dU               (M=64, K=64; both hi/lo, the hi*hi and hi*lo terms in
//                                        one N = 2 TV product)
//   epi     dRes -> workspace and dv; operand rows [-a_e (.) dRes ; b_e (.) dO]
//   MMA-C'  dS_all += [K^T | Q^T] [-a (.) dRes ; b (.) dO]   (M=dk=128, K=128, N=NE;
//           K^T and Q^T read MN-major from the TMA key/query tile)
//   epi     dS_{[c]} from TMEM -> operand of the previous chunk and checkpoint; once the
//           previous chunk's MMA-A' is issued, the slab is rescaled in place by its gamma^C.
// Layout of the M=64 products in TMEM: row r sits on lane 32 * (r / 16) + r % 16,
// so lanes 0-15 of each warp own the row work and lanes 16-31 the dO rows.
// Warps 0-3 / 4-7 take the first / second half of each slice's TV value columns.  E is a
// compile-time parameter (per-slice loops unroll; each thread keeps its row's coefficients,
// read from the slice-major coefficient block, in registers).
// Precision, TMA prefetch, bounded waits, the slice-block layout of the state
// operand and the TMA-stored checkpoints as in the forward kernel.
#include <cstring>
#include <type_traits>

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

struct TcBwdArgs {
    const float* coef;   // forward workspace coefficient blocks [B,H,NT, 3*64*E+16]
    const float* dht;
    void* dv_out;
    float* dh0;
    float* dUbuf;
    float* dRbuf;
    float* dSck;
    int* err;
    const int4* dtab;    // packed documents: (first token, chunks, first chunk, tokens); else NULL
    int T, H, dv, E, NT, use_delta, out_f32, ck_tiles;
    int dk;              // key dimension: 128, or 64 padded to 128 by zero rows (TMA fill)
};

template <int TV>
__host__ __device__ constexpr size_t tc_bwd_smem_c(int E) {
    return 1024 + 8 * kBoxBytes + size_t(E) * TV * 512 + 64 * TV * 2 + 64 * TV * 4 +
           2 * (3 * 64 * E + 16) * 4;
}
// CTAs per SM the launch bounds plan for: two (at most 128 registers a thread) when two fit
// in shared memory, else one.
template <int TV, int E>
__host__ __device__ constexpr int bwd_min_blocks() {
    return tc_bwd_smem_c<TV>(E) <= 113 * 1024 ? 2 : 1;
}

template <int TV, int E>
__global__ void __launch_bounds__(kThreads, (bwd_min_blocks<TV, E>()))
bwd_recurrence_tc_kernel(const __grid_constant__ CUtensorMap map_k,
                         const __grid_constant__ CUtensorMap map_q,
                         const __grid_constant__ CUtensorMap map_do,
                         const __grid_constant__ CUtensorMap map_bt,
                         const __grid_constant__ CUtensorMap map_ck,
                         const __grid_constant__ CUtensorMap map_dv, const TcBwdArgs p) {
    constexpr int TVH = TV / 2;                      // value columns per thread
    constexpr int GRP0 = TVH >= 32 ? 1 : 32 / TVH;
    constexpr int GRP = GRP0 < E ? GRP0 : E;         // slices per batch of TMEM loads
    static_assert(E % GRP == 0, "slices per batch must divide E");
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
    constexpr int NE = E * TV;
    constexpr int CB = 3 * 64 * E + 16;
    uint8_t* sKQ = sm;                       // 2 blocks x [K rows | Q rows] x 128 B
    uint8_t* sBT = sKQ + 4 * kBoxBytes;      // A hi, A lo, T hi, T lo (64 x 64 each, row-major:
                                             // the MN-major A operands A^T and T^T)
    uint8_t* sReg = sBT + 4 * kBoxBytes;     // NE * 512 bytes, reused:
    uint8_t* sDh = sReg;                     //   dS' hi / lo: E blocks [dk][TV] (MMA-A',
    uint8_t* sDl = sReg + NE * 256;          //   checkpoint source)
    uint8_t* sBh = sReg;                     //   [-a dRes ; b dO] [128][NE] hi / lo (MMA-C')
    uint8_t* sBl = sReg + NE * 256;
    uint8_t* sdO = sReg + NE * 512;          // dO [64][TV] bf16, MN-major operand (TMA, swizzled)
    uint8_t* sDvo = sdO + 64 * TV * 2;       // dv tile [64][TV] (TMA store)
    uint8_t* sUh = sDvo;                     // dU [64][TV] hi / lo, MN-major (MMA-B'), in the dv
    uint8_t* sUl = sDvo + TV * 128;          // tile's space: the checkpoint copy of dS' proceeds
                                             // under the dU epilogue and MMA-B' 
    float* sCoef = reinterpret_cast<float*>(sDvo + 64 * TV * 4);   // 2 x CB

    __shared__ __align__(8) uint64_t bar_kq, bar_av, bar_mma;
    __shared__ uint32_t tmem_slot;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int r = tid & 127;                 // TMEM lane of the dS slab: row d
    const int cofs = (tid >> 7) * TVH;       // this thread's first column within a slice
    const int nb = blockIdx.x, h = blockIdx.y, sb = blockIdx.z;   // sb: sequence or document
    const int n0 = nb * TV;
    const int T = p.T, H = p.H, dv = p.dv, NT = p.NT;
    // hi and lo halves of dS' side by side in one N = 2 NE product K dS' (half the UMMAs on
    // the chain) when N fits one instruction; dRes takes 2 TV columns (hi*hi + lo*hi, hi*lo)
    constexpr bool kSide = 2 * NE <= 256;
    // P' by halves of the slices (the second product issued once the first is consumed) when
    // all of it, Y and the slab do not fit the 512 TMEM columns together
    constexpr bool kSplitP = !kSide && 2 * NE + 2 * TV > 512;
    constexpr int EP = kSplitP ? E / 2 : E;    // slices per P' product
    static_assert(!kSplitP || (E % 2 == 0 && (E / 2) % GRP == 0), "P' halves: whole batches");
    constexpr int kPc = kSide ? 2 * NE : EP * TV;   // TMEM columns of P'
    static_assert(kPc + 2 * TV + NE <= 512, "TMEM map");
    constexpr uint32_t tcols = (kPc + 2 * TV + NE <= 256) ? 256u : 512u;
    constexpr uint64_t kSwz = swizzle_code(2 * TV);
    // token batch, first token, tokens, chunks and first chunk (in the workspaces) of this state
    int b = sb, tbeg = 0, tlen = T, nct = NT, cb = 0;
    if (p.dtab) {
        const int4 dd = p.dtab[sb];
        b = 0; tbeg = dd.x; nct = dd.y; cb = dd.z; tlen = dd.w;
    }
    if (nct == 0) {   // empty document: the gradient of the initial state is that of the final one
        if (p.dh0 && r < p.dk)
            for (int e = 0; e < E; ++e)
                for (int n = cofs; n < cofs + TVH; ++n) {
                    const size_t o = ((size_t(sb * H + h) * E + e) * p.dk + r) * dv + n0 + n;
                    p.dh0[o] = p.dht ? p.dht[o] : 0.f;
                }
        return;
    }
    // M=64 row owned by this thread (lanes 0-15) or whose dO part it prepares (lanes 16-31)
    const bool row_thread = lane < 16;
    const int r64 = 16 * (warp & 3) + (lane & 15);

    if (warp == 0) {
        tmem_alloc(&tmem_slot, tcols);
        tmem_relinquish();
    }
    if (tid == 0) {
        mbar_init(&bar_kq, 1);
        mbar_init(&bar_av, 1);
        mbar_init(&bar_mma, 1);
        fence_barrier_init();
        tma_prefetch_desc(&map_k);
        tma_prefetch_desc(&map_q);
        tma_prefetch_desc(&map_do);
        tma_prefetch_desc(&map_bt);
        if (p.ck_tiles) tma_prefetch_desc(&map_ck);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tP = tmem_slot;                   // [0, kPc): K dS' (hi part, lo part)
    const uint32_t tY = tmem_slot + kPc;             // [kPc, kPc + 2 TV): A^T dO, then dRes
    const uint32_t tS = tmem_slot + kPc + 2 * TV;    // then NE columns: dS

    auto issue_kq = [&](int c) {
        mbar_arrive_expect_tx(&bar_kq, 4 * kBoxBytes);
        for (int j = 0; j < 2; ++j) {
            tma_load_4d(sKQ + j * 2 * kBoxBytes, &map_k, &bar_kq, 64 * j, h, tbeg + c * 64, b);
            tma_load_4d(sKQ + j * 2 * kBoxBytes + kBoxBytes, &map_q, &bar_kq, 64 * j, h, tbeg + c * 64, b);
        }
    };
    auto issue_av = [&](int c) {
        const size_t idx = size_t(b * H + h) * NT + cb + c;
        mbar_arrive_expect_tx(&bar_av, 4 * kBoxBytes + 64 * TV * 2 + CB * 4);
        for (int j = 0; j < 4; ++j) tma_load_2d(sBT + j * kBoxBytes, &map_bt, &bar_av, 0, int(idx * 256 + 64 * j));
        tma_load_4d(sdO, &map_do, &bar_av, n0, h, tbeg + c * 64, b);
        bulk_load(sCoef + (c & 1) * CB, p.coef + idx * CB, CB * 4, &bar_av);
    };
    // This thread's part (row r, TVH columns) of slice e of the gradient at the end of chunk
    // c -> the operand of MMA-A'(c), and the fp32 checkpoint when checkpoints are not tiles
    auto put_operand = [&](int c, int e, const float* v) {
#pragma unroll
        for (int n = 0; n < TVH; n += 8)
            st8_split(sDh, sDl, e * blk_bytes<TV>() + blk_offset<TV>(r, cofs + n), v + n);
        if (!p.ck_tiles && r < p.dk) {
            const size_t slab = (((size_t(b) * H + h) * NT + cb + c) * E + e) * p.dk * dv;
            store_f32_row(p.dSck + slab + size_t(r) * dv + n0 + cofs, v, TVH);
        }
    };
    auto stage_operand = [&](int c) {
        #pragma unroll
        for (int e0 = 0; e0 < E; e0 += GRP) {
            float v[GRP * TVH];
#pragma unroll
            for (int g = 0; g < GRP; ++g) tmem_ld<TVH>(tmem_lane_addr(tS, warp, (e0 + g) * TV + cofs), v + g * TVH);
            tmem_wait_ld();
#pragma unroll
            for (int g = 0; g < GRP; ++g) put_operand(c, e0 + g, v + g * TVH);
        }
    };
    // The slab rescaled in place by gamma^C_c: chunk c's MMA-C' accumulates onto it.
    auto scale_state = [&](int c) {
        const float* gc = sCoef + (c & 1) * CB + 3 * 64 * E;
        #pragma unroll
        for (int e0 = 0; e0 < E; e0 += GRP) {
            float v[GRP * TVH];
#pragma unroll
            for (int g = 0; g < GRP; ++g) tmem_ld<TVH>(tmem_lane_addr(tS, warp, (e0 + g) * TV + cofs), v + g * TVH);
            tmem_wait_ld();
#pragma unroll
            for (int g = 0; g < GRP; ++g) {
                const float gm = gc[e0 + g];
#pragma unroll
                for (int i = 0; i < TVH; ++i) v[g * TVH + i] *= gm;
                tmem_st<TVH>(tmem_lane_addr(tS, warp, (e0 + g) * TV + cofs), v + g * TVH);
            }
        }
        tmem_wait_st();
    };
    // Gradient of the final state (dht or zero): operand of MMA-A'(nct-1) and the scaled slab.
    auto stage_dht = [&](int c) {
        const float* gc = sCoef + (c & 1) * CB + 3 * 64 * E;
        #pragma unroll
        for (int e = 0; e < E; ++e) {
            float v[TVH];
            if (p.dht && r < p.dk) {
                const float4* src = reinterpret_cast<const float4*>(
                    p.dht + ((size_t(sb * H + h) * E + e) * p.dk + r) * dv + n0 + cofs);
#pragma unroll
                for (int i = 0; i < TVH / 4; ++i) {
                    const float4 x = src[i];
                    v[4 * i] = x.x; v[4 * i + 1] = x.y; v[4 * i + 2] = x.z; v[4 * i + 3] = x.w;
                }
            } else {
#pragma unroll
                for (int i = 0; i < TVH; ++i) v[i] = 0.f;
            }
            put_operand(c, e, v);
            const float gm = gc[e];
#pragma unroll
            for (int i = 0; i < TVH; ++i) v[i] *= gm;
            tmem_st<TVH>(tmem_lane_addr(tS, warp, e * TV + cofs), v);
        }
        tmem_wait_st();
    };

    // Checkpoint of dS' at the end of chunk c: this CTA's columns of the slice blocks,
    // stored by TMA (thread 0, once the operand of chunk c is complete in shared memory).
    auto issue_ckpt = [&](int c) {
        if (!p.ck_tiles) return;
        tma_store_4d(&map_ck, sDh, n0, 0, ((b * H + h) * NT + cb + c) * E, 0);   // [hi|lo][E][dk][TV]
        bulk_commit();
    };

    // MMA-A' for slices [half * EP, half * EP + EP) into P' (thread 0)
    auto issue_pa = [&](int half) {
        // dS' lo blocks follow the hi blocks: one descriptor spans both when side by side
        const uint32_t ida = idesc_bf16_f32(64, kSide ? 2 * NE : EP * TV, 0, 1);
        // descriptors built once; each K step advances their start addresses
        const uint32_t hb = uint32_t(half) * EP * blk_bytes<TV>();
        const uint64_t a0 = smem_desc(smem_u32(sKQ), 16, 1024);
        const uint64_t dh0 = smem_desc(smem_u32(sDh) + hb, blk_bytes<TV>(), 16 * TV, kSwz);
        const uint64_t dl0 = smem_desc(smem_u32(sDl) + hb, blk_bytes<TV>(), 16 * TV, kSwz);
#pragma unroll
        for (int ks = 0; ks < kDk / 16; ++ks) {
            if (ks * 16 >= p.dk) break;   // the padded key rows are zero
            const int blk = ks >> 2, kk = (ks & 3) * 16;
            const uint64_t ad = desc_add(a0, blk * 2 * kBoxBytes + kk * 2);
            const uint32_t ko = ks * 32 * TV;   // 16 rows of the slice blocks per K step
            umma_bf16(tP, ad, desc_add(dh0, ko), ida, ks > 0 ? 1u : 0u);
            if (!kSide) umma_bf16(tP, ad, desc_add(dl0, ko), ida, 1u);
        }
    };

    // MMA-0 of the chunk whose A^T/T^T and dO tiles are in shared memory (thread 0): Y = A^T dO
    auto issue_y = [&]() {
        const uint32_t id0 = idesc_bf16_f32(64, TV, 1, 1);
        const uint64_t o0 = smem_desc(smem_u32(sdO), blk_bytes<TV>(), 16 * TV, kSwz);
        // A^T MN-major: K = the rows of A (16 per step, 2048 bytes), M = its 64 columns
        const uint64_t t0d = smem_desc(smem_u32(sBT), 2 * kBoxBytes, 1024);
#pragma unroll
        for (int ks = 0; ks < 4; ++ks) {
            const uint64_t bd = desc_add(o0, ks * 32 * TV);
            umma_bf16(tY, desc_add(t0d, ks * 2048), bd, id0, ks > 0 ? 1u : 0u);
            umma_bf16(tY, desc_add(t0d, kBoxBytes + ks * 2048), bd, id0, 1u);
        }
    };

    bool failed = false;
    uint32_t mma_phase = 0;
    int pending_mma = 0;
    bool y_early = false;   // thread 0: the next chunk's MMA-0 issued, not yet committed
    bool scaled = true;   // the slab already holds gamma^C-scaled values for the current chunk
    if (tid == 0) {
        issue_kq(nct - 1);
        issue_av(nct - 1);
    }
    if (!mbar_wait(&bar_av, 0)) failed = true;
    if (__syncthreads_or(failed)) failed = true;
    if (!failed) {
        stage_dht(nct - 1);
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        tc_fence_after();
    }

    for (int c = nct - 1; c >= 0 && !failed; --c) {
        const int it = nct - 1 - c;                // iteration index (barrier phases)
        const int t0 = tbeg + c * 64, n = min(64, tlen - c * 64);
        // dv leaves as one TMA store of the chunk's tile, except for a packed document's partial
        // last chunk, whose tile rows past its end belong to the next document
        const bool tma_dv = !p.dtab || n == 64;
        const float* cf = sCoef + (c & 1) * CB;
        const float* ae = cf;
        const float* be = cf + 64 * E;
        const float* we = cf + 128 * E;
        // previous chunk's key and query boxes into L2 (their TMA load waits for MMA-C')
        if (tid == 0 && c > 0)
            for (int j = 0; j < 2; ++j) {
                tma_prefetch_l2_4d(&map_k, 64 * j, h, tbeg + (c - 1) * 64, b);
                tma_prefetch_l2_4d(&map_q, 64 * j, h, tbeg + (c - 1) * 64, b);
            }
        bool ok = mbar_wait(&bar_kq, it & 1);
        if (__syncthreads_or(!ok)) { failed = true; break; }
        tc_fence_after();

        // ---- MMA-A' (P' = K dS') and MMA-0 (Y = A^T dO; issued at the end of the previous
        // chunk, off the chain, except for the first); one commit covers both
        if (tid == 0) {
            if (!y_early) issue_y();
            issue_pa(0);
            umma_commit(&bar_mma);
            y_early = false;
            issue_ckpt(c);   // the dS' blocks were completed before the last barrier
        }
        pending_mma = 1;
        // while the products run: the slab rescaled by this chunk's gamma^C (MMA-C' of this
        // chunk accumulates onto it), and the dO row of this thread's M=64 row (lanes 16-31)
        if (!scaled) scale_state(c);
        scaled = false;
        float dorow[TVH];
        if (!row_thread) {
#pragma unroll
            for (int i = 0; i < TVH; i += 8) {
                const uint4 u = *reinterpret_cast<const uint4*>(sdO + blk_offset<TV>(r64, cofs + i));
                const __nv_bfloat162* pb = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const float2 f = __bfloat1622float2(pb[j]);
                    dorow[i + 2 * j] = f.x;
                    dorow[i + 2 * j + 1] = f.y;
                }
            }
        }
        ok = mbar_wait(&bar_mma, mma_phase);
        mma_phase ^= 1;
        // dU is written next into the dv tile's space, so the previous chunk's dv copy must
        // have read it (the checkpoint copy, the most recent group, may still be reading dS')
        if (tid == 0) {
            if (p.ck_tiles) bulk_wait_read_but_last();
            else bulk_wait_read_all();   // no checkpoint copies: the dv copy is the last group
        }
        if (__syncthreads_or(!ok)) { failed = true; break; }
        pending_mma = 0;
        tc_fence_after();

        // ---- dU = Y + sum_e w_e (.) P'_e   (row threads; the loads are warp-wide)
        {
            float du[TVH], wr[E];
#pragma unroll
            for (int e = 0; e < E; ++e) wr[e] = row_thread ? we[e * 64 + r64] : 0.f;
            tmem_ld<TVH>(tmem_lane_addr(tY, warp, cofs), du);
            // adds w_e (.) P'_e for the EP slices from EB on (P' columns from 0)
            auto add_p = [&](auto eb) {
                constexpr int EB = decltype(eb)::value;
#pragma unroll
                for (int e0 = 0; e0 < EP; e0 += GRP) {
                    float pv[GRP * TVH];
#pragma unroll
                    for (int g = 0; g < GRP; ++g) tmem_ld<TVH>(tmem_lane_addr(tP, warp, (e0 + g) * TV + cofs), pv + g * TVH);
                    if constexpr (kSide) {   // the lo part of K dS'
                        float pl[GRP * TVH];
#pragma unroll
                        for (int g = 0; g < GRP; ++g)
                            tmem_ld<TVH>(tmem_lane_addr(tP, warp, NE + (e0 + g) * TV + cofs), pl + g * TVH);
                        tmem_wait_ld();
#pragma unroll
                        for (int i = 0; i < GRP * TVH; ++i) pv[i] += pl[i];
                    } else {
                        tmem_wait_ld();
                    }
#pragma unroll
                    for (int g = 0; g < GRP; ++g)
#pragma unroll
                        for (int i = 0; i < TVH; ++i) du[i] = fmaf(wr[EB + e0 + g], pv[g * TVH + i], du[i]);
                }
            };
            add_p(std::integral_constant<int, 0>{});
            if constexpr (kSplitP) {   // the second half of the slices into the same columns
                tc_fence_before();
                __syncthreads();
                tc_fence_after();
                if (tid == 0) {
                    issue_pa(1);
                    umma_commit(&bar_mma);
                }
                pending_mma = 1;
                ok = mbar_wait(&bar_mma, mma_phase);
                mma_phase ^= 1;
                if (__syncthreads_or(!ok)) { failed = true; break; }
                pending_mma = 0;
                tc_fence_after();
                add_p(std::integral_constant<int, EP>{});
            }
            if (row_thread) {
#pragma unroll
                for (int i = 0; i < TVH; i += 8) st8_split(sUh, sUl, blk_offset<TV>(r64, cofs + i), du + i);
                if (p.ck_tiles) store_tok_tile(p.dUbuf, (size_t(b) * H + h) * NT + cb + c, dv, r64, n0 + cofs, du, TVH, r64 < n);
                else if (r64 < n) store_f32_row(p.dUbuf + tok_idx(b, t0 + r64, h, n0 + cofs, T, H, dv), du, TVH);
            }
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        tc_fence_after();

        // ---- MMA-B': dRes = T^T dU   (into tY; dU MN-major)
        if (tid == 0) {
            // T^T_hi [dU_hi | dU_lo] (N = 2 TV: the lo block is the next swizzle atom, TV * 128
            // bytes on) into tY columns [0, 2 TV), and T^T_lo dU_hi into [0, TV)
            const uint32_t idb2 = idesc_bf16_f32(64, 2 * TV, 1, 1);
            const uint32_t idb = idesc_bf16_f32(64, TV, 1, 1);
            const uint64_t t0d = smem_desc(smem_u32(sBT), 2 * kBoxBytes, 1024);   // T^T MN-major
            const uint64_t u0 = smem_desc(smem_u32(sUh), TV * 128, 16 * TV, kSwz);
#pragma unroll
            for (int ks = 0; ks < 4; ++ks) {
                const uint64_t th = desc_add(t0d, 2 * kBoxBytes + ks * 2048);
                const uint64_t tl = desc_add(t0d, 3 * kBoxBytes + ks * 2048);
                const uint64_t uh = desc_add(u0, ks * 32 * TV);
                umma_bf16(tY, th, uh, idb2, ks > 0 ? 1u : 0u);
                umma_bf16(tY, tl, uh, idb, 1u);
            }
            umma_commit(&bar_mma);
        }
        pending_mma = 1;
        ok = mbar_wait(&bar_mma, mma_phase);
        mma_phase ^= 1;
        if (tid == 0) bulk_wait_read_all();   // the MMA-C' operand rows overwrite dS' next
        if (__syncthreads_or(!ok)) { failed = true; break; }
        pending_mma = 0;
        tc_fence_after();
        if (tid == 0 && c > 0) issue_av(c - 1);   // A^T/T^T tiles, dO tile, other coef buffer free

        // ---- operand rows of MMA-C': [-a_e (.) dRes ; b_e (.) dO]
        {
            float dr[TVH], cr[E];   // -a_e (row threads) or b_e (dO rows) of this thread's row
#pragma unroll
            for (int e = 0; e < E; ++e) cr[e] = row_thread ? -ae[e * 64 + r64] : be[e * 64 + r64];
            {
                float drl[TVH];
                tmem_ld<TVH>(tmem_lane_addr(tY, warp, cofs), dr);
                tmem_ld<TVH>(tmem_lane_addr(tY, warp, TV + cofs), drl);
                tmem_wait_ld();
#pragma unroll
                for (int i = 0; i < TVH; ++i) dr[i] += drl[i];
            }
            if (row_thread) {
                if (tma_dv) {   // row of the dv tile; thread 0 stores the tile after the barrier
                    if (p.out_f32) store_f32_row(reinterpret_cast<float*>(sDvo) + r64 * TV + cofs, dr, TVH);
                    else store_row(sDvo, size_t(r64) * TV + cofs, dr, TVH, 0);
                }
                if (r64 < n) {
                    const size_t off = tok_idx(b, t0 + r64, h, n0 + cofs, T, H, dv);
                    if (!p.ck_tiles) store_f32_row(p.dRbuf + off, dr, TVH);
                    if (!tma_dv) store_row(p.dv_out, off, dr, TVH, p.out_f32);
                }
                if (p.ck_tiles && p.use_delta) {   // -dRes, the operand sign the gradient kernel uses
                    float ndr[TVH];
#pragma unroll
                    for (int i = 0; i < TVH; ++i) ndr[i] = -dr[i];
                    store_tok_tile(p.dRbuf, (size_t(b) * H + h) * NT + cb + c, dv, r64, n0 + cofs, ndr, TVH, r64 < n);
                }
                if (p.use_delta) {
#pragma unroll
                    for (int e = 0; e < E; ++e) {
                        const float a = cr[e];
                        float x[TVH];
#pragma unroll
                        for (int i = 0; i < TVH; ++i) x[i] = a * dr[i];
#pragma unroll
                        for (int i = 0; i < TVH; i += 8)
                            st8_split(sBh, sBl, sw128_offset(r64, e * TV + cofs + i, 128), x + i);
                    }
                }
            } else {
#pragma unroll
                for (int e = 0; e < E; ++e) {
                    const float bq = cr[e];
                    float x[TVH];
#pragma unroll
                    for (int i = 0; i < TVH; ++i) x[i] = bq * dorow[i];
#pragma unroll
                    for (int i = 0; i < TVH; i += 8)
                        st8_split(sBh, sBl, sw128_offset(64 + r64, e * TV + cofs + i, 128), x + i);
                }
            }
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        tc_fence_after();

        // ---- MMA-C': dS += [K^T | Q^T] [-a dRes ; b dO]   (sGLA: query half only)
        if (tid == 0) {
            const uint32_t idc = idesc_bf16_f32(128, NE, 1, 1);
            const uint64_t a0 = smem_desc(smem_u32(sKQ), 2 * kBoxBytes, 1024);
            const uint64_t bh0 = smem_desc(smem_u32(sBh), 128 * 128, 1024);
            const uint64_t bl0 = smem_desc(smem_u32(sBl), 128 * 128, 1024);
            for (int ks = p.use_delta ? 0 : 4; ks < 8; ++ks) {
                const uint64_t ad = desc_add(a0, ks * 2048);
                umma_bf16(tS, ad, desc_add(bh0, ks * 2048), idc, 1u);
                umma_bf16(tS, ad, desc_add(bl0, ks * 2048), idc, 1u);
            }
            umma_commit(&bar_mma);
            if (tma_dv) {   // rows past T are skipped by the store
                tma_store_4d(&map_dv, sDvo, n0, h, t0, b);
                bulk_commit();
            }
        }
        pending_mma = 1;
        ok = mbar_wait(&bar_mma, mma_phase);
        mma_phase ^= 1;
        if (c > 0) ok = ok && mbar_wait(&bar_av, (it + 1) & 1);   // gamma^C of chunk c-1
        if (__syncthreads_or(!ok)) { failed = true; break; }
        pending_mma = 0;
        tc_fence_after();
        if (tid == 0 && c > 0) {
            issue_kq(c - 1);
            // chunk c-1's MMA-0: its tiles have arrived (bar_av above), and Y is free (this
            // chunk's dRes was read before MMA-C'); it runs under the operand staging below
            issue_y();
            y_early = true;
        }

        if (c > 0) {
            stage_operand(c - 1);   // its gamma^C scaling follows the next MMA-A' issue
        } else if (p.dh0) {
            #pragma unroll
            for (int e0 = 0; e0 < E; e0 += GRP) {
                float v[GRP * TVH];
#pragma unroll
                for (int g = 0; g < GRP; ++g) tmem_ld<TVH>(tmem_lane_addr(tS, warp, (e0 + g) * TV + cofs), v + g * TVH);
                tmem_wait_ld();
#pragma unroll
                for (int g = 0; g < GRP; ++g)
                    if (r < p.dk)
                        store_f32_row(p.dh0 + ((size_t(sb * H + h) * E + e0 + g) * p.dk + r) * dv + n0 + cofs,
                                      v + g * TVH, TVH);
            }
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        tc_fence_after();
    }

    if (failed && tid == 0) {
        record_device_error(p.err, TLA_ERR_TIMEOUT);
        if (pending_mma) mbar_wait(&bar_mma, mma_phase ^ 1);
        if (y_early) {   // an MMA-0 issued ahead and not yet committed
            umma_commit(&bar_mma);
            mbar_wait(&bar_mma, mma_phase);
        }
    }
    if (tid == 0) bulk_wait_all();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tmem_dealloc(tmem_slot, tcols);
}

template <int TV, int E>
cudaError_t launch_tv(const tla_problem& p, const FwdPlan& fp, const char* fws, const BwdPlan& bp,
                      char* bws, const void* dO, const float* dht, void* dv, float* dh0, int* err,
                      cudaStream_t s) {
    if (p.E != E || fp.tc_tv != TV) return cudaErrorInvalidValue;
    CUtensorMap mk, mq, mo, mb, mc, mdv;
    const int NT = fp.NT;
    if (!make_token_map(&mk, p.k, p.B, p.T, p.H, p.dk, 64, 64, true) ||
        !make_token_map(&mq, p.q, p.B, p.T, p.H, p.dk, 64, 64, true) ||
        !make_token_map_sw(&mo, dO, p.B, p.T, p.H, p.dv, TV, 64) ||
        !make_matrix_map(&mb, fws + fp.BT, (long long)p.B * p.H * NT * 256, 64, 64, 64) ||
        !make_token_map(&mdv, dv, p.B, p.T, p.H, p.dv, TV, 64, false,
                        p.out_dtype == TLA_FP32 ? 4 : 2))
        return cudaErrorInvalidValue;
    memset(&mc, 0, sizeof(mc));   // unused unless the checkpoints are tiles
    if (fp.ck_tiles &&
        !make_ckpt_map(&mc, bws + bp.dS, (long long)p.B * p.H * NT * p.E, p.dv, TV, p.E, 2 * TV))
        return cudaErrorInvalidValue;
    TcBwdArgs a;
    a.coef = (const float*)(fws + fp.coef);
    a.dht = dht;
    a.dv_out = dv;
    a.dh0 = dh0;
    a.dUbuf = (float*)(bws + bp.dU);
    a.dRbuf = (float*)(bws + bp.dRes);
    a.dSck = (float*)(bws + bp.dS);
    a.err = err;
    a.T = p.T; a.H = p.H; a.dv = p.dv; a.E = p.E; a.NT = NT;
    a.use_delta = p.use_delta; a.out_f32 = p.out_dtype == TLA_FP32;
    a.ck_tiles = fp.ck_tiles;
    a.dk = p.dk;
    a.dtab = p.cu_seqlens ? (const int4*)(fws + fp.dtab) : nullptr;
    const size_t smem = tc_bwd_smem_c<TV>(E);
    auto kern = bwd_recurrence_tc_kernel<TV, E>;
    cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    dim3 grid(p.dv / TV, p.H, fp.nseq);
    prof_before("bwd_recurrence_tc", s);
    kern<<<grid, kThreads, smem, s>>>(mk, mq, mo, mb, mc, mdv, a);
    prof_after(s);
    return cudaGetLastError();
}

}  // namespace

// The backward recurrence runs on tensor cores when the forward used them and
// the dS slab, the M=64 products and their operands fit TMEM (512 columns) and
// shared memory.
int tc_bwd_ok(const tla_problem& p, int tv) {
    if (tv == 0) return 0;
    const int ne = p.E * tv;
    int pc = 2 * ne <= 256 ? 2 * ne : ne;   // TMEM columns of K dS' (side by side or not)
    if (pc == ne && pc + 2 * tv + ne > 512 && p.E % 2 == 0) pc = ne / 2;   // by halves of the slices
    if (pc + 2 * tv + ne > 512) return 0;
    const size_t smem = tv == 16 ? tc_bwd_smem_c<16>(p.E)
                                 : tv == 32 ? tc_bwd_smem_c<32>(p.E) : tc_bwd_smem_c<64>(p.E);
    return smem <= 227 * 1024 ? 1 : 0;
}

cudaError_t launch_bwd_recurrence_tc(const tla_problem& p, const FwdPlan& fp, const char* fws,
                                     const BwdPlan& bp, char* bws, const void* dO,
                                     const float* dht, void* dv, float* dh0, int* err,
                                     cudaStream_t s) {
    // one instance per slice count the tensor-core path takes (tc_fwd_tv, tc_bwd_ok)
    switch (p.E) {
        case 1: return launch_tv<64, 1>(p, fp, fws, bp, bws, dO, dht, dv, dh0, err, s);
        case 2: return launch_tv<32, 2>(p, fp, fws, bp, bws, dO, dht, dv, dh0, err, s);
        case 3: return launch_tv<64, 3>(p, fp, fws, bp, bws, dO, dht, dv, dh0, err, s);
        case 4: return launch_tv<16, 4>(p, fp, fws, bp, bws, dO, dht, dv, dh0, err, s);
        case 6: return launch_tv<32, 6>(p, fp, fws, bp, bws, dO, dht, dv, dh0, err, s);
        case 8: return launch_tv<16, 8>(p, fp, fws, bp, bws, dO, dht, dv, dh0, err, s);
        case 12: return launch_tv<16, 12>(p, fp, fws, bp, bws, dO, dht, dv, dh0, err, s);
        case 16: return launch_tv<16, 16>(p, fp, fws, bp, bws, dO, dht, dv, dh0, err, s);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace tla
