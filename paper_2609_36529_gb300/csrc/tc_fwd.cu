// Tensor-core (tcgen05) forward recurrence over chunks, Appendix A, Eq. joint-chunk.
//
// One CTA of 8 warps per (b, h, block of TV value columns); value columns never
// interact (Section 2.5, Eq. slices), so each CTA carries its own E x dk x TV
// slab of the fp32 state in tensor memory for the whole sequence.  Per chunk of
// C = 64 positions, with a_e = k'_e (.) gamma_e, b_e = q'_e (.) gamma_e and
// w_e = k'_e (.) gamma^C_e / gamma_e (precomputed per chunk by the prep kernel):
//   MMA-A  P  = [K; Q] S_all          (M=128 rows: 64 key rows, 64 query rows;
//                                      N = NE = E*TV columns, slice-major; K = dk; the hi
//                                      and lo halves of S side by side, N = 2 NE, when
//                                      that fits one instruction)
//   epi-A  Res = V - sum_e diag(a_e) P_K,e   (delta rule; sGLA: Res = V)
//          Oi  = sum_e diag(b_e) P_Q,e       (kept in registers)
//   MMA-B  [U; Oa] = [T; A T] Res      (M=128, K=64; T and A T from the prep kernel; the
//                                      hi*hi and hi*lo terms in one N = 2 TV product)
//   epi-B  O = Oi + Oa;  Ut_e = diag(w_e) U
//   MMA-C  S_all += K^T [Ut_1 .. Ut_E] (M=dk=128, K=64, N=NE; K^T read MN-major
//                                      straight from the TMA-loaded key tile)
//   epi-C  S_{[c+1]} from TMEM: operand of the next MMA-A (also the checkpoint);
//          once that product is issued, the TMEM slab is rescaled in place by
//          gamma^C of the next chunk for its MMA-C (off the critical path).
// Accumulation is fp32 in TMEM.  Keys and queries are bf16 inputs and enter the
// products exactly; every other operand (the state, Res, T, A T, Ut) is carried
// as a pair of bf16 values hi + lo (lo = bf16 of the rounding remainder), and
// each product sums the hi*hi, hi*lo and lo*hi terms (only x*hi and x*lo when
// the other side is an exact key or query).  This keeps the products near fp32
// accuracy: with a single bf16 rounding of those operands the error of o and of
// the state reaches the 2e-2 x RMS parity bound.
// Thread layout: warp w reads TMEM lanes 32 (w % 4) .. +31 (the rows of every
// product), and warps 0-3 / 4-7 take the first / second half of each slice's TV
// value columns, so every epilogue is split over 256 threads; TMEM loads of
// several slices are issued before one wait.  E is a compile-time parameter, so the
// per-slice loops unroll and each thread holds its row's coefficients (read from the
// slice-major coefficient block, conflict-free) in registers.  The state, Res and Ut operands
// are stored MN-major (value columns contiguous: 16-byte stores of a thread's
// row).  The state operand is kept as one swizzled [dk][TV] block per slice
// (tc_common.cuh); a chunk's checkpoint leaves shared memory as one TMA tensor
// store of those blocks into the row-major [dk][dv] hi and lo matrices of its
// slices (tma_host.h).  Key, query, value tiles, the [T; A T] tiles and the
// coefficient block arrive by TMA, prefetched one chunk ahead as soon as their
// buffers are free.  Every mbarrier wait is bounded by the GPU global timer; on
// expiry the CTA records TLA_ERR_TIMEOUT and leaves after a bounded drain of
// its outstanding work.
#include <algorithm>
#include <cstring>

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
constexpr int kBoxBytes = 64 * 64 * 2;  // one 64 x 64 bf16 TMA box

struct TcFwdArgs {
    const float* coef;   // [B,H,NT, 3*64*E + 16] per-chunk coefficient blocks
    const float* h0;
    void* o;
    float* ht;
    float* Sck;
    float* Ubuf;
    float* Rbuf;
    int* err;
    const int4* dtab;    // packed documents: (first token, chunks, first chunk, tokens); else NULL
    int T, H, dv, E, NT, use_delta, save, out_f32, ck_tiles;
    int dk;              // key dimension: 128, or 64 padded to 128 by zero rows (TMA fill)
};

template <int TV>
__host__ __device__ constexpr size_t tc_fwd_smem_c(int E) {
    return 1024 + 4 * kBoxBytes + 4 * kBoxBytes + size_t(E) * TV * 512 + 64 * TV * 2 + 64 * TV * 4 +
           2 * (3 * 64 * E + 16) * 4;
}
// CTAs per SM the launch bounds plan for: two (at most 128 registers a thread) when two fit
// in shared memory, else one.
template <int TV, int E>
__host__ __device__ constexpr int fwd_min_blocks() {
    return tc_fwd_smem_c<TV>(E) <= 113 * 1024 ? 2 : 1;
}

template <int TV, int E>
__global__ void __launch_bounds__(kThreads, (fwd_min_blocks<TV, E>()))
fwd_recurrence_tc_kernel(const __grid_constant__ CUtensorMap map_k,
                         const __grid_constant__ CUtensorMap map_q,
                         const __grid_constant__ CUtensorMap map_v,
                         const __grid_constant__ CUtensorMap map_a2,
                         const __grid_constant__ CUtensorMap map_ck,
                         const __grid_constant__ CUtensorMap map_o, const TcFwdArgs p) {
    constexpr int TVH = TV / 2;             // value columns per thread
    constexpr int GRP0 = TVH >= 32 ? 1 : 32 / TVH;
    constexpr int GRP = GRP0 < E ? GRP0 : E;   // slices per batch of TMEM loads
    static_assert(E % GRP == 0, "slices per batch must divide E");
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
    constexpr int NE = E * TV;
    constexpr int CB = 3 * 64 * E + 16;        // floats per coefficient block
    uint8_t* sKQ = sm;                         // 2 blocks x [K rows 0-63 | Q rows 64-127] x 128 B
    uint8_t* sA2 = sKQ + 4 * kBoxBytes;        // [T; A T] 128 x 64 bf16: hi tile, lo tile
    uint8_t* sReg = sA2 + 4 * kBoxBytes;       // shared region, NE * 512 bytes:
    uint8_t* sSh = sReg;                       //   S_all hi: E blocks [dk][TV] (MMA-A operand,
    uint8_t* sSl = sReg + NE * 256;            //   S_all lo                     checkpoint source)
    uint8_t* sUh = sReg;                       //   Ut [64][NE] hi, lo, MN-major (after MMA-B)
    uint8_t* sUl = sUh + NE * 128;
    __nv_bfloat16* sV = reinterpret_cast<__nv_bfloat16*>(sReg + NE * 512);  // [64][TV]
    uint8_t* sOo = sReg + NE * 512 + 64 * TV * 2;                             // o tile [64][TV] (TMA store)
    uint8_t* sRh = sOo;                        // Res [64][TV] hi, lo, MN-major (epi-A to MMA-B),
    uint8_t* sRl = sOo + TV * 128;             // in the o tile's space: the checkpoint copy of
                                               // the state operand proceeds under epi-A and MMA-B
    float* sCoef = reinterpret_cast<float*>(sOo + 64 * TV * 4);               // 2 x CB

    __shared__ __align__(8) uint64_t bar_kq, bar_av, bar_mma;
    __shared__ uint32_t tmem_slot;

    const int tid = threadIdx.x, warp = tid >> 5;
    const int r = tid & 127;                   // TMEM lane: row of every product
    const int cofs = (tid >> 7) * TVH;         // this thread's first column within a slice
    const int nb = blockIdx.x, h = blockIdx.y, sb = blockIdx.z;   // sb: sequence or document
    const int n0 = nb * TV;
    const int T = p.T, H = p.H, dv = p.dv, NT = p.NT;
    // hi and lo halves of the state product side by side in one N = 2 NE product (half the
    // UMMAs on the chain) when N fits one instruction; P then takes 2 NE columns
    constexpr bool kSide = 2 * NE <= 256;
    constexpr int kPc = kSide ? 2 * NE : NE;   // TMEM columns of P
    constexpr uint32_t tcols = (kPc + NE <= 256) ? 256u : 512u;
    constexpr uint64_t kSwz = swizzle_code(2 * TV);
    // token batch, first token, tokens, chunks and first chunk (in the workspace) of this state
    int b = sb, tbeg = 0, tlen = T, nct = NT, cb = 0;
    if (p.dtab) {
        const int4 dd = p.dtab[sb];
        b = 0; tbeg = dd.x; nct = dd.y; cb = dd.z; tlen = dd.w;
    }
    if (nct == 0) {   // empty document: the final state is the initial one
        if (p.ht && r < p.dk)
            for (int e = 0; e < E; ++e)
                for (int n = cofs; n < cofs + TVH; ++n) {
                    const size_t o = ((size_t(sb * H + h) * E + e) * p.dk + r) * dv + n0 + n;
                    p.ht[o] = p.h0 ? p.h0[o] : 0.f;
                }
        return;
    }

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
        tma_prefetch_desc(&map_v);
        tma_prefetch_desc(&map_a2);
        if (p.save && p.ck_tiles) tma_prefetch_desc(&map_ck);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tP = tmem_slot;         // columns [0, kPc): P (hi part, then lo part when
                                           // side by side), then [U; Oa] in [0, 2 TV)
    const uint32_t tS = tmem_slot + kPc;   // columns [kPc, kPc + NE): the state slab

    auto issue_kq = [&](int c) {
        mbar_arrive_expect_tx(&bar_kq, 4 * kBoxBytes);
        for (int j = 0; j < 2; ++j) {
            tma_load_4d(sKQ + j * 2 * kBoxBytes, &map_k, &bar_kq, 64 * j, h, tbeg + c * 64, b);
            tma_load_4d(sKQ + j * 2 * kBoxBytes + kBoxBytes, &map_q, &bar_kq, 64 * j, h, tbeg + c * 64, b);
        }
    };
    // [T; A T] hi/lo and V of chunk c, and its coefficient block into buffer c & 1
    auto issue_av = [&](int c) {
        const size_t idx = size_t(b * H + h) * NT + cb + c;
        mbar_arrive_expect_tx(&bar_av, 4 * kBoxBytes + 64 * TV * 2 + CB * 4);
        tma_load_2d(sA2, &map_a2, &bar_av, 0, int(idx * 256));
        tma_load_2d(sA2 + 2 * kBoxBytes, &map_a2, &bar_av, 0, int(idx * 256 + 128));
        tma_load_4d(sV, &map_v, &bar_av, n0, h, tbeg + c * 64, b);
        bulk_load(sCoef + (c & 1) * CB, p.coef + idx * CB, CB * 4, &bar_av);
    };
    // This thread's part (row r, TVH columns) of slice e of S_{[c]} -> the bf16 hi/lo
    // operand block of MMA-A, and the fp32 checkpoint when checkpoints are not tiles (tiles:
    // issue_ckpt stores the operand blocks).
    auto put_operand = [&](int c, int e, const float* v) {
#pragma unroll
        for (int n = 0; n < TVH; n += 8)
            st8_split(sSh, sSl, e * blk_bytes<TV>() + blk_offset<TV>(r, cofs + n), v + n);
        if (p.save && !p.ck_tiles && r < p.dk) {
            const size_t slab = (((size_t(b) * H + h) * NT + cb + c) * E + e) * p.dk * dv;
            store_f32_row(p.Sck + slab + size_t(r) * dv + n0 + cofs, v, TVH);
        }
    };
    // Operand of MMA-A(c) from the state slab in TMEM (S_{[c]}, the result of MMA-C(c-1)).
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
    // The slab rescaled in place by gamma^C_c: chunk c's state update accumulates onto it.
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
    // Initial state (h0 or zero): the operand of MMA-A(0) and the gamma^C_0-scaled slab.
    auto stage_h0 = [&]() {
        const float* gc = sCoef + 3 * 64 * E;
#pragma unroll
        for (int e = 0; e < E; ++e) {
            float v[TVH];
            if (p.h0 && r < p.dk) {
                const float4* src = reinterpret_cast<const float4*>(
                    p.h0 + ((size_t(sb * H + h) * E + e) * p.dk + r) * dv + n0 + cofs);
#pragma unroll
                for (int i = 0; i < TVH / 4; ++i) {
                    const float4 x = src[i];
                    v[4 * i] = x.x; v[4 * i + 1] = x.y; v[4 * i + 2] = x.z; v[4 * i + 3] = x.w;
                }
            } else {
#pragma unroll
                for (int i = 0; i < TVH; ++i) v[i] = 0.f;
            }
            put_operand(0, e, v);
            const float gm = gc[e];
#pragma unroll
            for (int i = 0; i < TVH; ++i) v[i] *= gm;
            tmem_st<TVH>(tmem_lane_addr(tS, warp, e * TV + cofs), v);
        }
        tmem_wait_st();
    };
    // Checkpoint of S_{[c]} (bf16 hi/lo) for the backward: this CTA's columns of the slice
    // blocks, stored by TMA (thread 0, after the operand is complete).
    auto issue_ckpt = [&](int c) {
        if (!(p.save && p.ck_tiles)) return;
        tma_store_4d(&map_ck, sSh, n0, 0, ((b * H + h) * NT + cb + c) * E, 0);   // [hi|lo][E][dk][TV]
        bulk_commit();
    };
    // MMA-A: P = [K; Q] S_all    (B = S_all, MN-major, hi and lo)
    auto issue_mma_a = [&]() {
        // descriptors built once; each K step advances their start addresses
        const uint64_t a0 = smem_desc(smem_u32(sKQ), 16, 1024);
        const uint64_t bh0 = smem_desc(smem_u32(sSh), blk_bytes<TV>(), 16 * TV, kSwz);
        const uint64_t bl0 = smem_desc(smem_u32(sSl), blk_bytes<TV>(), 16 * TV, kSwz);
        // B = the slice blocks: 16 rows (two 8-row groups) per K step, one TV-column swizzle
        // atom per slice; the lo blocks follow the hi blocks, so one descriptor spans both
        const uint32_t idesc = idesc_bf16_f32(128, kSide ? 2 * NE : NE, 0, 1);
#pragma unroll
        for (int ks = 0; ks < kDk / 16; ++ks) {
            if (ks * 16 >= p.dk) break;   // the padded key rows are zero
            const int blk = ks >> 2, kk = (ks & 3) * 16;
            const uint64_t ad = desc_add(a0, blk * 2 * kBoxBytes + kk * 2);
            const uint32_t ko = ks * 32 * TV;
            umma_bf16(tP, ad, desc_add(bh0, ko), idesc, ks > 0 ? 1u : 0u);
            if (!kSide) umma_bf16(tP, ad, desc_add(bl0, ko), idesc, 1u);
        }
        umma_commit(&bar_mma);
    };

    // this thread's columns of P for slices e0 .. e0 + GRP - 1 (the hi and lo parts summed
    // when the halves were multiplied side by side)
    auto load_p = [&](int e0, float* pv) {
#pragma unroll
        for (int g = 0; g < GRP; ++g) tmem_ld<TVH>(tmem_lane_addr(tP, warp, (e0 + g) * TV + cofs), pv + g * TVH);
        if constexpr (kSide) {
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
    };

    bool failed = false;
    uint32_t mma_phase = 0;
    int pending_mma = 0;
    if (tid == 0) {
        issue_kq(0);
        issue_av(0);
    }
    if (!mbar_wait(&bar_av, 0)) failed = true;
    if (__syncthreads_or(failed)) failed = true;
    if (!failed) {
        stage_h0();
        fence_proxy_async_smem();
        tc_fence_before();
        const bool ok = mbar_wait(&bar_kq, 0);
        if (__syncthreads_or(!ok)) failed = true;
        tc_fence_after();
        if (!failed) {
            if (tid == 0) {
                issue_mma_a();
                issue_ckpt(0);
            }
            pending_mma = 1;
        }
    }

    for (int c = 0; c < nct && !failed; ++c) {
        const int t0 = tbeg + c * 64, n = min(64, tlen - c * 64);
        // o leaves as one TMA store of the chunk's tile, except for a packed document's partial
        // last chunk, whose tile rows past its end belong to the next document
        const bool tma_o = !p.dtab || n == 64;
        const float* cf = sCoef + (c & 1) * CB;
        const float* ae = cf;
        const float* be = cf + 64 * E;
        const float* we = cf + 128 * E;
        // next chunk's key and query boxes into L2: their TMA load is issued only once
        // MMA-C(c) has released the tile, and then waits on the chain
        if (tid == 0 && c + 1 < nct)
            for (int j = 0; j < 2; ++j) {
                tma_prefetch_l2_4d(&map_k, 64 * j, h, tbeg + (c + 1) * 64, b);
                tma_prefetch_l2_4d(&map_q, 64 * j, h, tbeg + (c + 1) * 64, b);
            }
        // ---- wait for MMA-A(c) (issued at the end of the previous step); Res is written
        // next into the o tile's space, so the previous chunk's o copy must have read it (the
        // checkpoint copy, the most recent group, may still be reading the state operand)
        bool ok = mbar_wait(&bar_mma, mma_phase);
        mma_phase ^= 1;
        if (tid == 0) {
            if (p.save && p.ck_tiles) bulk_wait_read_but_last();
            else bulk_wait_read_all();   // no checkpoint copies: the o copy is the last group
        }
        tc_fence_before();
        if (__syncthreads_or(!ok)) { failed = true; break; }
        pending_mma = 0;
        tc_fence_after();

        // ---- epi-A: Res (key rows) and the inter-chunk read (query rows).  The per-row
        // coefficients of this thread's row for every slice come first (slice-major block:
        // a warp reads 32 consecutive rows of one slice), then the products.
        float oi[TVH], res[TVH], cr[E];
        {
            const float* crow = (r < 64 ? ae + r : be + (r - 64));
#pragma unroll
            for (int e = 0; e < E; ++e) cr[e] = crow[e * 64];
        }
        if (r < 64) {
            {
                const uint4* vrow = reinterpret_cast<const uint4*>(sV + r * TV + cofs);
#pragma unroll
                for (int i = 0; i < TVH / 8; ++i) {
                    uint4 u = vrow[i];
                    const __nv_bfloat162* pr = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        float2 f = __bfloat1622float2(pr[j]);
                        res[8 * i + 2 * j] = f.x;
                        res[8 * i + 2 * j + 1] = f.y;
                    }
                }
            }
            if (p.use_delta) {
#pragma unroll
                for (int e0 = 0; e0 < E; e0 += GRP) {
                    float pv[GRP * TVH];
                    load_p(e0, pv);
#pragma unroll
                    for (int g = 0; g < GRP; ++g)
#pragma unroll
                        for (int i = 0; i < TVH; ++i) res[i] = fmaf(-cr[e0 + g], pv[g * TVH + i], res[i]);
                }
            }
#pragma unroll
            for (int i = 0; i < TVH; i += 8) st8_split(sRh, sRl, blk_offset<TV>(r, cofs + i), res + i);
        } else {
#pragma unroll
            for (int i = 0; i < TVH; ++i) oi[i] = 0.f;
#pragma unroll
            for (int e0 = 0; e0 < E; e0 += GRP) {
                float pv[GRP * TVH];
                load_p(e0, pv);
#pragma unroll
                for (int g = 0; g < GRP; ++g)
#pragma unroll
                    for (int i = 0; i < TVH; ++i) oi[i] = fmaf(cr[e0 + g], pv[g * TVH + i], oi[i]);
            }
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        tc_fence_after();

        // ---- MMA-B: [U; Oa] = [T; A T] Res  (into columns [0, TV); Res MN-major)
        if (tid == 0) {
            // [T; A T]_hi [Res_hi | Res_lo] (N = 2 TV: the lo block is the next swizzle atom,
            // TV * 128 bytes on) into columns [0, 2 TV), and [T; A T]_lo Res_hi into [0, TV)
            const uint32_t idesc2 = idesc_bf16_f32(128, 2 * TV, 0, 1);
            const uint32_t idesc = idesc_bf16_f32(128, TV, 0, 1);
            const uint64_t ah0 = smem_desc(smem_u32(sA2), 16, 1024);
            const uint64_t bh0 = smem_desc(smem_u32(sRh), TV * 128, 16 * TV, kSwz);
#pragma unroll
            for (int ks = 0; ks < 4; ++ks) {
                const uint64_t ah = desc_add(ah0, ks * 32);
                const uint64_t al = desc_add(ah0, 2 * kBoxBytes + ks * 32);
                const uint64_t bh = desc_add(bh0, ks * 32 * TV);
                umma_bf16(tP, ah, bh, idesc2, ks > 0 ? 1u : 0u);
                umma_bf16(tP, al, bh, idesc, 1u);
            }
            umma_commit(&bar_mma);
        }
        pending_mma = 1;
        if (r < 64 && p.Rbuf) {   // while MMA-B runs
            if (p.ck_tiles) store_tok_tile(p.Rbuf, (size_t(b) * H + h) * NT + cb + c, dv, r, n0 + cofs, res, TVH, r < n);
            else if (r < n) store_f32_row(p.Rbuf + tok_idx(b, t0 + r, h, n0 + cofs, T, H, dv), res, TVH);
        }
        ok = mbar_wait(&bar_mma, mma_phase);
        mma_phase ^= 1;
        if (tid == 0) bulk_wait_read_all();   // Ut overwrites the state operand next
        if (__syncthreads_or(!ok)) { failed = true; break; }
        pending_mma = 0;
        tc_fence_after();
        if (tid == 0 && c + 1 < nct) issue_av(c + 1);   // [T; A T], V and the other coef buffer are free

        // ---- epi-B: Ut operand (key rows); O = Oi + Oa (query rows)
        float d2[TVH];
        if (r < 64) {
#pragma unroll
            for (int e = 0; e < E; ++e) cr[e] = we[e * 64 + r];
        }
        {
            float d2l[TVH];
            tmem_ld<TVH>(tmem_lane_addr(tP, warp, cofs), d2);
            tmem_ld<TVH>(tmem_lane_addr(tP, warp, TV + cofs), d2l);
            tmem_wait_ld();
#pragma unroll
            for (int i = 0; i < TVH; ++i) d2[i] += d2l[i];
        }
        if (r < 64) {
#pragma unroll
            for (int e = 0; e < E; ++e) {
                const float wv = cr[e];
                float u[TVH];
#pragma unroll
                for (int i = 0; i < TVH; ++i) u[i] = wv * d2[i];
#pragma unroll
                for (int i = 0; i < TVH; i += 8) st8_split(sUh, sUl, sw128_offset(r, e * TV + cofs + i, 64), u + i);
            }
        } else {
#pragma unroll
            for (int i = 0; i < TVH; ++i) d2[i] += oi[i];
            if (tma_o) {   // row of the o tile; thread 0 stores the tile after the barrier
                const int rq = r - 64;
                if (p.out_f32) store_f32_row(reinterpret_cast<float*>(sOo) + rq * TV + cofs, d2, TVH);
                else store_row(sOo, size_t(rq) * TV + cofs, d2, TVH, 0);
            }
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        tc_fence_after();

        // ---- MMA-C: S_all += K^T Ut   (A = K^T MN-major from the key rows; B = Ut MN-major)
        if (tid == 0) {
            const uint32_t idesc = idesc_bf16_f32(128, NE, 1, 1);
            const uint64_t a0 = smem_desc(smem_u32(sKQ), 2 * kBoxBytes, 1024);
            const uint64_t uh0 = smem_desc(smem_u32(sUh), 64 * 128, 1024);
            const uint64_t ul0 = smem_desc(smem_u32(sUl), 64 * 128, 1024);
#pragma unroll
            for (int ks = 0; ks < 4; ++ks) {
                const uint64_t ad = desc_add(a0, ks * 2048);
                umma_bf16(tS, ad, desc_add(uh0, ks * 2048), idesc, 1u);
                umma_bf16(tS, ad, desc_add(ul0, ks * 2048), idesc, 1u);
            }
            umma_commit(&bar_mma);
            if (tma_o) {   // rows past T are skipped by the store
                tma_store_4d(&map_o, sOo, n0, h, t0, b);
                bulk_commit();
            }
        }
        pending_mma = 1;
        {   // while MMA-C runs: U (key rows) and o (query rows) to global memory
            if (r < 64) {
                if (p.save) {
                    if (p.ck_tiles) store_tok_tile(p.Ubuf, (size_t(b) * H + h) * NT + cb + c, dv, r, n0 + cofs, d2, TVH, r < n);
                    else if (r < n) store_f32_row(p.Ubuf + tok_idx(b, t0 + r, h, n0 + cofs, T, H, dv), d2, TVH);
                }
            } else if (!tma_o && r - 64 < n) {
                store_row(p.o, tok_idx(b, t0 + r - 64, h, n0 + cofs, T, H, dv), d2, TVH, p.out_f32);
            }
        }
        ok = mbar_wait(&bar_mma, mma_phase);
        mma_phase ^= 1;
        if (c + 1 < nct) ok = ok && mbar_wait(&bar_av, (c + 1) & 1);   // chunk c+1's gamma^C
        if (__syncthreads_or(!ok)) { failed = true; break; }
        pending_mma = 0;
        tc_fence_after();
        if (tid == 0 && c + 1 < nct) issue_kq(c + 1);   // key/query buffer is free

        // ---- epi-C: next chunk's state operand, MMA-A(c+1) and its checkpoint, then the
        // gamma^C-scaled slab for MMA-C(c+1)
        if (c + 1 < nct) {
            stage_operand(c + 1);
            fence_proxy_async_smem();
            tc_fence_before();
            ok = mbar_wait(&bar_kq, (c + 1) & 1);
            if (__syncthreads_or(!ok)) { failed = true; break; }
            tc_fence_after();
            if (tid == 0) {
                issue_mma_a();
                issue_ckpt(c + 1);
            }
            pending_mma = 1;
            scale_state(c + 1);   // ordered before MMA-C(c+1) by the barriers in between
        } else if (p.ht) {
#pragma unroll
            for (int e0 = 0; e0 < E; e0 += GRP) {
                float v[GRP * TVH];
#pragma unroll
                for (int g = 0; g < GRP; ++g) tmem_ld<TVH>(tmem_lane_addr(tS, warp, (e0 + g) * TV + cofs), v + g * TVH);
                tmem_wait_ld();
#pragma unroll
                for (int g = 0; g < GRP; ++g)
                    if (r < p.dk)
                        store_f32_row(p.ht + ((size_t(sb * H + h) * E + e0 + g) * p.dk + r) * dv + n0 + cofs,
                                      v + g * TVH, TVH);
            }
        }
    }

    if (failed) {
        // Bounded drain of products still in flight, then leave (copies that never
        // complete expire with the same bound in the waits above).
        if (tid == 0) {
            record_device_error(p.err, TLA_ERR_TIMEOUT);
            if (pending_mma) mbar_wait(&bar_mma, mma_phase ^ 1);
        }
    }
    if (tid == 0) bulk_wait_all();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tmem_dealloc(tmem_slot, tcols);
}

template <int TV, int E>
cudaError_t launch_tv(const tla_problem& p, const FwdPlan& fp, char* ws, int save, int* err,
                      cudaStream_t s) {
    if (p.E != E || fp.tc_tv != TV) return cudaErrorInvalidValue;
    CUtensorMap mk, mq, mv, ma, mc, mo;
    const int NT = fp.NT;
    if (!make_token_map(&mk, p.k, p.B, p.T, p.H, p.dk, 64, 64, true) ||
        !make_token_map(&mq, p.q, p.B, p.T, p.H, p.dk, 64, 64, true) ||
        !make_token_map(&mv, p.v, p.B, p.T, p.H, p.dv, TV, 64, false) ||
        !make_matrix_map(&ma, ws + fp.A2, (long long)p.B * p.H * NT * 256, 64, 64, 128) ||
        !make_token_map(&mo, p.o, p.B, p.T, p.H, p.dv, TV, 64, false, p.out_dtype == TLA_FP32 ? 4 : 2))
        return cudaErrorInvalidValue;
    memset(&mc, 0, sizeof(mc));   // unused unless tile checkpoints are saved
    if (save && fp.ck_tiles &&
        !make_ckpt_map(&mc, ws + fp.S, (long long)p.B * p.H * NT * p.E, p.dv, TV, p.E, 2 * TV))
        return cudaErrorInvalidValue;
    TcFwdArgs a;
    a.coef = (const float*)(ws + fp.coef);
    a.h0 = p.h0;
    a.o = p.o;
    a.ht = p.ht;
    a.Sck = save ? (float*)(ws + fp.S) : nullptr;
    a.Ubuf = save ? (float*)(ws + fp.U) : nullptr;
    a.Rbuf = (save && (p.use_delta || fp.ck_tiles)) ? (float*)(ws + fp.Res) : nullptr;
    a.err = err;
    a.T = p.T; a.H = p.H; a.dv = p.dv; a.E = p.E; a.NT = NT;
    a.use_delta = p.use_delta; a.save = save; a.out_f32 = p.out_dtype == TLA_FP32;
    a.ck_tiles = fp.ck_tiles;
    a.dk = p.dk;
    a.dtab = p.cu_seqlens ? (const int4*)(ws + fp.dtab) : nullptr;
    const size_t smem = tc_fwd_smem_c<TV>(E);
    auto kern = fwd_recurrence_tc_kernel<TV, E>;
    cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    dim3 grid(p.dv / TV, p.H, fp.nseq);
    prof_before("fwd_recurrence_tc", s);
    kern<<<grid, kThreads, smem, s>>>(mk, mq, mv, ma, mc, mo, a);
    prof_after(s);
    return cudaGetLastError();
}

}  // namespace

// Value columns per CTA of the tensor-core recurrence (0: not eligible).  The
// state and Ut operands are MN-major with 64-column swizzle atoms, so E * TV must
// be a multiple of 64 (and at most 256, the widest UMMA and half of TMEM).
int tc_fwd_tv(const tla_problem& p) {
    // d_k = 64 runs as d_k = 128 with zero key rows: the key/query boxes past d_k are filled
    // with zeros by the copy engine, so the state's padded rows stay zero
    if (p.dtype != TLA_BF16 || (p.dk != kDk && p.dk != 64)) return 0;
    const int cand[3] = {16, 32, 64};
    for (int tv : cand) {
        const int ne = p.E * tv;
        if (p.dv % tv == 0 && ne % 64 == 0 && ne <= 256) return tv;
    }
    return 0;
}

cudaError_t launch_fwd_recurrence_tc(const tla_problem& p, const FwdPlan& fp, char* ws,
                                     int save_for_bwd, int* err, cudaStream_t s) {
    // one instance per slice count the tensor-core path takes (tc_fwd_tv)
    switch (p.E) {
        case 1: return launch_tv<64, 1>(p, fp, ws, save_for_bwd, err, s);
        case 2: return launch_tv<32, 2>(p, fp, ws, save_for_bwd, err, s);
        case 3: return launch_tv<64, 3>(p, fp, ws, save_for_bwd, err, s);
        case 4: return launch_tv<16, 4>(p, fp, ws, save_for_bwd, err, s);
        case 6: return launch_tv<32, 6>(p, fp, ws, save_for_bwd, err, s);
        case 8: return launch_tv<16, 8>(p, fp, ws, save_for_bwd, err, s);
        case 12: return launch_tv<16, 12>(p, fp, ws, save_for_bwd, err, s);
        case 16: return launch_tv<16, 16>(p, fp, ws, save_for_bwd, err, s);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace tla
