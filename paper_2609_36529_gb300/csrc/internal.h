// Host-side interfaces between the C ABI (tla_api.cu) and the kernel files.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>

#include <cuda_bf16.h>

#include "../../include/tla.h"

namespace tla {

// Byte offsets of the private buffers inside the caller's workspaces.
struct FwdPlan {
    int NT;              // chunks per sequence, ceil(T / 64); packed documents: all chunks
    int nseq;            // independent states: B, or the number of packed documents
    size_t ctab;         // packed documents: int2 [NT] (first token, rows) of every chunk
    size_t dtab;         // packed documents: int4 [n_docs] (first token, chunks, first chunk, tokens)
    int tv;              // value columns per CTA of the SIMT recurrence
    size_t G;            // fp32 [B,T,H,E] chunk-local inclusive log-decay
    size_t A;            // fp32 [B,H,NT,64,64] Q K^T (.) R' (lower incl. diagonal)
    size_t N;            // fp32 [B,H,NT,64,64] (I + L)^{-1} (delta rule only)
    size_t S;            // fp32 [B,H,NT,E,dk,dv] chunk-start states (save_for_bwd)
    size_t U;            // delta-corrected values (save_for_bwd): fp32 [B,T,H,dv], or token tiles
    size_t Res;          // residual V - W (save_for_bwd; delta rule, or any rule with token
                         // tiles, where sGLA stores V): fp32 [B,T,H,dv], or token tiles
    size_t A2;           // bf16 [B,H,NT,2,128,64] [T; A T] hi and lo tiles (tensor-core path)
    size_t coef;         // fp32 [B,H,NT,3*64*E+16] per-row coefficients (tensor-core path)
    size_t BT;           // bf16 [B,H,NT,4,64,64] A, T hi/lo row-major (tensor-core backward)
    int tcb;             // 1: the backward recurrence runs on tensor cores
    int ck_tiles;        // 1: state checkpoints (forward S, backward dS) are stored as bf16
                         //    hi/lo pairs: per (b,h,chunk,e) a row-major [dk][dv] hi matrix
                         //    then the lo matrix (same 4 bytes per element as fp32), written
                         //    and read by TMA (tma_host.h: make_ckpt_map); U, Res
                         //    and the backward's dU, -dRes are then token tiles: per
                         //    (b,h,chunk) 64 rows x dv bf16 hi then lo, SW128 K-major 64-row
                         //    blocks, rows past T zero; with d_k = 64 a checkpoint keeps 128
                         //    rows, the last 64 zero
    int tc_tv;           // value columns per CTA of the tensor-core recurrence (0: SIMT)
    int need_A;          // 1: the fp32 A matrices are read (a CUDA-core recurrence follows)
    size_t bytes;        // total
};

struct BwdPlan {
    int tv;
    size_t dU;           // fp32 [B,T,H,dv], or token tiles (FwdPlan::ck_tiles)
    size_t dRes;         // fp32 [B,T,H,dv] dRes, or token tiles of -dRes (delta rule)
    size_t dS;           // fp32 [B,H,NT,E,dk,dv] gradient of the state at each chunk's end
    size_t dgE;          // per-head gate: fp32 [B,T,H,E] per-slice gate gradient before the sum
    size_t gscr;         // tensor-core chunk gradients with E > 8: fp32 [B,H,NT,3,64,E] partials
    size_t bytes;
};

// Kernel timing hooks (active between tla_profile_begin / tla_profile_end).
void prof_before(const char* name, cudaStream_t s);
void prof_after(cudaStream_t s);

// Bracket one launch: PROF_LAUNCH("name", stream, kernel<<<...>>>(...));
#define PROF_LAUNCH(name, stream, ...)   \
    do {                                 \
        ::tla::prof_before(name, stream); \
        __VA_ARGS__;                     \
        ::tla::prof_after(stream);       \
    } while (0)

FwdPlan plan_fwd(const tla_problem& p, int save_for_bwd);
// Chunks of a problem: ceil(T / 64) per sequence, or the sum over packed documents.
int chunk_count(const tla_problem& p);
BwdPlan plan_bwd(const tla_problem& p);

// SIMT path (fp32 arithmetic on CUDA cores; any supported dtype).
cudaError_t launch_gate_cumsum(const tla_problem& p, const FwdPlan& fp, const char* ws, float* G,
                               cudaStream_t s);
cudaError_t launch_chunk_prep(const tla_problem& p, const float* G, float* A, float* N,
                              cudaStream_t s);
// Per-chunk preparation of the tensor-core path (A, N, [T; A T], [A; T], coefficients).
cudaError_t launch_chunk_prep_tc(const tla_problem& p, const FwdPlan& fp, char* ws, int* err,
                                 cudaStream_t s);
// Tensor-core chunk-parallel gradients (requires the tensor-core backward recurrence).
int tc_grads_ok(const tla_problem& p, const FwdPlan& fp);
int tc_grads_shape_ok(const tla_problem& p);
cudaError_t launch_bwd_chunk_grads_tc(const tla_problem& p, const FwdPlan& fp, const char* fws,
                                      const BwdPlan& bp, char* bws, const void* dO,
                                      void* dq, void* dk, void* dq2, void* dk2, float* dbeta,
                                      float* dg, int* err, cudaStream_t s);
// Tensor-core backward recurrence (requires the tensor-core forward layout).
int tc_bwd_ok(const tla_problem& p, int tv);
cudaError_t launch_bwd_recurrence_tc(const tla_problem& p, const FwdPlan& fp, const char* fws,
                                     const BwdPlan& bp, char* bws, const void* dO,
                                     const float* dht, void* dv, float* dh0, int* err,
                                     cudaStream_t s);

// Tensor-core path (bf16 inputs, dk = 128): value columns per CTA, or 0 if not eligible.
int tc_fwd_tv(const tla_problem& p);
cudaError_t launch_fwd_recurrence_tc(const tla_problem& p, const FwdPlan& fp, char* ws,
                                     int save_for_bwd, int* err, cudaStream_t s);
cudaError_t launch_fwd_recurrence(const tla_problem& p, const FwdPlan& fp, char* ws,
                                  int save_for_bwd, cudaStream_t s);
cudaError_t launch_bwd_recurrence(const tla_problem& p, const FwdPlan& fp, const char* fws,
                                  const BwdPlan& bp, char* bws, const void* dO,
                                  const float* dht, void* dv, float* dh0, cudaStream_t s);
cudaError_t launch_bwd_chunk_grads(const tla_problem& p, const FwdPlan& fp, const char* fws,
                                   const BwdPlan& bp, const char* bws, const void* dO,
                                   void* dq, void* dk, void* dq2, void* dk2, float* dbeta,
                                   float* dg, cudaStream_t s);

// dst[i] = sum_e src[i * E + e] (gradient of a per-head gate).
cudaError_t launch_sum_slices(const float* src, float* dst, long long n, int E, cudaStream_t s);

// Decode step.
cudaError_t launch_decode_step(int B, int H, int dk, int dv, int E, int use_delta, int dtype,
                               const void* q, const void* k, const void* v, const void* q2,
                               const void* k2, const float* g, const float* beta,
                               float* state, void* o, int* err, cudaStream_t s);

}  // namespace tla
