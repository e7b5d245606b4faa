/*
 * tla.h - C ABI of the GB300 (sm_103a) triadic linear attention library.
 *
 * Triadic linear attention (arXiv 2609.36529) keeps, per head, a third-order
 * state S in R^{E x dk x dv} (slice e = S[:, e, :] of the paper's d x E x d
 * tensor, stored here as [E][dk][dv]).  Each token
 *   1. decays every slice by its own forget gate alpha_{t,e}     (Section 2.4, Eq. forget3)
 *   2. with the joint-key delta rule, erases the value read at the joint key
 *      k (x) k', scaled by beta_t: u = beta (v - S x1 k x2 k')   (Section 2.4, Eq. gdn3)
 *      without it ("sGLA"): u = beta v                           (Algorithm 2)
 *   3. writes k (x) k' (x) u                                     (Section 2.2, Eq. la3)
 *   4. reads o = S x1 q x2 q' after the write                   (Section 2.2, Eq. la3)
 * tla_chunk_fwd / tla_chunk_bwd compute this for whole sequences with the
 * chunkwise-parallel form of Appendix A (Eq. joint-gram, joint-solve,
 * joint-chunk); tla_decode_step advances the recurrence by one token.
 *
 * Conventions shared by every entry point
 *  - Every pointer is a DEVICE pointer (cudaMalloc / PyTorch CUDA memory) unless
 *    stated otherwise; the caller owns every buffer, including workspaces.
 *    The library allocates no device memory.
 *  - All tensors are dense, row-major, contiguous.  Token tensors use the
 *    layout [B, T, H, D]; states use [B, H, E, dk, dv].  Every pointer must be
 *    16-byte aligned (PyTorch and cudaMalloc allocations are); an unaligned
 *    pointer is rejected with TLA_ERR_INVALID_ARG.
 *  - `dtype` (tla_dtype) is the element type of q, k, v, q2, k2; `out_dtype`
 *    that of o and of their gradients.  Log-gates g, beta, states h0/ht/dh0,
 *    dg and dbeta are fp32.  Arithmetic accumulates in fp32 throughout.
 *  - q, k, q2, k2 are expected to be L2-normalised by the caller (Algorithm 2
 *    normalises them before the operator); no 1/sqrt(d) scale is applied.
 *    g holds log alpha <= 0 (log of the per-slice forget gate).
 *  - `stream` is a cudaStream_t passed as void*; NULL means the legacy default
 *    stream.  Calls only enqueue work: they never synchronise the device.
 *  - Argument errors are detected on the host before anything is launched and
 *    return a negative status; nothing is written in that case.  Launch errors,
 *    and a failed lookup of the device error word below, return TLA_ERR_CUDA.
 *    Device-side bounded waits that expire record an error word that
 *    tla_last_device_status() reports (TLA_ERR_TIMEOUT).
 *  - Results are deterministic: no floating-point atomics (Appendix A, Kernels).
 */
#ifndef TLA_H
#define TLA_H

#include <stddef.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    TLA_OK = 0,
    TLA_ERR_INVALID_ARG = -1,  /* bad pointer, size, alignment or combination */
    TLA_ERR_UNSUPPORTED = -2,  /* valid request outside the supported shapes   */
    TLA_ERR_CUDA = -3,         /* a CUDA launch or runtime call failed          */
    TLA_ERR_TIMEOUT = -4,      /* a device-side bounded wait expired            */
    TLA_ERR_WORKSPACE = -5     /* workspace missing or smaller than required    */
} tla_status;

typedef enum { TLA_BF16 = 0, TLA_FP32 = 1 } tla_dtype;

/*
 * One chunkwise problem: B sequences of T tokens, H heads.
 * Supported: 1 <= dk, dv <= 128 with dk, dv multiples of 16; 1 <= E <= 32, with
 * dk <= 64 when E > 16 (the paper's E = 16/32 variants use d_k = 32/64);
 * chunk == 64 (the paper's C, Appendix A); T >= 1 (a last partial chunk is
 * allowed); B*H <= 65535.
 */
typedef struct {
    int B, T, H;
    int dk, dv, E;
    int chunk;           /* must be 64                                         */
    int dtype;           /* tla_dtype of q, k, v, q2, k2                       */
    int out_dtype;       /* tla_dtype of o (forward) and of dq, dk, dv, dq2,
                            dk2 (backward).  TLA_FP32 keeps the fp32
                            accumulation of bf16 inputs; TLA_BF16 rounds.      */
    int use_delta;       /* 1: triadic Gated DeltaNet (Eq. gdn3); 0: sGLA      */
    const void *q;       /* [B,T,H,dk]                                          */
    const void *k;       /* [B,T,H,dk]                                          */
    const void *v;       /* [B,T,H,dv]                                          */
    const void *q2;      /* [B,T,H,E]  second query q'                          */
    const void *k2;      /* [B,T,H,E]  second key k'                            */
    const float *g;      /* [B,T,H,E]  log forget gates, <= 0                   */
    const float *beta;   /* [B,T,H] write strength in (0,1); NULL => 1.
                            Required when use_delta == 1.                       */
    const float *h0;     /* [B,H,E,dk,dv] initial state; NULL => zero state     */
    void *o;             /* [B,T,H,dv] out_dtype output (written)               */
    float *ht;           /* [B,H,E,dk,dv] final state (written); may be NULL    */
    /* Packed documents (Appendix A, Kernels: variable-length sequences packed
     * into one batch, each evolved from its own initial state).  NULL: B
     * independent sequences of T tokens.  Otherwise a HOST array of n_docs + 1
     * token offsets, cu_seqlens[0] = 0 <= cu_seqlens[i] <= cu_seqlens[i+1],
     * cu_seqlens[n_docs] = T, with B = 1: document i is tokens
     * [cu_seqlens[i], cu_seqlens[i+1]) of the single sequence, its chunks start
     * at its first token (the last one may be partial; empty documents are
     * allowed), and h0, ht, dht and dh0 are [n_docs,H,E,dk,dv].  The library
     * copies a chunk table built from it into the forward workspace (a
     * cudaMemcpyAsync from pageable host memory on the call's stream), so the
     * backward reads it from there.  Packed documents run on the tensor-core
     * path only (bf16 inputs, dk = 128, dv a multiple of 64, E <= 8, save or
     * not); other shapes return TLA_ERR_UNSUPPORTED.                        */
    const int *cu_seqlens;
    int n_docs;
    /* 1: one scalar log forget gate per head and token, shared by all E slices
     * (the per-head gate variant): g is [B,T,H] and the backward's dg is
     * [B,T,H].  0: g and dg are [B,T,H,E].                                   */
    int gate_per_head;
} tla_problem;

/*
 * Workspace of tla_chunk_fwd in bytes (a multiple of 256; the workspace pointer
 * must be 256-byte aligned).  With save_for_bwd != 0 the workspace also keeps
 * what tla_chunk_bwd needs (chunk-start states, delta-corrected values, the
 * per-chunk UT-transform matrices); it must then stay untouched until the
 * matching tla_chunk_bwd has run.  Returns 0 for an invalid problem.
 */
size_t tla_fwd_workspace_bytes(const tla_problem *p, int save_for_bwd);

/*
 * Chunkwise-parallel forward (Appendix A, Eq. joint-chunk): writes p->o and,
 * when non-NULL, p->ht.  Steps: per-slice chunk-local cumulative log decay;
 * per chunk R, R' (Eq. joint-gram), A = QK^T (.) R' and the UT transform
 * T (Eq. joint-solve); then the recurrence over chunks carrying the state.
 */
tla_status tla_chunk_fwd(const tla_problem *p, void *workspace, size_t workspace_bytes,
                         int save_for_bwd, void *stream);

/*
 * Forward without a caller-provided workspace, for callers that cannot allocate
 * device memory (a host runtime that owns all device memory, a serving process
 * that forbids allocation after start-up, a fixed committed memory budget).
 * The paper has no counterpart: this is an interface convenience.  Same
 * computation and outputs as tla_chunk_fwd(p, ws, bytes, save_for_bwd = 0, stream),
 * with the workspace taken from a fixed device buffer built into the library
 * (tla_noalloc_scratch_bytes() bytes, 64 MiB, held by every GPU that loads the
 * library until the process exits).  Allocates nothing.
 *  - Returns TLA_ERR_WORKSPACE, launching nothing, when
 *    tla_fwd_workspace_bytes(p, 0) exceeds the buffer; other argument errors
 *    as tla_chunk_fwd.
 *  - All calls share the buffer: calls that overlap on the GPU (other streams,
 *    unordered host threads) race on it.  Nothing in it needs clearing.
 *  - The first call on each device looks up the buffer's device address; make
 *    it before capturing the stream into a CUDA graph.
 */
tla_status tla_chunk_fwd_noalloc(const tla_problem *p, void *stream);

/* Size in bytes of the built-in buffer used by tla_chunk_fwd_noalloc. */
size_t tla_noalloc_scratch_bytes(void);

/* Workspace of tla_chunk_bwd in bytes (multiple of 256, 256-byte aligned). */
size_t tla_bwd_workspace_bytes(const tla_problem *p);

/*
 * Backward of tla_chunk_fwd (Appendix A, Kernels: a reverse recurrence over
 * chunks producing each chunk's state gradient, then every chunk's remaining
 * gradients in parallel, reduced in a fixed order).
 *   fwd_ws  workspace of a tla_chunk_fwd(p, ..., save_for_bwd=1) call on the
 *           same problem and inputs (read only).
 *   dO      [B,T,H,dv] dtype (the input dtype), gradient of o.
 *   dht     [B,H,E,dk,dv] fp32 gradient of ht, or NULL (=> 0).
 *   dq, dk  [B,T,H,dk];  dv [B,T,H,dv];  dq2, dk2 [B,T,H,E]: all out_dtype.
 *   dbeta   [B,T,H] fp32; required iff p->beta != NULL, else must be NULL.
 *   dg      [B,T,H,E] fp32 gradient of the log-gates ([B,T,H] with gate_per_head).
 *   dh0     [B,H,E,dk,dv] fp32; required iff p->h0 != NULL, else must be NULL.
 */
tla_status tla_chunk_bwd(const tla_problem *p, const void *fwd_ws, size_t fwd_ws_bytes,
                         const void *dO, const float *dht,
                         void *dq, void *dk, void *dv, void *dq2, void *dk2,
                         float *dbeta, float *dg, float *dh0,
                         void *workspace, size_t workspace_bytes, void *stream);

/*
 * One recurrent decode step for B sequences (Algorithm 2, one iteration; Eq.
 * forget3 then Eq. gdn3 or the sGLA write, then the read of Eq. la3):
 *   q, k [B,H,dk] dtype; v [B,H,dv] dtype; q2, k2 [B,H,E] dtype;
 *   g [B,H,E] fp32; beta [B,H] fp32 or NULL (=> 1; required if use_delta);
 *   state [B,H,E,dk,dv] fp32, updated in place; o [B,H,dv] dtype (written).
 * Supported: dk, dv multiples of 16 up to 128, 1 <= E <= 32 with E*dk <= 2048,
 * B*H <= 65535.  A per-head gate is passed as E equal values of g.
 * No workspace.  Each (b, h, 16 value columns) slab of the state is read once
 * and written once (through shared memory by TMA when E*dk <= 1024 and is a
 * multiple of 64); a bounded wait on that copy that expires records
 * TLA_ERR_TIMEOUT for tla_last_device_status().
 */
tla_status tla_decode_step(int B, int H, int dk, int dv, int E, int use_delta, int dtype,
                           const void *q, const void *k, const void *v,
                           const void *q2, const void *k2, const float *g,
                           const float *beta, float *state, void *o, void *stream);

/* Human-readable name of a status code (static string). */
const char *tla_status_string(int status);

/*
 * Layer input path of Algorithm 2 (Appendix A, Input projections): from the
 * output P of the one projection GEMM to the operator's inputs.  The GEMMs
 * themselves (W u for P, W_alpha u, W_beta u) are plain GEMMs of the caller.
 * Per (b, t, h), with C = 2 dk + dv + 2 E channels per head ordered
 * [q | k | v | q' | k']:
 *   a_c(t) = sum_{j<K} conv_w[h,c,j] P_c(t - K + 1 + j)   (causal depthwise
 *            convolution of width K; P before token 0 is zero)
 *   q = n(silu(a_q)), k = n(silu(a_k)), v = silu(a_v),
 *   q' = n(softplus(a_q')), k' = n(softplus(a_k')), n(x) = x / sqrt(|x|^2 + eps)
 *   g = log alpha = -exp(A_log) softplus(gate_in + gate_bias),  beta = sigmoid(beta_in)
 * All pointers 16-byte aligned; sizes as stated; outputs are written.
 */
typedef struct {
    int B, T, H, dk, dv, E;
    int K;               /* convolution width, 1..4                              */
    int dtype;           /* tla_dtype of P and of q, k, v, q2, k2                */
    float eps;           /* L2-normalisation epsilon                             */
    const void *P;       /* [B,T,H,C] projection output                          */
    const float *conv_w; /* [H,C,K]                                              */
    const float *gate_in;   /* [B,T,H,E]  W_alpha u                              */
    const float *gate_bias; /* [H,E]                                             */
    const float *A_log;     /* [H,E]                                             */
    const float *beta_in;   /* [B,T,H]  W_beta u, or NULL (then beta is NULL)    */
    void *q, *k, *v, *q2, *k2;   /* [B,T,H,dk|dk|dv|E|E] dtype                  */
    float *g;            /* [B,T,H,E]                                            */
    float *beta;         /* [B,T,H], NULL iff beta_in is NULL                    */
} tla_prologue_args;

/* Forward of the input path.  Supported: dk, dv multiples of 16 up to 128,
 * 1 <= E <= 32, 1 <= K <= 4, B*H <= 65535. */
tla_status tla_layer_prologue(const tla_prologue_args *a, void *stream);

/* Workspace of tla_layer_prologue_bwd in bytes (per-segment partial sums). */
size_t tla_layer_prologue_bwd_workspace_bytes(const tla_prologue_args *a);

/*
 * Backward of the input path.  grad_dtype is the tla_dtype of dq, dk, dv, dq2,
 * dk2 (what tla_chunk_bwd produced); dg [B,T,H,E] and dbeta [B,T,H] are fp32
 * (dbeta NULL iff beta_in NULL).  Writes dP [B,T,H,C] (dtype), dconv_w [H,C,K],
 * dgate_in [B,T,H,E], dgate_bias [H,E], dA_log [H,E] and dbeta_in [B,T,H] (fp32).
 * The sums over tokens are taken in a fixed order (deterministic).
 */
tla_status tla_layer_prologue_bwd(const tla_prologue_args *a, int grad_dtype, const void *dq,
                                  const void *dk, const void *dv, const void *dq2,
                                  const void *dk2, const float *dg, const float *dbeta,
                                  void *dP, float *dconv_w, float *dgate_in, float *dgate_bias,
                                  float *dA_log, float *dbeta_in, void *workspace,
                                  size_t workspace_bytes, void *stream);

/*
 * Input projection of Algorithm 2 fused with the input path above (Appendix A, Input
 * projections: one GEMM produces q, k, v, k', q' of every head, then one causal depthwise
 * convolution processes them).  From the normalised layer input u:
 *   P[b,t,h,c] = sum_i u[b,t,i] W[h*C + c, i]      (C = 2 dk + dv + 2 E, [q | k | v | q' | k'])
 * on the tensor cores, then in the same kernel, per (b, t, h), the prologue of
 * tla_layer_prologue on P (convolution of width K, SiLU / softplus, L2 normalisation, log
 * gates from gate_in, beta from beta_in).  P is written only when P != NULL (the backward
 * of the input path, tla_layer_prologue_bwd, takes it).
 * Supported: dk, dv in {64, 128}, 1 <= E <= 16, 1 <= K <= 4, Dm a multiple of 64,
 * bf16 u, W and outputs; all pointers 16-byte aligned.
 */
typedef struct {
    int B, T, H, dk, dv, E;
    int K;               /* convolution width, 1..4                                  */
    int Dm;              /* model width (the GEMM's K dimension)                      */
    float eps;           /* L2-normalisation epsilon                                  */
    const void *u;       /* [B,T,Dm] bf16 layer input                                 */
    const void *W;       /* [H*C, Dm] bf16 projection weight (output channel major)   */
    const float *conv_w; /* [H,C,K]                                                   */
    const float *gate_in;   /* [B,T,H,E]  W_alpha u                                   */
    const float *gate_bias; /* [H,E]                                                  */
    const float *A_log;     /* [H,E]                                                  */
    const float *beta_in;   /* [B,T,H]  W_beta u, or NULL (then beta is NULL)         */
    void *q, *k, *v, *q2, *k2;   /* [B,T,H,dk|dk|dv|E|E] bf16 (written)                */
    float *g;            /* [B,T,H,E] (written)                                       */
    float *beta;         /* [B,T,H] (written), NULL iff beta_in is NULL               */
    void *P;             /* [B,T,H,C] bf16 projection output (written), or NULL       */
} tla_projection_args;

tla_status tla_layer_projection(const tla_projection_args *a, void *stream);

/*
 * Output gate of Algorithm 2: per (b, t, h) over dv channels
 *   y = o / sqrt(mean(o^2) + eps) * w_norm * sigmoid(z).
 */
typedef struct {
    int B, T, H, dv;
    int o_dtype;         /* tla_dtype of o (the operator's output)               */
    int dtype;           /* tla_dtype of z and y                                 */
    float eps;
    const void *o;       /* [B,T,H,dv]                                           */
    const void *z;       /* [B,T,H,dv]  gate pre-activation (W_g2 W_g1 u + b_g)   */
    const float *w_norm; /* [dv]                                                 */
    void *y;             /* [B,T,H,dv] (written)                                 */
} tla_gate_args;

/* Forward of the output gate (dv a multiple of 16 up to 128). */
tla_status tla_output_gate(const tla_gate_args *a, void *stream);

/* Workspace of tla_output_gate_bwd in bytes. */
size_t tla_output_gate_bwd_workspace_bytes(const tla_gate_args *a);

/* Backward: dy [B,T,H,dv] (dtype) -> d_o (o_dtype), dz (dtype), dw_norm [dv]
 * fp32 (fixed-order sums). */
tla_status tla_output_gate_bwd(const tla_gate_args *a, const void *dy, void *d_o, void *dz,
                               float *dw_norm, void *workspace, size_t workspace_bytes,
                               void *stream);

/*
 * Synchronises `stream`, then returns TLA_ERR_TIMEOUT if a device-side bounded
 * wait of any kernel launched since the previous call expired (and clears that
 * record), TLA_ERR_CUDA if the stream reports an error, else TLA_OK.
 * The record is ONE word per device, shared by every stream and host thread
 * that uses the library on that device: only `stream` is synchronised, so a
 * timeout in a kernel still running on another stream may be reported by a
 * later call, and a timeout on another stream is reported (and cleared) by
 * whichever call reads the word first.  Callers with several streams should
 * synchronise all of them before reading the status.
 */
tla_status tla_last_device_status(void *stream);

/*
 * Self-test of the failure-detection path.  Launches one CTA whose threads wait on
 * an mbarrier that nothing ever arrives at, with the same bounded wait the
 * tensor-core kernels use but a limit of `timeout_ns` nanoseconds of GPU global
 * time (1 .. 10^9).  The wait expires, the CTA records TLA_ERR_TIMEOUT in the
 * device error word and returns, so the next tla_last_device_status() reports
 * TLA_ERR_TIMEOUT and the context stays usable.  Returns TLA_ERR_INVALID_ARG for a
 * limit outside the range, else the launch status.
 */
tla_status tla_selftest_bounded_wait(unsigned long long timeout_ns, void *stream);

/*
 * Kernel timing (tracing).  After tla_profile_begin(), every kernel the library
 * launches is bracketed by CUDA events recorded on its launch stream (event
 * objects are created on first use and reused; no device memory is allocated).
 * tla_profile_end() synchronises `stream`, stops recording and reports, per
 * kernel name in first-launch order, the number of launches and the summed
 * device time in milliseconds.  It returns the number of distinct kernels
 * written (at most max_kernels), or a negative status.  names_out receives
 * max_kernels fixed-size slots of 64 bytes (NUL-terminated names).
 */
tla_status tla_profile_begin(void);
int tla_profile_end(void *stream, char *names_out, int *launches_out, float *ms_out,
                    int max_kernels);

/* Library version string, e.g. "tla 0.1 sm_103a". */
const char *tla_version(void);

#ifdef __cplusplus
}
#endif

#endif /* TLA_H */
