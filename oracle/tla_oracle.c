/*
 * Float64 CPU oracle for triadic linear attention (test infrastructure).
 *
 * This file is NOT part of the product path.  Only the test-suite, the smoke
 * check and the benchmark's CPU-baseline leg load it.  It shares no code,
 * header, table or helper with the CUDA library: it is a plain, slow,
 * deliberately obvious restatement of the paper's equations.
 *
 * Paper: "Triadic Linear Attention: Three-Dimensional Recurrent States for
 * Long-Context Sequence Modeling" (arXiv 2609.36529).
 *
 * Layouts (all row-major, contiguous):
 *   q, k        [B, T, H, dk]
 *   v, o        [B, T, H, dv]
 *   q2, k2, g   [B, T, H, E]     (q2/k2 are the paper's q', k'; g = log alpha <= 0)
 *   beta        [B, T, H]        (NULL => beta == 1)
 *   state       [B, H, E, dk, dv] (slice e of the paper's d x E x d tensor S)
 *
 * Pins (checked by tests/test_oracle_*.py, see the test files):
 *   token forward      pinned (E=1 textbook GDN / gated LA, materialised
 *                      attention sum, flattened joint-key GDN, closed form at
 *                      T=1, delta-rule and capacity invariants)
 *   token backward     pinned (central finite differences; autograd of an
 *                      independently written flattened form)
 *   chunk forward      pinned (agrees with the token recurrence, including
 *                      extreme within-chunk decay)
 *   decode step        pinned (one token of the pinned token recurrence)
 *   layer prologue     pinned (torch F.conv1d / F.silu / F.softplus restatement,
 *   and output gate     its autograd for the backward, causality, unit norms)
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define IDX_TOK(b, t, h, i, T, H, D) ((((size_t)(b) * (T) + (t)) * (H) + (h)) * (D) + (i))

int tla_oracle_num_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

void tla_oracle_set_threads(int n) {
#ifdef _OPENMP
    if (n > 0) omp_set_num_threads(n);
#else
    (void)n;
#endif
}

/* ------------------------------------------------------------------------ */
/* One token of the recurrence for one head.                                 */
/*                                                                           */
/* Section 2.4, Eq. (forget3) and Eq. (gdn3), in the order of Algorithm 2:   */
/*   1. decay every slice by its own gate:  S_e <- alpha_e S_e               */
/*   2. (delta rule) read what the joint key k (x) k' currently stores:      */
/*        r = S x_1 k x_2 k' = sum_e k'_e S_e^T k,  u = beta (v - r)         */
/*      (no delta rule, "sGLA"):  u = beta v   (Algorithm 2, write k (x) beta k' (x) v) */
/*   3. write the triadic outer product:  S_e <- S_e + k'_e k u^T            */
/*   4. read after the write (Eq. la3):  o = S x_1 q x_2 q' = sum_e q'_e S_e^T q */
/* S is [E][dk][dv].  r_out / u_out (dv each) may be NULL.                   */
/* ------------------------------------------------------------------------ */
static void token_step(int dk, int dv, int E, int use_delta,
                       const double *q, const double *k, const double *v,
                       const double *q2, const double *k2, const double *g,
                       double beta, double *S, double *o,
                       double *r_out, double *u_out, double *tmp /* dv */) {
    /* 1. per-slice decay */
    for (int e = 0; e < E; ++e) {
        double a = exp(g[e]);
        double *Se = S + (size_t)e * dk * dv;
        for (int i = 0; i < dk * dv; ++i) Se[i] *= a;
    }
    /* 2. erase read and delta-corrected value */
    double *u = tmp;
    for (int j = 0; j < dv; ++j) u[j] = 0.0;
    if (use_delta) {
        for (int e = 0; e < E; ++e) {
            const double *Se = S + (size_t)e * dk * dv;
            for (int i = 0; i < dk; ++i) {
                double c = k2[e] * k[i];
                for (int j = 0; j < dv; ++j) u[j] += c * Se[(size_t)i * dv + j];
            }
        }
    }
    for (int j = 0; j < dv; ++j) {
        double r = u[j];
        if (r_out) r_out[j] = r;
        u[j] = use_delta ? beta * (v[j] - r) : beta * v[j];
        if (u_out) u_out[j] = u[j];
    }
    /* 3. write k (x) k' (x) u */
    for (int e = 0; e < E; ++e) {
        double *Se = S + (size_t)e * dk * dv;
        for (int i = 0; i < dk; ++i) {
            double c = k2[e] * k[i];
            for (int j = 0; j < dv; ++j) Se[(size_t)i * dv + j] += c * u[j];
        }
    }
    /* 4. read with both queries */
    for (int j = 0; j < dv; ++j) o[j] = 0.0;
    for (int e = 0; e < E; ++e) {
        const double *Se = S + (size_t)e * dk * dv;
        for (int i = 0; i < dk; ++i) {
            double c = q2[e] * q[i];
            for (int j = 0; j < dv; ++j) o[j] += c * Se[(size_t)i * dv + j];
        }
    }
}

/* Gather one token's vectors of head (b,h) from the [B,T,H,*] arrays. */
typedef struct {
    const double *q, *k, *v, *q2, *k2, *g;
    double beta;
} tok_view;

static tok_view view_tok(const double *q, const double *k, const double *v,
                         const double *q2, const double *k2, const double *g,
                         const double *beta, int b, int t, int h,
                         int T, int H, int dk, int dv, int E) {
    tok_view tv;
    tv.q = q + IDX_TOK(b, t, h, 0, T, H, dk);
    tv.k = k + IDX_TOK(b, t, h, 0, T, H, dk);
    tv.v = v + IDX_TOK(b, t, h, 0, T, H, dv);
    tv.q2 = q2 + IDX_TOK(b, t, h, 0, T, H, E);
    tv.k2 = k2 + IDX_TOK(b, t, h, 0, T, H, E);
    tv.g = g + IDX_TOK(b, t, h, 0, T, H, E);
    tv.beta = beta ? beta[((size_t)b * T + t) * H + h] : 1.0;
    return tv;
}

/* ------------------------------------------------------------------------ */
/* Token-by-token forward (Eq. forget3 + Eq. gdn3, read per Eq. la3).         */
/* h0 may be NULL (zero state); ht may be NULL.                              */
/* ------------------------------------------------------------------------ */
void tla_oracle_forward(int B, int T, int H, int dk, int dv, int E, int use_delta,
                        const double *q, const double *k, const double *v,
                        const double *q2, const double *k2, const double *g,
                        const double *beta, const double *h0,
                        double *o, double *ht) {
    const size_t ssz = (size_t)E * dk * dv;
#pragma omp parallel for schedule(dynamic, 1)
    for (int bh = 0; bh < B * H; ++bh) {
        int b = bh / H, h = bh % H;
        double *S = (double *)malloc(ssz * sizeof(double));
        double *tmp = (double *)malloc((size_t)dv * sizeof(double));
        if (h0) memcpy(S, h0 + (size_t)bh * ssz, ssz * sizeof(double));
        else memset(S, 0, ssz * sizeof(double));
        for (int t = 0; t < T; ++t) {
            tok_view tv = view_tok(q, k, v, q2, k2, g, beta, b, t, h, T, H, dk, dv, E);
            token_step(dk, dv, E, use_delta, tv.q, tv.k, tv.v, tv.q2, tv.k2, tv.g,
                       tv.beta, S, o + IDX_TOK(b, t, h, 0, T, H, dv), NULL, NULL, tmp);
        }
        if (ht) memcpy(ht + (size_t)bh * ssz, S, ssz * sizeof(double));
        free(S);
        free(tmp);
    }
}

/* ------------------------------------------------------------------------ */
/* Single-token decode step: exactly one step of the token recurrence above  */
/* for every (b,h), updating state in place.                                  */
/*   q,k [B,H,dk]; v,o [B,H,dv]; q2,k2,g [B,H,E]; beta [B,H] or NULL          */
/* ------------------------------------------------------------------------ */
void tla_oracle_decode_step(int B, int H, int dk, int dv, int E, int use_delta,
                            const double *q, const double *k, const double *v,
                            const double *q2, const double *k2, const double *g,
                            const double *beta, double *state, double *o) {
    const size_t ssz = (size_t)E * dk * dv;
#pragma omp parallel for schedule(dynamic, 1)
    for (int bh = 0; bh < B * H; ++bh) {
        double *tmp = (double *)malloc((size_t)dv * sizeof(double));
        token_step(dk, dv, E, use_delta, q + (size_t)bh * dk, k + (size_t)bh * dk,
                   v + (size_t)bh * dv, q2 + (size_t)bh * E, k2 + (size_t)bh * E,
                   g + (size_t)bh * E, beta ? beta[bh] : 1.0,
                   state + (size_t)bh * ssz, o + (size_t)bh * dv, NULL, NULL, tmp);
        free(tmp);
    }
}

/* ------------------------------------------------------------------------ */
/* Backward of the token recurrence (hand-derived back-propagation through    */
/* time of token_step).  Given do [B,T,H,dv] and dht (NULL => 0), writes      */
/* dq, dk, dv_, dq2, dk2, dg (all required), dbeta (required iff beta given)  */
/* and dh0 (required iff h0 given).                                           */
/*                                                                            */
/* Reverse of one step, with S the post-write state and Shat = alpha (.) S_prev: */
/*   o  = sum_e q'_e S_e^T q        : dS_e += q'_e q do^T,                    */
/*                                    dq = sum_e q'_e S_e do, dq'_e = q^T S_e do */
/*   S_e = Shat_e + k'_e k u^T      : du = sum_e k'_e dS_e^T k,               */
/*                                    dk = sum_e k'_e dS_e u, dk'_e = k^T dS_e u, */
/*                                    dShat_e = dS_e                           */
/*   delta: u = beta (v - r), r = sum_e k'_e Shat_e^T k                       */
/*          dv = beta du, dbeta = du . (v - r), dr = -beta du,                */
/*          dShat_e += k'_e k dr^T, dk += sum_e k'_e Shat_e dr,               */
/*          dk'_e += k^T Shat_e dr                                            */
/*   no delta: u = beta v : dv = beta du, dbeta = du . v                      */
/*   Shat_e = alpha_e S_prev_e      : dg_e = <dShat_e, Shat_e>_F,             */
/*                                    dS_prev_e = alpha_e dShat_e             */
/* States are recomputed per segment of SEG tokens from float64 checkpoints.  */
/* ------------------------------------------------------------------------ */
#define SEG 64

void tla_oracle_backward(int B, int T, int H, int dk, int dv, int E, int use_delta,
                         const double *q, const double *k, const double *v,
                         const double *q2, const double *k2, const double *g,
                         const double *beta, const double *h0,
                         const double *dout, const double *dht,
                         double *dq, double *dk_, double *dv_, double *dq2,
                         double *dk2, double *dbeta, double *dg, double *dh0) {
    const size_t ssz = (size_t)E * dk * dv;
    const int nseg = (T + SEG - 1) / SEG;
#pragma omp parallel for schedule(dynamic, 1)
    for (int bh = 0; bh < B * H; ++bh) {
        int b = bh / H, h = bh % H;
        double *ck = (double *)malloc((size_t)(nseg > 0 ? nseg : 1) * ssz * sizeof(double));
        double *Sprev = (double *)malloc((size_t)SEG * ssz * sizeof(double));
        double *rseg = (double *)malloc((size_t)SEG * dv * sizeof(double));
        double *useg = (double *)malloc((size_t)SEG * dv * sizeof(double));
        double *S = (double *)malloc(ssz * sizeof(double));
        double *Shat = (double *)malloc(ssz * sizeof(double));
        double *Spost = (double *)malloc(ssz * sizeof(double));
        double *dS = (double *)malloc(ssz * sizeof(double));
        double *tmp = (double *)malloc((size_t)dv * 4 * sizeof(double));
        double *otmp = tmp + dv, *du = tmp + 2 * dv, *dr = tmp + 3 * dv;

        /* forward pass storing the state at the start of every segment */
        if (h0) memcpy(S, h0 + (size_t)bh * ssz, ssz * sizeof(double));
        else memset(S, 0, ssz * sizeof(double));
        for (int t = 0; t < T; ++t) {
            if (t % SEG == 0) memcpy(ck + (size_t)(t / SEG) * ssz, S, ssz * sizeof(double));
            tok_view tv = view_tok(q, k, v, q2, k2, g, beta, b, t, h, T, H, dk, dv, E);
            token_step(dk, dv, E, use_delta, tv.q, tv.k, tv.v, tv.q2, tv.k2, tv.g,
                       tv.beta, S, otmp, NULL, NULL, tmp);
        }

        if (dht) memcpy(dS, dht + (size_t)bh * ssz, ssz * sizeof(double));
        else memset(dS, 0, ssz * sizeof(double));

        for (int sgi = nseg - 1; sgi >= 0; --sgi) {
            int t0 = sgi * SEG, t1 = t0 + SEG < T ? t0 + SEG : T;
            /* recompute the segment, keeping S_prev, r and u of every token */
            memcpy(S, ck + (size_t)sgi * ssz, ssz * sizeof(double));
            for (int t = t0; t < t1; ++t) {
                memcpy(Sprev + (size_t)(t - t0) * ssz, S, ssz * sizeof(double));
                tok_view tv = view_tok(q, k, v, q2, k2, g, beta, b, t, h, T, H, dk, dv, E);
                token_step(dk, dv, E, use_delta, tv.q, tv.k, tv.v, tv.q2, tv.k2, tv.g,
                           tv.beta, S, otmp, rseg + (size_t)(t - t0) * dv,
                           useg + (size_t)(t - t0) * dv, tmp);
            }
            for (int t = t1 - 1; t >= t0; --t) {
                tok_view tv = view_tok(q, k, v, q2, k2, g, beta, b, t, h, T, H, dk, dv, E);
                const double *sp = Sprev + (size_t)(t - t0) * ssz;
                const double *u = useg + (size_t)(t - t0) * dv;
                const double *r = rseg + (size_t)(t - t0) * dv;
                const double *dov = dout + IDX_TOK(b, t, h, 0, T, H, dv);
                double *dqv = dq + IDX_TOK(b, t, h, 0, T, H, dk);
                double *dkv = dk_ + IDX_TOK(b, t, h, 0, T, H, dk);
                double *dvv = dv_ + IDX_TOK(b, t, h, 0, T, H, dv);
                double *dq2v = dq2 + IDX_TOK(b, t, h, 0, T, H, E);
                double *dk2v = dk2 + IDX_TOK(b, t, h, 0, T, H, E);
                double *dgv = dg + IDX_TOK(b, t, h, 0, T, H, E);
                /* Shat and post-write S */
                for (int e = 0; e < E; ++e) {
                    double a = exp(tv.g[e]);
                    for (int i = 0; i < dk; ++i)
                        for (int j = 0; j < dv; ++j) {
                            size_t x = ((size_t)e * dk + i) * dv + j;
                            Shat[x] = a * sp[x];
                            Spost[x] = Shat[x] + tv.k2[e] * tv.k[i] * u[j];
                        }
                }
                /* read: o = sum_e q'_e S_e^T q */
                for (int i = 0; i < dk; ++i) dqv[i] = 0.0;
                for (int e = 0; e < E; ++e) {
                    double acc_e = 0.0;
                    for (int i = 0; i < dk; ++i) {
                        double s = 0.0;
                        for (int j = 0; j < dv; ++j) s += Spost[((size_t)e * dk + i) * dv + j] * dov[j];
                        dqv[i] += tv.q2[e] * s;
                        acc_e += tv.q[i] * s;
                    }
                    dq2v[e] = acc_e;
                }
                for (int e = 0; e < E; ++e)
                    for (int i = 0; i < dk; ++i) {
                        double c = tv.q2[e] * tv.q[i];
                        for (int j = 0; j < dv; ++j) dS[((size_t)e * dk + i) * dv + j] += c * dov[j];
                    }
                /* write: S_e = Shat_e + k'_e k u^T */
                for (int j = 0; j < dv; ++j) du[j] = 0.0;
                for (int i = 0; i < dk; ++i) dkv[i] = 0.0;
                for (int e = 0; e < E; ++e) {
                    double acc_e = 0.0;
                    for (int i = 0; i < dk; ++i) {
                        double s = 0.0;
                        for (int j = 0; j < dv; ++j) {
                            double d = dS[((size_t)e * dk + i) * dv + j];
                            du[j] += tv.k2[e] * tv.k[i] * d;
                            s += d * u[j];
                        }
                        dkv[i] += tv.k2[e] * s;
                        acc_e += tv.k[i] * s;
                    }
                    dk2v[e] = acc_e;
                }
                double db = 0.0;
                if (use_delta) {
                    for (int j = 0; j < dv; ++j) {
                        dvv[j] = tv.beta * du[j];
                        db += du[j] * (tv.v[j] - r[j]);
                        dr[j] = -tv.beta * du[j];
                    }
                    for (int e = 0; e < E; ++e) {
                        double acc_e = 0.0;
                        for (int i = 0; i < dk; ++i) {
                            double s = 0.0;
                            double c = tv.k2[e] * tv.k[i];
                            for (int j = 0; j < dv; ++j) {
                                size_t x = ((size_t)e * dk + i) * dv + j;
                                s += Shat[x] * dr[j];
                                dS[x] += c * dr[j]; /* dS now holds dShat */
                            }
                            dkv[i] += tv.k2[e] * s;
                            acc_e += tv.k[i] * s;
                        }
                        dk2v[e] += acc_e;
                    }
                } else {
                    for (int j = 0; j < dv; ++j) {
                        dvv[j] = tv.beta * du[j];
                        db += du[j] * tv.v[j];
                    }
                }
                if (dbeta) dbeta[((size_t)b * T + t) * H + h] = db;
                /* decay: Shat_e = alpha_e S_prev_e */
                for (int e = 0; e < E; ++e) {
                    double a = exp(tv.g[e]);
                    double s = 0.0;
                    for (size_t x = (size_t)e * dk * dv; x < (size_t)(e + 1) * dk * dv; ++x) {
                        s += dS[x] * Shat[x];
                        dS[x] *= a;
                    }
                    dgv[e] = s;
                }
            }
        }
        if (dh0) memcpy(dh0 + (size_t)bh * ssz, dS, ssz * sizeof(double));
        free(ck); free(Sprev); free(rseg); free(useg); free(S); free(Shat);
        free(Spost); free(dS); free(tmp);
    }
}

/* ------------------------------------------------------------------------ */
/* Chunkwise form (Appendix A, Eq. joint-gram, Eq. joint-solve,               */
/* Eq. joint-chunk), written out with explicit matrices for one head at a      */
/* time.  C positions per chunk; the last chunk may be shorter.  Used by the   */
/* tests to pin the chunk equations against the token recurrence.             */
/*                                                                            */
/*   G_{r,e}     = sum_{j<=r} log alpha_{j,e}  (chunk-local, inclusive)       */
/*   Gamma_e(r,s)= exp(G_{r,e} - G_{s,e}) for r >= s, else 0                  */
/*   R  = sum_e (k'_e k'_e^T) (.) Gamma_e,  R' = sum_e (q'_e k'_e^T) (.) Gamma_e */
/*   T  = (I + tril(diag(beta)(K K^T (.) R), -1))^{-1} diag(beta)   (delta)   */
/*   T  = diag(beta)                                                 (sGLA)   */
/*   U  = T (V - sum_e diag(k'_e (.) gamma_e) K S_e)   (sGLA: U = T V)         */
/*   O  = sum_e diag(q'_e (.) gamma_e) Q S_e + (Q K^T (.) R') U               */
/*   S_e <- gamma^C_e S_e + K^T diag(k'_e (.) gamma^C_e / gamma_e) U          */
/* Every decay factor is exp of a non-positive difference of log sums.         */
/* ------------------------------------------------------------------------ */
void tla_oracle_chunk_forward(int B, int T, int H, int dk, int dv, int E, int use_delta,
                              int C, const double *q, const double *k, const double *v,
                              const double *q2, const double *k2, const double *g,
                              const double *beta, const double *h0,
                              double *o, double *ht) {
    const size_t ssz = (size_t)E * dk * dv;
#pragma omp parallel for schedule(dynamic, 1)
    for (int bh = 0; bh < B * H; ++bh) {
        int b = bh / H, h = bh % H;
        double *S = (double *)malloc(ssz * sizeof(double));
        double *G = (double *)malloc((size_t)C * E * sizeof(double));
        double *R = (double *)malloc((size_t)C * C * sizeof(double));
        double *Rq = (double *)malloc((size_t)C * C * sizeof(double));
        double *L = (double *)malloc((size_t)C * C * sizeof(double));
        double *Tm = (double *)malloc((size_t)C * C * sizeof(double));
        double *Res = (double *)malloc((size_t)C * dv * sizeof(double));
        double *U = (double *)malloc((size_t)C * dv * sizeof(double));
        double *bt = (double *)malloc((size_t)C * sizeof(double));
        if (h0) memcpy(S, h0 + (size_t)bh * ssz, ssz * sizeof(double));
        else memset(S, 0, ssz * sizeof(double));
        for (int c0 = 0; c0 < T; c0 += C) {
            int n = T - c0 < C ? T - c0 : C;
#define KR(r, i) k[IDX_TOK(b, c0 + (r), h, (i), T, H, dk)]
#define QR(r, i) q[IDX_TOK(b, c0 + (r), h, (i), T, H, dk)]
#define VR(r, j) v[IDX_TOK(b, c0 + (r), h, (j), T, H, dv)]
#define K2(r, e) k2[IDX_TOK(b, c0 + (r), h, (e), T, H, E)]
#define Q2(r, e) q2[IDX_TOK(b, c0 + (r), h, (e), T, H, E)]
            for (int e = 0; e < E; ++e) {
                double acc = 0.0;
                for (int r = 0; r < n; ++r) {
                    acc += g[IDX_TOK(b, c0 + r, h, e, T, H, E)];
                    G[r * E + e] = acc;
                }
            }
            for (int r = 0; r < n; ++r) bt[r] = beta ? beta[((size_t)b * T + c0 + r) * H + h] : 1.0;
            /* R, R' element by element (Eq. joint-gram) */
            for (int r = 0; r < n; ++r)
                for (int s = 0; s < n; ++s) {
                    double a = 0.0, aq = 0.0;
                    if (r >= s)
                        for (int e = 0; e < E; ++e) {
                            double gam = exp(G[r * E + e] - G[s * E + e]);
                            a += K2(r, e) * K2(s, e) * gam;
                            aq += Q2(r, e) * K2(s, e) * gam;
                        }
                    R[r * C + s] = a;
                    Rq[r * C + s] = aq;
                }
            /* T (Eq. joint-solve) by forward substitution of (I + L) X = diag(beta) */
            for (int r = 0; r < n; ++r)
                for (int s = 0; s < n; ++s) {
                    double x = 0.0;
                    if (use_delta && r > s) {
                        double kk = 0.0;
                        for (int i = 0; i < dk; ++i) kk += KR(r, i) * KR(s, i);
                        x = bt[r] * kk * R[r * C + s];
                    }
                    L[r * C + s] = x;
                }
            for (int s = 0; s < n; ++s)
                for (int r = 0; r < n; ++r) {
                    double x = (r == s) ? bt[s] : 0.0;
                    if (use_delta)
                        for (int j = 0; j < r; ++j) x -= L[r * C + j] * Tm[j * C + s];
                    Tm[r * C + s] = x;
                }
            /* residual V - sum_e diag(k'_e gamma_e) K S_e  (delta rule only) */
            for (int r = 0; r < n; ++r)
                for (int j = 0; j < dv; ++j) {
                    double w = 0.0;
                    if (use_delta)
                        for (int e = 0; e < E; ++e) {
                            double a = K2(r, e) * exp(G[r * E + e]);
                            const double *Se = S + (size_t)e * dk * dv;
                            double s = 0.0;
                            for (int i = 0; i < dk; ++i) s += KR(r, i) * Se[(size_t)i * dv + j];
                            w += a * s;
                        }
                    Res[r * dv + j] = VR(r, j) - w;
                }
            /* U = T Res */
            for (int r = 0; r < n; ++r)
                for (int j = 0; j < dv; ++j) {
                    double s = 0.0;
                    for (int x = 0; x < n; ++x) s += Tm[r * C + x] * Res[x * dv + j];
                    U[r * dv + j] = s;
                }
            /* O */
            for (int r = 0; r < n; ++r)
                for (int j = 0; j < dv; ++j) {
                    double acc = 0.0;
                    for (int e = 0; e < E; ++e) {
                        double a = Q2(r, e) * exp(G[r * E + e]);
                        const double *Se = S + (size_t)e * dk * dv;
                        double s = 0.0;
                        for (int i = 0; i < dk; ++i) s += QR(r, i) * Se[(size_t)i * dv + j];
                        acc += a * s;
                    }
                    for (int s = 0; s <= r; ++s) {
                        double qk = 0.0;
                        for (int i = 0; i < dk; ++i) qk += QR(r, i) * KR(s, i);
                        acc += qk * Rq[r * C + s] * U[s * dv + j];
                    }
                    o[IDX_TOK(b, c0 + r, h, j, T, H, dv)] = acc;
                }
            /* state update */
            for (int e = 0; e < E; ++e) {
                double gC = G[(n - 1) * E + e];
                double dec = exp(gC);
                double *Se = S + (size_t)e * dk * dv;
                for (int i = 0; i < dk; ++i)
                    for (int j = 0; j < dv; ++j) {
                        double s = 0.0;
                        for (int r = 0; r < n; ++r)
                            s += KR(r, i) * K2(r, e) * exp(gC - G[r * E + e]) * U[r * dv + j];
                        Se[(size_t)i * dv + j] = dec * Se[(size_t)i * dv + j] + s;
                    }
            }
#undef KR
#undef QR
#undef VR
#undef K2
#undef Q2
        }
        if (ht) memcpy(ht + (size_t)bh * ssz, S, ssz * sizeof(double));
        free(S); free(G); free(R); free(Rq); free(L); free(Tm); free(Res); free(U); free(bt);
    }
}

/* ------------------------------------------------------------------------
 * Layer input path and output gate of Algorithm 2 (and the input-projection
 * paragraph of Appendix A): what surrounds the operator in a triadic layer.
 *
 * Input prologue, per (b, t, h), with C = 2 dk + dv + 2 E channels per head in
 * the order [q | k | v | q' | k'] of the projection output P [B,T,H,C]:
 *   a_c(t) = sum_{j<K} w[h,c,j] P_c(t - K + 1 + j)      causal depthwise conv
 *            (P before the first token is zero)
 *   q = n(silu(a_q)), k = n(silu(a_k)), v = silu(a_v),
 *   q' = n(softplus(a_q')), k' = n(softplus(a_k')),
 *   n(x) = x / sqrt(sum x^2 + eps)                       (L2 normalisation)
 *   g_e = log alpha_e = -exp(A_log[h,e]) softplus(gate_in_e + gate_bias[h,e])
 *   beta = sigmoid(beta_in)
 * Output gate, per (b, t, h) over the dv channels:
 *   y = o / sqrt(mean(o^2) + eps) * w_norm * sigmoid(z)
 * The backward functions are the hand-derived chains of these definitions.
 * ---------------------------------------------------------------------- */
static double o_sigmoid(double x) { return 1.0 / (1.0 + exp(-x)); }
static double o_softplus(double x) { return x > 30.0 ? x : log1p(exp(x)); }

/* Pre-activation a[C] of one token of one head (causal depthwise convolution). */
static void conv_token(const double *P, const double *w, int T, int H, int C, int K,
                       int b, int t, int h, double *a) {
    for (int c = 0; c < C; ++c) {
        double acc = 0.0;
        for (int j = 0; j < K; ++j) {
            const int ts = t - K + 1 + j;
            if (ts >= 0) acc += w[((size_t)h * C + c) * K + j] * P[IDX_TOK(b, ts, h, c, T, H, C)];
        }
        a[c] = acc;
    }
}

void tla_oracle_prologue(int B, int T, int H, int dk, int dv, int E, int K, double eps,
                         const double *P, const double *w, const double *gate_in,
                         const double *gate_bias, const double *A_log, const double *beta_in,
                         double *q, double *k, double *v, double *q2, double *k2, double *g,
                         double *beta) {
    const int C = 2 * dk + dv + 2 * E;
#pragma omp parallel for collapse(2) schedule(static)
    for (int b = 0; b < B; ++b)
        for (int t = 0; t < T; ++t) {
            double *a = (double *)malloc(sizeof(double) * C);
            for (int h = 0; h < H; ++h) {
                conv_token(P, w, T, H, C, K, b, t, h, a);
                /* groups: offset, width, activation (0 silu, 1 softplus), normalised, output */
                const int off[5] = {0, dk, 2 * dk, 2 * dk + dv, 2 * dk + dv + E};
                const int wid[5] = {dk, dk, dv, E, E};
                const int act[5] = {0, 0, 0, 1, 1};
                const int nrm[5] = {1, 1, 0, 1, 1};
                double *dst[5] = {q, k, v, q2, k2};
                for (int gi = 0; gi < 5; ++gi) {
                    double ss = 0.0;
                    for (int i = 0; i < wid[gi]; ++i) {
                        const double x = a[off[gi] + i];
                        const double y = act[gi] ? o_softplus(x) : x * o_sigmoid(x);
                        a[off[gi] + i] = y;
                        ss += y * y;
                    }
                    const double scale = nrm[gi] ? 1.0 / sqrt(ss + eps) : 1.0;
                    for (int i = 0; i < wid[gi]; ++i)
                        dst[gi][IDX_TOK(b, t, h, i, T, H, wid[gi])] = a[off[gi] + i] * scale;
                }
                for (int e = 0; e < E; ++e) {
                    const size_t i = IDX_TOK(b, t, h, e, T, H, E);
                    g[i] = -exp(A_log[h * E + e]) * o_softplus(gate_in[i] + gate_bias[h * E + e]);
                }
                if (beta_in) {
                    const size_t i = ((size_t)b * T + t) * H + h;
                    beta[i] = o_sigmoid(beta_in[i]);
                }
            }
            free(a);
        }
}

void tla_oracle_prologue_backward(int B, int T, int H, int dk, int dv, int E, int K, double eps,
                                  const double *P, const double *w, const double *gate_in,
                                  const double *gate_bias, const double *A_log,
                                  const double *beta_in, const double *dq, const double *dk_,
                                  const double *dv_, const double *dq2, const double *dk2,
                                  const double *dg, const double *dbeta, double *dP, double *dw,
                                  double *dgate_in, double *dgate_bias, double *dA_log,
                                  double *dbeta_in) {
    const int C = 2 * dk + dv + 2 * E;
    double *da = (double *)calloc((size_t)B * T * H * C, sizeof(double));
#pragma omp parallel for collapse(2) schedule(static)
    for (int b = 0; b < B; ++b)
        for (int t = 0; t < T; ++t) {
            double *a = (double *)malloc(sizeof(double) * C);
            double *y = (double *)malloc(sizeof(double) * C);
            for (int h = 0; h < H; ++h) {
                conv_token(P, w, T, H, C, K, b, t, h, a);
                const int off[5] = {0, dk, 2 * dk, 2 * dk + dv, 2 * dk + dv + E};
                const int wid[5] = {dk, dk, dv, E, E};
                const int act[5] = {0, 0, 0, 1, 1};
                const int nrm[5] = {1, 1, 0, 1, 1};
                const double *gy[5] = {dq, dk_, dv_, dq2, dk2};
                for (int gi = 0; gi < 5; ++gi) {
                    double ss = 0.0;
                    for (int i = 0; i < wid[gi]; ++i) {
                        const double x = a[off[gi] + i];
                        y[off[gi] + i] = act[gi] ? o_softplus(x) : x * o_sigmoid(x);
                        ss += y[off[gi] + i] * y[off[gi] + i];
                    }
                    const double n = nrm[gi] ? sqrt(ss + eps) : 1.0;
                    /* d(x/n)/dx: (dy - u (u.dy)) / n with u = x/n; identity without the norm */
                    double udy = 0.0;
                    for (int i = 0; i < wid[gi]; ++i)
                        udy += (y[off[gi] + i] / n) * gy[gi][IDX_TOK(b, t, h, i, T, H, wid[gi])];
                    for (int i = 0; i < wid[gi]; ++i) {
                        const double u = y[off[gi] + i] / n;
                        const double dyi = gy[gi][IDX_TOK(b, t, h, i, T, H, wid[gi])];
                        const double dx = nrm[gi] ? (dyi - u * udy) / n : dyi;
                        const double x = a[off[gi] + i], s = o_sigmoid(x);
                        const double dact = act[gi] ? s : s * (1.0 + x * (1.0 - s));
                        da[IDX_TOK(b, t, h, off[gi] + i, T, H, C)] = dx * dact;
                    }
                }
                for (int e = 0; e < E; ++e) {
                    const size_t i = IDX_TOK(b, t, h, e, T, H, E);
                    const double z = gate_in[i] + gate_bias[h * E + e];
                    dgate_in[i] = dg[i] * (-exp(A_log[h * E + e])) * o_sigmoid(z);
                }
                if (beta_in) {
                    const size_t i = ((size_t)b * T + t) * H + h;
                    const double s = o_sigmoid(beta_in[i]);
                    dbeta_in[i] = dbeta[i] * s * (1.0 - s);
                }
            }
            free(a);
            free(y);
        }
    /* transposed convolution and the weight correlation */
#pragma omp parallel for collapse(2) schedule(static)
    for (int b = 0; b < B; ++b)
        for (int t = 0; t < T; ++t)
            for (int h = 0; h < H; ++h)
                for (int c = 0; c < C; ++c) {
                    double acc = 0.0;
                    for (int j = 0; j < K; ++j) {
                        const int td = t + K - 1 - j;
                        if (td < T) acc += w[((size_t)h * C + c) * K + j] * da[IDX_TOK(b, td, h, c, T, H, C)];
                    }
                    dP[IDX_TOK(b, t, h, c, T, H, C)] = acc;
                }
#pragma omp parallel for collapse(2) schedule(static)
    for (int h = 0; h < H; ++h)
        for (int c = 0; c < C; ++c)
            for (int j = 0; j < K; ++j) {
                double acc = 0.0;
                for (int b = 0; b < B; ++b)
                    for (int t = 0; t < T; ++t) {
                        const int ts = t - K + 1 + j;
                        if (ts >= 0) acc += da[IDX_TOK(b, t, h, c, T, H, C)] * P[IDX_TOK(b, ts, h, c, T, H, C)];
                    }
                dw[((size_t)h * C + c) * K + j] = acc;
            }
    for (int h = 0; h < H; ++h)
        for (int e = 0; e < E; ++e) {
            double sb = 0.0, sa = 0.0;
            for (int b = 0; b < B; ++b)
                for (int t = 0; t < T; ++t) {
                    const size_t i = IDX_TOK(b, t, h, e, T, H, E);
                    const double z = gate_in[i] + gate_bias[h * E + e];
                    sb += dgate_in[i];
                    sa += dg[i] * (-exp(A_log[h * E + e]) * o_softplus(z));   /* dg * g */
                }
            dgate_bias[h * E + e] = sb;
            dA_log[h * E + e] = sa;
        }
    free(da);
}

void tla_oracle_gate_norm(int B, int T, int H, int dv, double eps, const double *o,
                          const double *z, const double *wn, double *y) {
#pragma omp parallel for collapse(2) schedule(static)
    for (int b = 0; b < B; ++b)
        for (int t = 0; t < T; ++t)
            for (int h = 0; h < H; ++h) {
                double ss = 0.0;
                for (int i = 0; i < dv; ++i) {
                    const double x = o[IDX_TOK(b, t, h, i, T, H, dv)];
                    ss += x * x;
                }
                const double r = 1.0 / sqrt(ss / dv + eps);
                for (int i = 0; i < dv; ++i) {
                    const size_t j = IDX_TOK(b, t, h, i, T, H, dv);
                    y[j] = o[j] * r * wn[i] * o_sigmoid(z[j]);
                }
            }
}

void tla_oracle_gate_norm_backward(int B, int T, int H, int dv, double eps, const double *o,
                                   const double *z, const double *wn, const double *dy,
                                   double *d_o, double *dz, double *dwn) {
    memset(dwn, 0, sizeof(double) * dv);
    for (int b = 0; b < B; ++b)
        for (int t = 0; t < T; ++t)
            for (int h = 0; h < H; ++h) {
                double ss = 0.0;
                for (int i = 0; i < dv; ++i) {
                    const double x = o[IDX_TOK(b, t, h, i, T, H, dv)];
                    ss += x * x;
                }
                const double r = 1.0 / sqrt(ss / dv + eps);
                double dot = 0.0;   /* sum_i dnh_i nh_i */
                for (int i = 0; i < dv; ++i) {
                    const size_t j = IDX_TOK(b, t, h, i, T, H, dv);
                    const double nh = o[j] * r, s = o_sigmoid(z[j]);
                    const double dnh = dy[j] * wn[i] * s;
                    dz[j] = dy[j] * nh * wn[i] * s * (1.0 - s);
                    dwn[i] += dy[j] * nh * s;
                    dot += dnh * nh;
                }
                for (int i = 0; i < dv; ++i) {
                    const size_t j = IDX_TOK(b, t, h, i, T, H, dv);
                    const double nh = o[j] * r, s = o_sigmoid(z[j]);
                    const double dnh = dy[j] * wn[i] * s;
                    d_o[j] = r * (dnh - nh * dot / dv);
                }
            }
}
