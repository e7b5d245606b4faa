"""Float64 CPU oracle for triadic linear attention.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
the ``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import
this package.  The product path (the CUDA library and its binding) never
imports it, and it never imports the product path.

Every function takes and returns float64 numpy arrays in the layouts of
``tla_oracle.c``:
  q, k [B,T,H,dk]; v, o [B,T,H,dv]; q2, k2, g [B,T,H,E]; beta [B,T,H];
  state [B,H,E,dk,dv].

Pins: see the header of ``tla_oracle.c``; every function here is pinned by a
``-m "not gpu"`` test (tests/test_oracle_*.py).
"""
import ctypes
import os

import numpy as np

from . import build as _build

_lib = None
_dp = ctypes.POINTER(ctypes.c_double)


def _load():
    global _lib
    if _lib is None:
        path = _build.build()
        lib = ctypes.CDLL(path)
        i = ctypes.c_int
        lib.tla_oracle_forward.argtypes = [i] * 7 + [_dp] * 10
        lib.tla_oracle_chunk_forward.argtypes = [i] * 8 + [_dp] * 10
        lib.tla_oracle_backward.argtypes = [i] * 7 + [_dp] * 18
        lib.tla_oracle_decode_step.argtypes = [i] * 6 + [_dp] * 9
        d = ctypes.c_double
        lib.tla_oracle_prologue.argtypes = [i] * 7 + [d] + [_dp] * 13
        lib.tla_oracle_prologue_backward.argtypes = [i] * 7 + [d] + [_dp] * 19
        lib.tla_oracle_gate_norm.argtypes = [i] * 4 + [d] + [_dp] * 4
        lib.tla_oracle_gate_norm_backward.argtypes = [i] * 4 + [d] + [_dp] * 7
        lib.tla_oracle_num_threads.restype = ctypes.c_int
        lib.tla_oracle_set_threads.argtypes = [i]
        _lib = lib
    return _lib


def _p(a):
    if a is None:
        return None
    assert a.dtype == np.float64 and a.flags["C_CONTIGUOUS"], "oracle wants C-contiguous float64"
    return a.ctypes.data_as(_dp)


def _f64(a):
    return None if a is None else np.ascontiguousarray(a, dtype=np.float64)


def num_threads() -> int:
    return _load().tla_oracle_num_threads()


def set_threads(n: int) -> None:
    _load().tla_oracle_set_threads(int(n))


def _dims(q, v, q2):
    B, T, H, dk = q.shape
    dv = v.shape[-1]
    E = q2.shape[-1]
    return B, T, H, dk, dv, E


def forward(q, k, v, q2, k2, g, beta=None, h0=None, use_delta=True):
    """Token-by-token recurrence (Eq. forget3 / Eq. gdn3, read per Eq. la3).

    Returns (o [B,T,H,dv], ht [B,H,E,dk,dv])."""
    q, k, v, q2, k2, g, beta, h0 = map(_f64, (q, k, v, q2, k2, g, beta, h0))
    B, T, H, dk, dv, E = _dims(q, v, q2)
    o = np.zeros((B, T, H, dv))
    ht = np.zeros((B, H, E, dk, dv))
    _load().tla_oracle_forward(B, T, H, dk, dv, E, int(bool(use_delta)), _p(q), _p(k), _p(v),
                               _p(q2), _p(k2), _p(g), _p(beta), _p(h0), _p(o), _p(ht))
    return o, ht


def chunk_forward(q, k, v, q2, k2, g, beta=None, h0=None, use_delta=True, chunk=64):
    """Chunkwise form of Appendix A (Eq. joint-gram, joint-solve, joint-chunk)."""
    q, k, v, q2, k2, g, beta, h0 = map(_f64, (q, k, v, q2, k2, g, beta, h0))
    B, T, H, dk, dv, E = _dims(q, v, q2)
    o = np.zeros((B, T, H, dv))
    ht = np.zeros((B, H, E, dk, dv))
    _load().tla_oracle_chunk_forward(B, T, H, dk, dv, E, int(bool(use_delta)), int(chunk),
                                     _p(q), _p(k), _p(v), _p(q2), _p(k2), _p(g), _p(beta),
                                     _p(h0), _p(o), _p(ht))
    return o, ht


def backward(q, k, v, q2, k2, g, dout, beta=None, h0=None, dht=None, use_delta=True):
    """Back-propagation through time of the token recurrence.

    Returns a dict with dq, dk, dv, dq2, dk2, dg and (when given) dbeta, dh0."""
    q, k, v, q2, k2, g, beta, h0, dout, dht = map(_f64, (q, k, v, q2, k2, g, beta, h0, dout, dht))
    B, T, H, dk, dv, E = _dims(q, v, q2)
    out = {n: np.zeros_like(a) for n, a in (("dq", q), ("dk", k), ("dv", v), ("dq2", q2),
                                           ("dk2", k2), ("dg", g))}
    out["dbeta"] = np.zeros((B, T, H)) if beta is not None else None
    out["dh0"] = np.zeros((B, H, E, dk, dv)) if h0 is not None else None
    _load().tla_oracle_backward(B, T, H, dk, dv, E, int(bool(use_delta)), _p(q), _p(k), _p(v),
                                _p(q2), _p(k2), _p(g), _p(beta), _p(h0), _p(dout), _p(dht),
                                _p(out["dq"]), _p(out["dk"]), _p(out["dv"]), _p(out["dq2"]),
                                _p(out["dk2"]), _p(out["dbeta"]), _p(out["dg"]), _p(out["dh0"]))
    return {n: a for n, a in out.items() if a is not None}


def decode_step(state, q, k, v, q2, k2, g, beta=None, use_delta=True):
    """One token of the recurrence for every (b,h); returns (o [B,H,dv], new state)."""
    q, k, v, q2, k2, g, beta = map(_f64, (q, k, v, q2, k2, g, beta))
    st = np.array(state, dtype=np.float64, order="C", copy=True)
    B, H, dk = q.shape
    dv = v.shape[-1]
    E = q2.shape[-1]
    o = np.zeros((B, H, dv))
    _load().tla_oracle_decode_step(B, H, dk, dv, E, int(bool(use_delta)), _p(q), _p(k), _p(v),
                                   _p(q2), _p(k2), _p(g), _p(beta), _p(st), _p(o))
    return o, st


def projection(u, W, H):
    """Input projection of Algorithm 2 / Appendix A (Input projections): one GEMM of the
    layer input u [B,T,Dm] with the weight W [H*C, Dm] (rows: head h's channels
    [q|k|v|q'|k'] at h*C..h*C+C-1), P[b,t,h,c] = sum_i u[b,t,i] W[h*C+c, i], in float64
    (the matrix product is the library primitive).  Returns P [B,T,H,C]."""
    u, W = _f64(u), _f64(W)
    B, T, Dm = u.shape
    C = W.shape[0] // H
    return (u.reshape(B * T, Dm) @ W.T).reshape(B, T, H, C)


def prologue(P, conv_w, gate_in, gate_bias, A_log, beta_in, dk, dv, E, eps=1e-6):
    """Layer input path of Algorithm 2: causal depthwise convolution of the projection
    output P [B,T,H,2dk+dv+2E] (per head [q|k|v|q'|k']) with conv_w [H,C,K], SiLU on
    q,k,v, softplus on q',k', L2 normalisation of q,k,q',k'; log gates
    -exp(A_log) softplus(gate_in + gate_bias) and beta = sigmoid(beta_in).
    Returns dict q, k, v, q2, k2, g, beta (beta None without beta_in)."""
    P, conv_w, gate_in, gate_bias, A_log, beta_in = map(
        _f64, (P, conv_w, gate_in, gate_bias, A_log, beta_in))
    B, T, H, C = P.shape
    K = conv_w.shape[-1]
    out = {"q": np.zeros((B, T, H, dk)), "k": np.zeros((B, T, H, dk)),
           "v": np.zeros((B, T, H, dv)), "q2": np.zeros((B, T, H, E)),
           "k2": np.zeros((B, T, H, E)), "g": np.zeros((B, T, H, E)),
           "beta": np.zeros((B, T, H)) if beta_in is not None else None}
    _load().tla_oracle_prologue(B, T, H, dk, dv, E, K, float(eps), _p(P), _p(conv_w),
                                _p(gate_in), _p(gate_bias), _p(A_log), _p(beta_in),
                                _p(out["q"]), _p(out["k"]), _p(out["v"]), _p(out["q2"]),
                                _p(out["k2"]), _p(out["g"]), _p(out["beta"]))
    return out


def prologue_backward(P, conv_w, gate_in, gate_bias, A_log, beta_in, grads, dk, dv, E,
                      eps=1e-6):
    """Gradients of prologue(): grads holds dq, dk, dv, dq2, dk2, dg (and dbeta).
    Returns dict dP, dconv_w, dgate_in, dgate_bias, dA_log (and dbeta_in)."""
    P, conv_w, gate_in, gate_bias, A_log, beta_in = map(
        _f64, (P, conv_w, gate_in, gate_bias, A_log, beta_in))
    gr = {n: _f64(grads.get(n)) for n in ("dq", "dk", "dv", "dq2", "dk2", "dg", "dbeta")}
    B, T, H, C = P.shape
    K = conv_w.shape[-1]
    out = {"dP": np.zeros_like(P), "dconv_w": np.zeros_like(conv_w),
           "dgate_in": np.zeros_like(gate_in), "dgate_bias": np.zeros_like(gate_bias),
           "dA_log": np.zeros_like(A_log),
           "dbeta_in": np.zeros_like(beta_in) if beta_in is not None else None}
    _load().tla_oracle_prologue_backward(
        B, T, H, dk, dv, E, K, float(eps), _p(P), _p(conv_w), _p(gate_in), _p(gate_bias),
        _p(A_log), _p(beta_in), _p(gr["dq"]), _p(gr["dk"]), _p(gr["dv"]), _p(gr["dq2"]),
        _p(gr["dk2"]), _p(gr["dg"]), _p(gr["dbeta"]), _p(out["dP"]), _p(out["dconv_w"]),
        _p(out["dgate_in"]), _p(out["dgate_bias"]), _p(out["dA_log"]), _p(out["dbeta_in"]))
    return {n: a for n, a in out.items() if a is not None}


def gate_norm(o, z, w_norm, eps=1e-6):
    """Output gate of Algorithm 2: RMSNorm(o) (weight w_norm [dv]) times sigmoid(z)."""
    o, z, w_norm = map(_f64, (o, z, w_norm))
    B, T, H, dv = o.shape
    y = np.zeros_like(o)
    _load().tla_oracle_gate_norm(B, T, H, dv, float(eps), _p(o), _p(z), _p(w_norm), _p(y))
    return y


def gate_norm_backward(o, z, w_norm, dy, eps=1e-6):
    """Gradients of gate_norm(): returns dict do, dz, dw_norm."""
    o, z, w_norm, dy = map(_f64, (o, z, w_norm, dy))
    B, T, H, dv = o.shape
    out = {"do": np.zeros_like(o), "dz": np.zeros_like(o), "dw_norm": np.zeros_like(w_norm)}
    _load().tla_oracle_gate_norm_backward(B, T, H, dv, float(eps), _p(o), _p(z), _p(w_norm),
                                          _p(dy), _p(out["do"]), _p(out["dz"]), _p(out["dw_norm"]))
    return out
