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
