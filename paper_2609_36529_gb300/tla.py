"""Thin ctypes binding of ``libtla.so`` (C ABI in include/tla.h).

Argument marshalling only: every step of the path runs in the library's CUDA
kernels.  Tensors must be contiguous CUDA tensors; outputs and workspaces are
allocated with PyTorch (the library itself allocates nothing).  Calls are
enqueued on the current PyTorch CUDA stream.  If the library is missing the
first call raises: there is no fallback.
"""
import ctypes
import os
from typing import Optional

import torch

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libtla.so")

TLA_BF16, TLA_FP32 = 0, 1
STATUS = {0: "TLA_OK", -1: "TLA_ERR_INVALID_ARG", -2: "TLA_ERR_UNSUPPORTED", -3: "TLA_ERR_CUDA",
          -4: "TLA_ERR_TIMEOUT", -5: "TLA_ERR_WORKSPACE"}

EXPORTED = ("tla_fwd_workspace_bytes", "tla_chunk_fwd", "tla_bwd_workspace_bytes",
            "tla_chunk_bwd", "tla_decode_step", "tla_status_string", "tla_last_device_status",
            "tla_version", "tla_chunk_fwd_noalloc", "tla_noalloc_scratch_bytes",
            "tla_layer_prologue", "tla_layer_prologue_bwd_workspace_bytes",
            "tla_layer_prologue_bwd", "tla_output_gate", "tla_output_gate_bwd_workspace_bytes",
            "tla_output_gate_bwd", "tla_selftest_bounded_wait", "tla_layer_projection")


class TlaError(RuntimeError):
    def __init__(self, fn, status):
        super().__init__(f"{fn} failed: {STATUS.get(status, status)}")
        self.status = status


class tla_problem(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int), ("T", ctypes.c_int), ("H", ctypes.c_int),
                ("dk", ctypes.c_int), ("dv", ctypes.c_int), ("E", ctypes.c_int),
                ("chunk", ctypes.c_int), ("dtype", ctypes.c_int), ("out_dtype", ctypes.c_int),
                ("use_delta", ctypes.c_int),
                ("q", ctypes.c_void_p), ("k", ctypes.c_void_p), ("v", ctypes.c_void_p),
                ("q2", ctypes.c_void_p), ("k2", ctypes.c_void_p), ("g", ctypes.c_void_p),
                ("beta", ctypes.c_void_p), ("h0", ctypes.c_void_p), ("o", ctypes.c_void_p),
                ("ht", ctypes.c_void_p), ("cu_seqlens", ctypes.POINTER(ctypes.c_int)),
                ("n_docs", ctypes.c_int), ("gate_per_head", ctypes.c_int)]


class tla_prologue_args(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int), ("T", ctypes.c_int), ("H", ctypes.c_int),
                ("dk", ctypes.c_int), ("dv", ctypes.c_int), ("E", ctypes.c_int),
                ("K", ctypes.c_int), ("dtype", ctypes.c_int), ("eps", ctypes.c_float),
                ("P", ctypes.c_void_p), ("conv_w", ctypes.c_void_p), ("gate_in", ctypes.c_void_p),
                ("gate_bias", ctypes.c_void_p), ("A_log", ctypes.c_void_p),
                ("beta_in", ctypes.c_void_p), ("q", ctypes.c_void_p), ("k", ctypes.c_void_p),
                ("v", ctypes.c_void_p), ("q2", ctypes.c_void_p), ("k2", ctypes.c_void_p),
                ("g", ctypes.c_void_p), ("beta", ctypes.c_void_p)]


class tla_projection_args(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int), ("T", ctypes.c_int), ("H", ctypes.c_int),
                ("dk", ctypes.c_int), ("dv", ctypes.c_int), ("E", ctypes.c_int),
                ("K", ctypes.c_int), ("Dm", ctypes.c_int), ("eps", ctypes.c_float),
                ("u", ctypes.c_void_p), ("W", ctypes.c_void_p), ("conv_w", ctypes.c_void_p),
                ("gate_in", ctypes.c_void_p), ("gate_bias", ctypes.c_void_p),
                ("A_log", ctypes.c_void_p), ("beta_in", ctypes.c_void_p),
                ("q", ctypes.c_void_p), ("k", ctypes.c_void_p), ("v", ctypes.c_void_p),
                ("q2", ctypes.c_void_p), ("k2", ctypes.c_void_p), ("g", ctypes.c_void_p),
                ("beta", ctypes.c_void_p), ("P", ctypes.c_void_p)]


class tla_gate_args(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int), ("T", ctypes.c_int), ("H", ctypes.c_int),
                ("dv", ctypes.c_int), ("o_dtype", ctypes.c_int), ("dtype", ctypes.c_int),
                ("eps", ctypes.c_float), ("o", ctypes.c_void_p), ("z", ctypes.c_void_p),
                ("w_norm", ctypes.c_void_p), ("y", ctypes.c_void_p)]


_lib = None


def lib():
    """Load libtla.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"CUDA library not built: {LIB_PATH} (run __graft_entry__.build())")
        L = ctypes.CDLL(LIB_PATH)
        P = ctypes.POINTER(tla_problem)
        vp, i, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t
        L.tla_fwd_workspace_bytes.argtypes = [P, i]
        L.tla_fwd_workspace_bytes.restype = sz
        L.tla_bwd_workspace_bytes.argtypes = [P]
        L.tla_bwd_workspace_bytes.restype = sz
        L.tla_chunk_fwd.argtypes = [P, vp, sz, i, vp]
        L.tla_chunk_fwd.restype = i
        L.tla_chunk_bwd.argtypes = [P, vp, sz, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp]
        L.tla_chunk_bwd.restype = i
        L.tla_decode_step.argtypes = [i] * 7 + [vp] * 10
        L.tla_decode_step.restype = i
        L.tla_status_string.argtypes = [i]
        L.tla_status_string.restype = ctypes.c_char_p
        L.tla_last_device_status.argtypes = [vp]
        L.tla_last_device_status.restype = i
        L.tla_selftest_bounded_wait.argtypes = [ctypes.c_ulonglong, vp]
        L.tla_selftest_bounded_wait.restype = i
        L.tla_version.restype = ctypes.c_char_p
        L.tla_chunk_fwd_noalloc.argtypes = [P, vp]
        L.tla_chunk_fwd_noalloc.restype = i
        L.tla_noalloc_scratch_bytes.restype = sz
        PA, GA = ctypes.POINTER(tla_prologue_args), ctypes.POINTER(tla_gate_args)
        L.tla_layer_prologue.argtypes = [PA, vp]
        L.tla_layer_prologue.restype = i
        L.tla_layer_prologue_bwd_workspace_bytes.argtypes = [PA]
        L.tla_layer_prologue_bwd_workspace_bytes.restype = sz
        L.tla_layer_prologue_bwd.argtypes = [PA, i] + [vp] * 14 + [sz, vp]
        L.tla_layer_prologue_bwd.restype = i
        L.tla_output_gate.argtypes = [GA, vp]
        L.tla_output_gate.restype = i
        L.tla_output_gate_bwd_workspace_bytes.argtypes = [GA]
        L.tla_output_gate_bwd_workspace_bytes.restype = sz
        L.tla_output_gate_bwd.argtypes = [GA, vp, vp, vp, vp, vp, sz, vp]
        L.tla_output_gate_bwd.restype = i
        L.tla_layer_projection.argtypes = [ctypes.POINTER(tla_projection_args), vp]
        L.tla_layer_projection.restype = i
        _lib = L
    return _lib


def _ptr(t: Optional[torch.Tensor]):
    if t is None:
        return None
    if not t.is_cuda or not t.is_contiguous():
        raise ValueError("tla wants contiguous CUDA tensors")
    return ctypes.c_void_p(t.data_ptr())


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return TLA_BF16
    if t.dtype == torch.float32:
        return TLA_FP32
    raise ValueError(f"unsupported dtype {t.dtype}")


def _stream():
    return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)


def _check(fn, status):
    if status != 0:
        raise TlaError(fn, status)


def _n_states(q, cu_seqlens):
    return q.shape[0] if cu_seqlens is None else len(cu_seqlens) - 1


def make_problem(q, k, v, q2, k2, g, beta=None, h0=None, o=None, ht=None, use_delta=True,
                 chunk=64, out_dtype=None, cu_seqlens=None):
    """cu_seqlens: None, or the host token offsets of packed documents (B = 1).
    A 3-d g ([B,T,H]) is one gate per head shared by all slices (gate_per_head)."""
    B, T, H, dk = q.shape
    p = tla_problem()
    p.B, p.T, p.H, p.dk, p.dv, p.E = B, T, H, dk, v.shape[-1], q2.shape[-1]
    p.chunk, p.dtype, p.use_delta = chunk, _dtype_code(q), int(bool(use_delta))
    p.gate_per_head = int(g.dim() == 3)
    if out_dtype is None:
        out_dtype = o.dtype if o is not None else torch.float32
    p.out_dtype = _dtype_code(torch.empty(0, dtype=out_dtype))
    for name, t in (("q", q), ("k", k), ("v", v), ("q2", q2), ("k2", k2), ("g", g),
                    ("beta", beta), ("h0", h0), ("o", o), ("ht", ht)):
        setattr(p, name, _ptr(t))
    if cu_seqlens is not None:
        cu = [int(x) for x in cu_seqlens]
        arr = (ctypes.c_int * len(cu))(*cu)
        p._cu_keepalive = arr   # the library reads it during the call
        p.cu_seqlens = ctypes.cast(arr, ctypes.POINTER(ctypes.c_int))
        p.n_docs = len(cu) - 1
    return p


def fwd_workspace_bytes(p: tla_problem, save_for_bwd: bool) -> int:
    return lib().tla_fwd_workspace_bytes(ctypes.byref(p), int(save_for_bwd))


def bwd_workspace_bytes(p: tla_problem) -> int:
    return lib().tla_bwd_workspace_bytes(ctypes.byref(p))


def _workspace(nbytes, device):
    # 256-byte alignment: PyTorch's CUDA caching allocator returns 512-byte aligned blocks
    return torch.empty(max(int(nbytes), 256), dtype=torch.uint8, device=device)


def tla_chunk_fwd(q, k, v, q2, k2, g, beta=None, h0=None, use_delta=True, save_for_bwd=False,
                  want_ht=True, o=None, ht=None, workspace=None, out_dtype=torch.float32,
                  cu_seqlens=None):
    """Chunkwise forward. Returns (o, ht or None, workspace).

    o is allocated in `out_dtype` (default fp32, the accumulation precision).  With
    cu_seqlens (host offsets of packed documents, B = 1) h0 and ht are per document."""
    B, T, H, _ = q.shape
    E, dv = q2.shape[-1], v.shape[-1]
    if o is None:
        o = torch.empty(B, T, H, dv, dtype=out_dtype, device=q.device)
    if ht is None and want_ht:
        ht = torch.empty(_n_states(q, cu_seqlens), H, E, q.shape[-1], dv, dtype=torch.float32,
                         device=q.device)
    p = make_problem(q, k, v, q2, k2, g, beta, h0, o, ht, use_delta, cu_seqlens=cu_seqlens)
    need = fwd_workspace_bytes(p, save_for_bwd)
    if need == 0:
        raise TlaError("tla_fwd_workspace_bytes", -1)
    if workspace is None or workspace.numel() < need:
        workspace = _workspace(need, q.device)
    _check("tla_chunk_fwd", lib().tla_chunk_fwd(ctypes.byref(p), _ptr(workspace), need,
                                                int(save_for_bwd), _stream()))
    return o, ht, workspace


def tla_chunk_fwd_noalloc(q, k, v, q2, k2, g, beta=None, h0=None, use_delta=True,
                          want_ht=True, o=None, ht=None, out_dtype=torch.float32,
                          cu_seqlens=None):
    """Forward through the entry point that allocates nothing (built-in scratch).

    Same defaults and results as tla_chunk_fwd(save_for_bwd=False).  A caller that
    cannot allocate passes o (and ht) preallocated; when they are None they are
    allocated here with PyTorch for convenience.  Returns (o, ht or None)."""
    B, T, H, _ = q.shape
    E, dv = q2.shape[-1], v.shape[-1]
    if o is None:
        o = torch.empty(B, T, H, dv, dtype=out_dtype, device=q.device)
    if ht is None and want_ht:
        ht = torch.empty(_n_states(q, cu_seqlens), H, E, q.shape[-1], dv, dtype=torch.float32,
                         device=q.device)
    p = make_problem(q, k, v, q2, k2, g, beta, h0, o, ht, use_delta, cu_seqlens=cu_seqlens)
    _check("tla_chunk_fwd_noalloc", lib().tla_chunk_fwd_noalloc(ctypes.byref(p), _stream()))
    return o, ht


def tla_chunk_bwd(q, k, v, q2, k2, g, dO, fwd_workspace, beta=None, h0=None, dht=None,
                  use_delta=True, workspace=None, grads=None, out_dtype=torch.float32,
                  cu_seqlens=None):
    """Backward of tla_chunk_fwd; fwd_workspace from a save_for_bwd=True forward.

    Returns (dict of gradients dq, dk, dv, dq2, dk2, dg[, dbeta][, dh0], workspace).
    dq, dk, dv, dq2, dk2 are in `out_dtype` (default fp32); dg, dbeta, dh0 fp32."""
    if grads is None:
        od = out_dtype
        grads = {"dq": torch.empty(q.shape, dtype=od, device=q.device),
                 "dk": torch.empty(k.shape, dtype=od, device=q.device),
                 "dv": torch.empty(v.shape, dtype=od, device=q.device),
                 "dq2": torch.empty(q2.shape, dtype=od, device=q.device),
                 "dk2": torch.empty(k2.shape, dtype=od, device=q.device),
                 "dg": torch.empty_like(g)}
        if beta is not None:
            grads["dbeta"] = torch.empty_like(beta)
        if h0 is not None:
            grads["dh0"] = torch.empty_like(h0)
    p = make_problem(q, k, v, q2, k2, g, beta, h0, use_delta=use_delta,
                     out_dtype=grads["dq"].dtype, cu_seqlens=cu_seqlens)
    # o is not read by the backward; a non-null placeholder satisfies validation
    p.o = _ptr(dO)
    need = bwd_workspace_bytes(p)
    if need == 0:
        raise TlaError("tla_bwd_workspace_bytes", -1)
    if workspace is None or workspace.numel() < need:
        workspace = _workspace(need, q.device)
    _check("tla_chunk_bwd", lib().tla_chunk_bwd(
        ctypes.byref(p), _ptr(fwd_workspace), fwd_workspace.numel(), _ptr(dO), _ptr(dht),
        _ptr(grads["dq"]), _ptr(grads["dk"]), _ptr(grads["dv"]), _ptr(grads["dq2"]),
        _ptr(grads["dk2"]), _ptr(grads.get("dbeta")), _ptr(grads["dg"]), _ptr(grads.get("dh0")),
        _ptr(workspace), need, _stream()))
    return grads, workspace


def tla_decode_step(state, q, k, v, q2, k2, g, beta=None, use_delta=True, o=None):
    """One decode step; updates `state` [B,H,E,dk,dv] fp32 in place and returns o [B,H,dv]."""
    B, H, dk = q.shape
    dv, E = v.shape[-1], q2.shape[-1]
    if o is None:
        o = torch.empty(B, H, dv, dtype=q.dtype, device=q.device)
    _check("tla_decode_step", lib().tla_decode_step(
        B, H, dk, dv, E, int(bool(use_delta)), _dtype_code(q), _ptr(q), _ptr(k), _ptr(v),
        _ptr(q2), _ptr(k2), _ptr(g), _ptr(beta), _ptr(state), _ptr(o), _stream()))
    return o


def tla_last_device_status() -> int:
    return lib().tla_last_device_status(_stream())


def tla_selftest_bounded_wait(timeout_ns: int) -> None:
    """Launch the failure-detection self-test (a bounded wait that must expire)."""
    _check("tla_selftest_bounded_wait", lib().tla_selftest_bounded_wait(int(timeout_ns), _stream()))


def tla_version() -> str:
    return lib().tla_version().decode()


# --- layer input path and output gate (Algorithm 2)

def _prologue_args(P, conv_w, gate_in, gate_bias, A_log, beta_in, dk, dv, E, eps, out):
    B, T, H, C = P.shape
    assert C == 2 * dk + dv + 2 * E, "P channels must be 2 dk + dv + 2 E per head"
    a = tla_prologue_args()
    a.B, a.T, a.H, a.dk, a.dv, a.E, a.K = B, T, H, dk, dv, E, conv_w.shape[-1]
    a.dtype, a.eps = _dtype_code(P), float(eps)
    for name, t in (("P", P), ("conv_w", conv_w), ("gate_in", gate_in), ("gate_bias", gate_bias),
                    ("A_log", A_log), ("beta_in", beta_in)):
        setattr(a, name, _ptr(t))
    for name in ("q", "k", "v", "q2", "k2", "g", "beta"):
        setattr(a, name, _ptr(out.get(name)))
    return a


def layer_prologue(P, conv_w, gate_in, gate_bias, A_log, beta_in, dk, dv, E, eps=1e-6):
    """Input path of Algorithm 2 from the projection output P [B,T,H,2dk+dv+2E] (per head
    [q|k|v|q'|k']): returns q, k, v, q2, k2 (P's dtype), g and beta (fp32)."""
    B, T, H, _ = P.shape
    dev, dt = P.device, P.dtype
    out = {"q": torch.empty(B, T, H, dk, dtype=dt, device=dev),
           "k": torch.empty(B, T, H, dk, dtype=dt, device=dev),
           "v": torch.empty(B, T, H, dv, dtype=dt, device=dev),
           "q2": torch.empty(B, T, H, E, dtype=dt, device=dev),
           "k2": torch.empty(B, T, H, E, dtype=dt, device=dev),
           "g": torch.empty(B, T, H, E, dtype=torch.float32, device=dev),
           "beta": torch.empty(B, T, H, dtype=torch.float32, device=dev)
           if beta_in is not None else None}
    a = _prologue_args(P, conv_w, gate_in, gate_bias, A_log, beta_in, dk, dv, E, eps, out)
    _check("tla_layer_prologue", lib().tla_layer_prologue(ctypes.byref(a), _stream()))
    return out


def layer_prologue_bwd(P, conv_w, gate_in, gate_bias, A_log, beta_in, dk, dv, E, grads,
                       eps=1e-6):
    """Backward of layer_prologue.  grads: dq, dk, dv, dq2, dk2 (one dtype), dg, dbeta.
    Returns dP (P's dtype), dconv_w, dgate_in, dgate_bias, dA_log, dbeta_in (fp32)."""
    a = _prologue_args(P, conv_w, gate_in, gate_bias, A_log, beta_in, dk, dv, E, eps, {})
    # output slots are not read by the backward; any non-null aligned pointer passes validation
    for name in ("q", "k", "v", "q2", "k2", "g"):
        setattr(a, name, _ptr(P))
    a.beta = _ptr(beta_in) if beta_in is not None else None
    f32 = dict(dtype=torch.float32, device=P.device)
    out = {"dP": torch.empty_like(P), "dconv_w": torch.empty_like(conv_w),
           "dgate_in": torch.empty_like(gate_in), "dgate_bias": torch.empty_like(gate_bias),
           "dA_log": torch.empty_like(A_log),
           "dbeta_in": torch.empty(beta_in.shape, **f32) if beta_in is not None else None}
    need = lib().tla_layer_prologue_bwd_workspace_bytes(ctypes.byref(a))
    if need == 0:
        raise TlaError("tla_layer_prologue_bwd_workspace_bytes", -1)
    ws = _workspace(need, P.device)
    _check("tla_layer_prologue_bwd", lib().tla_layer_prologue_bwd(
        ctypes.byref(a), _dtype_code(grads["dq"]), _ptr(grads["dq"]), _ptr(grads["dk"]),
        _ptr(grads["dv"]), _ptr(grads["dq2"]), _ptr(grads["dk2"]), _ptr(grads["dg"]),
        _ptr(grads.get("dbeta")), _ptr(out["dP"]), _ptr(out["dconv_w"]), _ptr(out["dgate_in"]),
        _ptr(out["dgate_bias"]), _ptr(out["dA_log"]), _ptr(out["dbeta_in"]), _ptr(ws), need,
        _stream()))
    return {n: t for n, t in out.items() if t is not None}


def _gate_args(o, z, w_norm, eps, y):
    B, T, H, dv = o.shape
    a = tla_gate_args()
    a.B, a.T, a.H, a.dv = B, T, H, dv
    a.o_dtype, a.dtype, a.eps = _dtype_code(o), _dtype_code(z), float(eps)
    a.o, a.z, a.w_norm, a.y = _ptr(o), _ptr(z), _ptr(w_norm), _ptr(y)
    return a


def output_gate(o, z, w_norm, eps=1e-6):
    """Output gate of Algorithm 2: RMSNorm(o) * w_norm * sigmoid(z), in z's dtype."""
    y = torch.empty(o.shape, dtype=z.dtype, device=o.device)
    a = _gate_args(o, z, w_norm, eps, y)
    _check("tla_output_gate", lib().tla_output_gate(ctypes.byref(a), _stream()))
    return y


def output_gate_bwd(o, z, w_norm, dy, eps=1e-6):
    """Backward of output_gate: returns do (o's dtype), dz (z's dtype), dw_norm (fp32)."""
    out = {"do": torch.empty_like(o), "dz": torch.empty_like(z), "dw_norm": torch.empty_like(w_norm)}
    a = _gate_args(o, z, w_norm, eps, dy)
    need = lib().tla_output_gate_bwd_workspace_bytes(ctypes.byref(a))
    if need == 0:
        raise TlaError("tla_output_gate_bwd_workspace_bytes", -1)
    ws = _workspace(need, o.device)
    _check("tla_output_gate_bwd", lib().tla_output_gate_bwd(
        ctypes.byref(a), _ptr(dy), _ptr(out["do"]), _ptr(out["dz"]), _ptr(out["dw_norm"]),
        _ptr(ws), need, _stream()))
    return out


# --- input projection GEMM fused with the input path (Algorithm 2)

def layer_projection(u, W, conv_w, gate_in, gate_bias, A_log, beta_in, dk, dv, E, eps=1e-6,
                     want_P=False):
    """One tensor-core GEMM P = u W^T (u [B,T,Dm] bf16, W [H*C, Dm] bf16, C = 2dk+dv+2E,
    per head [q|k|v|q'|k']) with the input path of layer_prologue applied in its epilogue.
    Returns q, k, v, q2, k2 (bf16), g and beta (fp32), and P (bf16) when want_P."""
    B, T, Dm = u.shape
    H = conv_w.shape[0]
    C = 2 * dk + dv + 2 * E
    assert W.shape == (H * C, Dm), "W must be [H * (2 dk + dv + 2 E), Dm]"
    dev, bf = u.device, torch.bfloat16
    out = {"q": torch.empty(B, T, H, dk, dtype=bf, device=dev),
           "k": torch.empty(B, T, H, dk, dtype=bf, device=dev),
           "v": torch.empty(B, T, H, dv, dtype=bf, device=dev),
           "q2": torch.empty(B, T, H, E, dtype=bf, device=dev),
           "k2": torch.empty(B, T, H, E, dtype=bf, device=dev),
           "g": torch.empty(B, T, H, E, dtype=torch.float32, device=dev),
           "beta": torch.empty(B, T, H, dtype=torch.float32, device=dev)
           if beta_in is not None else None,
           "P": torch.empty(B, T, H, C, dtype=bf, device=dev) if want_P else None}
    a = tla_projection_args()
    a.B, a.T, a.H, a.dk, a.dv, a.E = B, T, H, dk, dv, E
    a.K, a.Dm, a.eps = conv_w.shape[-1], Dm, float(eps)
    for name, t in (("u", u), ("W", W), ("conv_w", conv_w), ("gate_in", gate_in),
                    ("gate_bias", gate_bias), ("A_log", A_log), ("beta_in", beta_in)):
        setattr(a, name, _ptr(t))
    for name in ("q", "k", "v", "q2", "k2", "g", "beta", "P"):
        setattr(a, name, _ptr(out[name]))
    _check("tla_layer_projection", lib().tla_layer_projection(ctypes.byref(a), _stream()))
    return {n: t for n, t in out.items() if t is not None}
