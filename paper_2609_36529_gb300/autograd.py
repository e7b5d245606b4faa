"""torch.autograd binding of the chunkwise forward and backward (tla_chunk_fwd / tla_chunk_bwd).

Argument marshalling only: the forward saves its workspace for the backward, and the
backward runs the library's backward kernels; gradients come back in the inputs' dtypes.
"""
from typing import Optional, Sequence

import torch

from . import tla


class _TriadicLinearAttention(torch.autograd.Function):
    @staticmethod
    def forward(ctx, q, k, v, q2, k2, g, beta, h0, use_delta, cu_seqlens):
        o, ht, ws = tla.tla_chunk_fwd(q, k, v, q2, k2, g, beta, h0, use_delta=use_delta,
                                      save_for_bwd=True, want_ht=True, cu_seqlens=cu_seqlens)
        ctx.use_delta = use_delta
        ctx.cu_seqlens = cu_seqlens
        ctx.save_for_backward(q, k, v, q2, k2, g, beta, h0, ws)
        return o, ht

    @staticmethod
    def backward(ctx, do, dht):
        q, k, v, q2, k2, g, beta, h0, ws = ctx.saved_tensors
        grads, _ = tla.tla_chunk_bwd(q, k, v, q2, k2, g, do.to(q.dtype).contiguous(), ws,
                                     beta=beta, h0=h0,
                                     dht=None if dht is None else dht.float().contiguous(),
                                     use_delta=ctx.use_delta, cu_seqlens=ctx.cu_seqlens)

        def like(t, ref):
            return None if t is None else t.to(ref.dtype)

        return (like(grads["dq"], q), like(grads["dk"], k), like(grads["dv"], v),
                like(grads["dq2"], q2), like(grads["dk2"], k2), grads["dg"],
                grads.get("dbeta"), grads.get("dh0"), None, None)


def triadic_linear_attention(q, k, v, q2, k2, g, beta: Optional[torch.Tensor] = None,
                             h0: Optional[torch.Tensor] = None, use_delta: bool = True,
                             cu_seqlens: Optional[Sequence[int]] = None):
    """Chunkwise triadic linear attention with gradients (Appendix A forward and backward).

    q, k [B,T,H,dk]; v [B,T,H,dv]; q2, k2 [B,T,H,E] (bf16 or fp32, contiguous CUDA);
    g [B,T,H,E] (or [B,T,H], one gate per head) fp32 log forget gates; beta [B,T,H] or
    None; h0 [B,H,E,dk,dv] or None.  Returns (o [B,T,H,dv] fp32, ht [B,H,E,dk,dv] fp32)."""
    return _TriadicLinearAttention.apply(q, k, v, q2, k2, g, beta, h0, use_delta, cu_seqlens)
