"""Seeded synthetic inputs shaped like the paper's language-modelling workloads.

This module holds no arithmetic of the method itself: it only draws random
tensors and applies the input preconditions the paper's layer applies before
the operator (L2-normalised queries and keys, Algorithm 2; log-sigmoid forget
gates so that log alpha <= 0; beta in (0,1) through a sigmoid).  Both the CUDA
path's tests/benchmark and the oracle's tests draw their inputs here.

Recipe (fixed tensor order q, k, q2, k2, v, beta, g, h0, dO, one
``torch.Generator`` seeded with ``seed``):
  q, k   ~ N(0,1) [B,T,H,dk], L2-normalised per vector in fp32
  q2, k2 ~ N(0,1) [B,T,H,E],  L2-normalised per vector in fp32
  v      ~ N(0,1) [B,T,H,dv]
  beta   = sigmoid(N(0,1)) [B,T,H]              (only when requested)
  g      = logsigmoid(N(gate_mean, 1)) [B,T,H,E] (log forget gates, <= 0)
  h0     ~ N(0, h0_std^2) [B,H,E,dk,dv] fp32     (only when h0_std > 0)
  dO     ~ N(0,1) [B,T,H,dv]                      (only when requested)
q, k, q2, k2, v, dO are then cast to ``dtype``; g, beta, h0 stay fp32.
Packed documents: the same draws for one sequence of sum(lengths) tokens, initial
states per document from a generator seeded with ``seed + 1``, and document lengths
log-normal around a mean (sigma 1) with the last one cut to the total.
"""
from dataclasses import dataclass
from typing import Optional

import numpy as np
import torch


@dataclass(frozen=True)
class Workload:
    name: str
    B: int
    T: int
    H: int
    dk: int
    dv: int
    E: int
    dtype: str            # "fp32" | "bf16"
    use_delta: bool
    with_beta: bool
    h0_std: float = 0.0
    backward: bool = False
    chunk: int = 64


# The five workloads of the paper's setting (Section 3.1, Appendix A: d=128, C=64,
# E in {4,8,16}, 4k pretraining / 64k extension context).
SGLA_FWD_FP32 = Workload("sgla_fwd_fp32_B1_H2_T256_d32_E4", 1, 256, 2, 32, 32, 4, "fp32",
                         use_delta=False, with_beta=False)
GDN_FWD_BF16 = Workload("gdn_fwd_bf16_B4_H16_T4096_d128_E8", 4, 4096, 16, 128, 128, 8, "bf16",
                        use_delta=True, with_beta=True)
GDN_FWDBWD_BF16 = Workload("gdn_fwdbwd_bf16_B8_H16_T8192_d128_E4", 8, 8192, 16, 128, 128, 4,
                           "bf16", use_delta=True, with_beta=True, backward=True)
GDN_LONG_BF16 = Workload("gdn_fwd_bf16_B1_H32_T65536_d128_E16", 1, 65536, 32, 128, 128, 16,
                         "bf16", use_delta=True, with_beta=True, h0_std=0.1)
WORKLOADS = {w.name: w for w in (SGLA_FWD_FP32, GDN_FWD_BF16, GDN_FWDBWD_BF16, GDN_LONG_BF16)}


@dataclass(frozen=True)
class DecodeWorkload:
    name: str
    B: int
    H: int
    dk: int
    dv: int
    E: int
    steps: int
    prefill: int


DECODE = DecodeWorkload("decode_fp32_state_B256_H32_E8_d128", 256, 32, 128, 128, 8, 100, 512)


def torch_dtype(name: str) -> torch.dtype:
    return {"fp32": torch.float32, "bf16": torch.bfloat16}[name]


def _unit(x: torch.Tensor) -> torch.Tensor:
    return x / x.norm(dim=-1, keepdim=True).clamp_min(1e-12)


def chunk_inputs(B, T, H, dk, dv, E, dtype="bf16", with_beta=True, h0_std=0.0,
                 backward=False, device="cpu", seed=0, gate_mean=3.0,
                 gen: Optional[torch.Generator] = None):
    """Draw one batch of inputs for the chunkwise forward (and backward)."""
    dev = torch.device(device)
    if gen is None:
        gen = torch.Generator(device=dev)
        gen.manual_seed(seed)
    dt = torch_dtype(dtype)

    def randn(*shape):
        return torch.randn(*shape, generator=gen, device=dev, dtype=torch.float32)

    out = {}
    out["q"] = _unit(randn(B, T, H, dk)).to(dt)
    out["k"] = _unit(randn(B, T, H, dk)).to(dt)
    out["q2"] = _unit(randn(B, T, H, E)).to(dt)
    out["k2"] = _unit(randn(B, T, H, E)).to(dt)
    out["v"] = randn(B, T, H, dv).to(dt)
    out["beta"] = torch.sigmoid(randn(B, T, H)) if with_beta else None
    out["g"] = torch.nn.functional.logsigmoid(randn(B, T, H, E) + gate_mean)
    out["h0"] = randn(B, H, E, dk, dv) * h0_std if h0_std > 0 else None
    out["dO"] = randn(B, T, H, dv).to(dt) if backward else None
    return out


def packed_inputs(lens, H, dk, dv, E, dtype="bf16", with_beta=True, h0_std=0.0,
                  backward=False, device="cpu", seed=0):
    """Inputs of packed documents of the given lengths: one sequence of sum(lens) tokens
    (B = 1) drawn like chunk_inputs, initial states per document ([n_docs,H,E,dk,dv]) and
    the host token offsets cu_seqlens (n_docs + 1 values, starting at 0)."""
    T = int(sum(int(n) for n in lens))
    x = chunk_inputs(1, T, H, dk, dv, E, dtype, with_beta, 0.0, backward, device=device,
                     seed=seed)
    if h0_std > 0:
        gen = torch.Generator(device=torch.device(device))
        gen.manual_seed(seed + 1)
        x["h0"] = torch.randn(len(lens), H, E, dk, dv, generator=gen, device=torch.device(device),
                              dtype=torch.float32) * h0_std
    cu = [0]
    for n in lens:
        cu.append(cu[-1] + int(n))
    return x, cu


def packed_lengths(total, mean_len, seed=0, min_len=1):
    """Document lengths summing to `total`: log-normal around `mean_len` (sigma 1), the
    last one cut to fit -- a stand-in for the length mix of a packed pretraining batch."""
    rng = np.random.default_rng(seed)
    mu = np.log(mean_len) - 0.5
    lens = []
    left = int(total)
    while left > 0:
        n = max(min_len, int(rng.lognormal(mu, 1.0)))
        n = min(n, left)
        lens.append(n)
        left -= n
    return lens


def layer_inputs(B, T, H, dk, dv, E, K=4, dtype="bf16", device="cpu", seed=0):
    """Inputs of the layer input path and output gate (Algorithm 2), one generator:
    P ~ N(0,1) [B,T,H,2dk+dv+2E] (dtype), conv_w ~ N(0,1/K) [H,C,K], gate_in ~ N(0,1)
    [B,T,H,E], gate_bias ~ N(1,1) [H,E], A_log ~ N(-1,0.5^2) [H,E], beta_in ~ N(0,1) [B,T,H],
    o ~ N(0,1) [B,T,H,dv] fp32, z ~ N(0,1) [B,T,H,dv] (dtype), w_norm ~ 1 + 0.1 N(0,1) [dv];
    all but P and z fp32."""
    dev = torch.device(device)
    gen = torch.Generator(device=dev)
    gen.manual_seed(seed)
    dt = torch_dtype(dtype)
    C = 2 * dk + dv + 2 * E

    def randn(*shape):
        return torch.randn(*shape, generator=gen, device=dev, dtype=torch.float32)

    return {"P": randn(B, T, H, C).to(dt), "conv_w": randn(H, C, K) / K ** 0.5,
            "gate_in": randn(B, T, H, E), "gate_bias": randn(H, E) + 1.0,
            "A_log": 0.5 * randn(H, E) - 1.0, "beta_in": randn(B, T, H),
            "o": randn(B, T, H, dv), "z": randn(B, T, H, dv).to(dt),
            "w_norm": 1.0 + 0.1 * randn(dv)}


def projection_inputs(B, T, H, dk, dv, E, Dm, K=4, device="cpu", seed=0):
    """Inputs of the fused input projection (Algorithm 2): the normalised layer input
    u ~ N(0,1) [B,T,Dm] and the projection weight W ~ N(0, 1/Dm) [H*(2dk+dv+2E), Dm], both
    bf16, then the parameters of layer_inputs (conv_w, gate_in, gate_bias, A_log, beta_in;
    fp32) from the same generator."""
    dev = torch.device(device)
    gen = torch.Generator(device=dev)
    gen.manual_seed(seed)
    C = 2 * dk + dv + 2 * E

    def randn(*shape):
        return torch.randn(*shape, generator=gen, device=dev, dtype=torch.float32)

    return {"u": randn(B, T, Dm).to(torch.bfloat16),
            "W": (randn(H * C, Dm) / Dm ** 0.5).to(torch.bfloat16),
            "conv_w": randn(H, C, K) / K ** 0.5, "gate_in": randn(B, T, H, E),
            "gate_bias": randn(H, E) + 1.0, "A_log": 0.5 * randn(H, E) - 1.0,
            "beta_in": randn(B, T, H)}


def workload_inputs(w: Workload, device="cpu", seed=0, B=None, T=None, H=None):
    """Inputs of a named workload, optionally with a reduced B/T/H for tests."""
    return chunk_inputs(B or w.B, T or w.T, H or w.H, w.dk, w.dv, w.E, w.dtype, w.with_beta,
                        w.h0_std, w.backward, device=device, seed=seed)


def decode_inputs(B, H, dk, dv, E, dtype="fp32", with_beta=True, device="cpu",
                  gen: Optional[torch.Generator] = None, seed=0):
    """Inputs of one decode step: q,k [B,H,dk]; v [B,H,dv]; q2,k2,g [B,H,E]; beta [B,H]."""
    dev = torch.device(device)
    if gen is None:
        gen = torch.Generator(device=dev)
        gen.manual_seed(seed)
    d = chunk_inputs(B, 1, H, dk, dv, E, dtype, with_beta, device=dev, gen=gen)
    return {n: (None if t is None else t[:, 0].contiguous()) for n, t in d.items()
            if n not in ("h0", "dO")}
