"""Layer input path and output gate (Algorithm 2) through the C ABI against the float64
oracle, and a whole layer forward (prologue -> chunkwise operator -> output gate).

Tolerances: fp32 results max|err| <= 1e-4 * RMS(oracle); results stored in bf16 add
their rounding, |err| <= 1e-4 * RMS + 2^-8 |ref|; the whole bf16 layer 2e-2 * RMS."""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_36529_gb300 import inputs, tla

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__ as ge
    ge.build()
    assert torch.cuda.is_available()


def _np(t):
    return None if t is None else t.detach().double().cpu().numpy()


def close(name, got, ref, tol=1e-4, rounded=False):
    got, ref = _np(got), np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, (name, got.shape, ref.shape)
    assert np.isfinite(got).all(), name
    rms = float(np.sqrt(np.mean(ref ** 2)))
    bound = tol * rms + (2.0 ** -8 * np.abs(ref) if rounded else 0.0)
    excess = float((np.abs(got - ref) - bound).max())
    assert excess <= 0, f"{name}: exceeds the bound by {excess:.3e} (RMS {rms:.3e})"


# the last shape has an odd channel count C (E odd): the scalar-access path of the prologue
SHAPES = [(128, 128, 4, 4), (64, 64, 8, 3), (32, 128, 32, 1), (16, 32, 3, 2)]
ARGS = ("P", "conv_w", "gate_in", "gate_bias", "A_log", "beta_in")


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
@pytest.mark.parametrize("dk,dv,E,K", SHAPES)
def test_prologue_forward(dtype, dk, dv, E, K):
    x = inputs.layer_inputs(2, 130, 3, dk, dv, E, K, dtype=dtype, device="cuda", seed=dk + E)
    got = tla.layer_prologue(*(x[n] for n in ARGS), dk, dv, E)
    torch.cuda.synchronize()
    ref = oracle.prologue(*(_np(x[n]) for n in ARGS), dk, dv, E)
    for n in ("q", "k", "v", "q2", "k2"):
        close(n, got[n], ref[n], rounded=dtype == "bf16")
    close("g", got["g"], ref["g"])
    close("beta", got["beta"], ref["beta"])


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
@pytest.mark.parametrize("dk,dv,E,K", SHAPES)
def test_prologue_backward(dtype, dk, dv, E, K):
    B, T, H = 2, 300, 3   # two token segments of the backward, the second ragged
    x = inputs.layer_inputs(B, T, H, dk, dv, E, K, dtype=dtype, device="cuda", seed=7 + dk)
    gen = torch.Generator("cuda").manual_seed(3)
    grads = {n: torch.randn(B, T, H, w, device="cuda", generator=gen)
             for n, w in (("dq", dk), ("dk", dk), ("dv", dv), ("dq2", E), ("dk2", E), ("dg", E))}
    grads["dbeta"] = torch.randn(B, T, H, device="cuda", generator=gen)
    got = tla.layer_prologue_bwd(*(x[n] for n in ARGS), dk, dv, E, grads)
    torch.cuda.synchronize()
    ref = oracle.prologue_backward(*(_np(x[n]) for n in ARGS), {n: _np(t) for n, t in grads.items()},
                                   dk, dv, E)
    for n in ref:
        close(n, got[n], ref[n], rounded=(n == "dP" and dtype == "bf16"))


@pytest.mark.parametrize("T", [1, 2, 5])
def test_prologue_sequences_shorter_than_the_window(T):
    """Fewer tokens than the convolution's K = 4 taps, forward and backward."""
    dk, dv, E, K, B, H = 32, 32, 4, 4, 2, 2
    x = inputs.layer_inputs(B, T, H, dk, dv, E, K, dtype="fp32", device="cuda", seed=T)
    got = tla.layer_prologue(*(x[n] for n in ARGS), dk, dv, E)
    gen = torch.Generator("cuda").manual_seed(T)
    grads = {n: torch.randn(B, T, H, w, device="cuda", generator=gen)
             for n, w in (("dq", dk), ("dk", dk), ("dv", dv), ("dq2", E), ("dk2", E), ("dg", E))}
    grads["dbeta"] = torch.randn(B, T, H, device="cuda", generator=gen)
    gotb = tla.layer_prologue_bwd(*(x[n] for n in ARGS), dk, dv, E, grads)
    torch.cuda.synchronize()
    ref = oracle.prologue(*(_np(x[n]) for n in ARGS), dk, dv, E)
    for n in ("q", "k", "v", "q2", "k2", "g", "beta"):
        close(n, got[n], ref[n])
    refb = oracle.prologue_backward(*(_np(x[n]) for n in ARGS), {n: _np(t) for n, t in grads.items()},
                                    dk, dv, E)
    for n in refb:
        close(n, gotb[n], refb[n])


@pytest.mark.parametrize("zdtype", ["fp32", "bf16"])
@pytest.mark.parametrize("dv", [128, 64, 16])
def test_output_gate_forward_and_backward(zdtype, dv):
    x = inputs.layer_inputs(2, 77, 3, 16, dv, 1, dtype=zdtype, device="cuda", seed=dv)
    y = tla.output_gate(x["o"], x["z"], x["w_norm"])
    gen = torch.Generator("cuda").manual_seed(1)
    dy = torch.randn(x["o"].shape, device="cuda", generator=gen).to(x["z"].dtype)
    g = tla.output_gate_bwd(x["o"], x["z"], x["w_norm"], dy)
    torch.cuda.synchronize()
    rounded = zdtype == "bf16"
    close("y", y, oracle.gate_norm(_np(x["o"]), _np(x["z"]), _np(x["w_norm"])), rounded=rounded)
    ref = oracle.gate_norm_backward(_np(x["o"]), _np(x["z"]), _np(x["w_norm"]), _np(dy))
    close("do", g["do"], ref["do"])
    close("dz", g["dz"], ref["dz"], rounded=rounded)
    close("dw_norm", g["dw_norm"], ref["dw_norm"])


def test_whole_layer_forward():
    """Prologue -> chunkwise triadic GDN (tensor-core path) -> output gate, bf16."""
    B, T, H, dk, dv, E = 2, 200, 2, 128, 128, 4
    x = inputs.layer_inputs(B, T, H, dk, dv, E, 4, dtype="bf16", device="cuda", seed=21)
    pro = tla.layer_prologue(*(x[n] for n in ARGS), dk, dv, E)
    o, _, _ = tla.tla_chunk_fwd(pro["q"], pro["k"], pro["v"], pro["q2"], pro["k2"], pro["g"],
                                pro["beta"], None, use_delta=True, want_ht=False)
    y = tla.output_gate(o, x["z"], x["w_norm"])
    torch.cuda.synchronize()
    assert tla.tla_last_device_status() == 0
    # each stage against the oracle on the exact values the GPU's next stage reads (the
    # prologue's own parity, including its bf16 rounding, is tested above)
    rp = oracle.prologue(*(_np(x[n]) for n in ARGS), dk, dv, E)
    for n in ("q", "k", "v", "q2", "k2"):
        close(n, pro[n], rp[n], rounded=True)
    ro, _ = oracle.forward(*(_np(pro[n]) for n in ("q", "k", "v", "q2", "k2", "g", "beta")),
                           None, use_delta=True)
    close("o", o, ro, tol=2e-2)
    ry = oracle.gate_norm(ro, _np(x["z"]), _np(x["w_norm"]))
    close("y", y, ry, tol=2e-2, rounded=True)
