"""GPU parity of the fused input projection (Algorithm 2; Appendix A, Input projections):
one tcgen05 GEMM P = u W^T whose epilogue runs the causal convolution, activations, L2
normalisations, log gates and beta.  Reference: the oracle's float64 projection of the same
bf16 u and W, then the oracle's input path on P.

Tolerances: the bf16-stored outputs (q, k, v, q', k', P) within 2e-2 x RMS plus their own
rounding (2^-8 |ref|); the fp32 gates and beta within 1e-4 x RMS (their inputs are fp32)."""
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
    return t.detach().double().cpu().numpy()


def close_rounded(name, got, ref, tol=2e-2, roundings=1):
    got = _np(got)
    rms = float(np.sqrt(np.mean(ref ** 2)))
    excess = np.abs(got - ref) - (tol * rms + roundings * 2.0 ** -8 * np.abs(ref))
    assert np.isfinite(got).all() and excess.max() <= 0, f"{name}: exceeds by {excess.max():.3e}"


def close(name, got, ref, tol):
    got = _np(got)
    rms = float(np.sqrt(np.mean(ref ** 2)))
    err = float(np.abs(got - ref).max())
    assert np.isfinite(got).all() and err <= tol * rms, f"{name}: {err:.3e} > {tol} x {rms:.3e}"


# (B, T, H, dk, dv, E, K, Dm): several 125-token blocks with a ragged last block, both head
# sizes, an odd slice count (scalar stores of q', k'), short windows, T below the halo
SHAPES = [(2, 300, 2, 128, 128, 4, 4, 256), (1, 130, 3, 64, 64, 3, 2, 128),
          (2, 64, 2, 128, 64, 8, 3, 192), (3, 2, 1, 64, 128, 16, 4, 64)]


@pytest.mark.parametrize("B,T,H,dk,dv,E,K,Dm", SHAPES)
def test_projection_matches_oracle(B, T, H, dk, dv, E, K, Dm):
    x = inputs.projection_inputs(B, T, H, dk, dv, E, Dm, K, device="cuda", seed=B * T + E)
    got = tla.layer_projection(x["u"], x["W"], x["conv_w"], x["gate_in"], x["gate_bias"],
                               x["A_log"], x["beta_in"], dk, dv, E, want_P=True)
    torch.cuda.synchronize()
    assert tla.tla_last_device_status() == 0
    P = oracle.projection(_np(x["u"]), _np(x["W"]), H)
    ref = oracle.prologue(P, _np(x["conv_w"]), _np(x["gate_in"]), _np(x["gate_bias"]),
                          _np(x["A_log"]), _np(x["beta_in"]), dk, dv, E)
    close_rounded("P", got["P"], P)
    for n in ("q", "k", "v", "q2", "k2"):
        close_rounded(n, got[n], ref[n])
    close("g", got["g"], ref["g"], 1e-4)
    close("beta", got["beta"], ref["beta"], 1e-4)


def test_projection_equals_gemm_then_prologue_without_beta():
    """Without beta_in, and against the two-kernel path on the kernel's own P: the fused
    epilogue gives what tla_layer_prologue gives on that P.  The fused path works on the fp32
    accumulator, the other on its bf16 rounding, and both outputs are bf16: the bound allows
    both roundings."""
    B, T, H, dk, dv, E, K, Dm = 1, 260, 2, 128, 128, 4, 4, 128
    x = inputs.projection_inputs(B, T, H, dk, dv, E, Dm, K, device="cuda", seed=5)
    got = tla.layer_projection(x["u"], x["W"], x["conv_w"], x["gate_in"], x["gate_bias"],
                               x["A_log"], None, dk, dv, E, want_P=True)
    two = tla.layer_prologue(got["P"], x["conv_w"], x["gate_in"], x["gate_bias"], x["A_log"],
                             None, dk, dv, E)
    torch.cuda.synchronize()
    assert "beta" not in got
    for n in ("q", "k", "v", "q2", "k2"):
        ref = _np(two[n])
        close_rounded(n, got[n], ref, roundings=2)
    close("g", got["g"], _np(two["g"]), 1e-6)
