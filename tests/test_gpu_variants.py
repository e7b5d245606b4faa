"""Shape and gate variants (Table 4's E = 16/32 with d_k = 32/64, and a single log gate per
head shared by every slice) through the C ABI against the float64 oracle.

A per-head gate is the per-slice form with the gate repeated over the slices, so the
oracle runs on the repeated gate and the per-head gradient is the sum over the slices of
the per-slice gradient (chain rule of the repetition).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_36529_gb300 import inputs, tla

pytestmark = pytest.mark.gpu

TOL = {"fp32": 1e-4, "bf16": 2e-2}


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__ as ge
    ge.build()
    assert torch.cuda.is_available()


def _np(t):
    return None if t is None else t.detach().double().cpu().numpy()


def close(name, got, ref, tol, rel_l2=None):
    got = np.asarray(_np(got) if isinstance(got, torch.Tensor) else got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, (name, got.shape, ref.shape)
    assert np.isfinite(got).all(), name
    rms = float(np.sqrt(np.mean(ref ** 2)))
    if rms == 0.0:
        assert np.abs(got).max() <= 1e-6, name
        return
    err = float(np.abs(got - ref).max())
    assert err <= tol * rms, f"{name}: max|err| {err:.3e} > {tol} x RMS {rms:.3e}"
    if rel_l2 is not None:
        rl = float(np.linalg.norm(got - ref) / np.linalg.norm(ref))
        assert rl < rel_l2, f"{name}: rel L2 {rl:.3e}"


def run_both(x, use_delta, dht=None):
    o, ht, ws = tla.tla_chunk_fwd(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"], x["beta"],
                                  x["h0"], use_delta=use_delta, save_for_bwd=True)
    grads, _ = tla.tla_chunk_bwd(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"], x["dO"], ws,
                                 beta=x["beta"], h0=x["h0"], dht=dht, use_delta=use_delta)
    torch.cuda.synchronize()
    assert tla.tla_last_device_status() == 0
    return o, ht, grads


def oracle_both(x, use_delta, g_slices, dht=None):
    c = {n: _np(t) for n, t in x.items()}
    ro, rht = oracle.forward(c["q"], c["k"], c["v"], c["q2"], c["k2"], g_slices, c["beta"],
                             c["h0"], use_delta=use_delta)
    rg = oracle.backward(c["q"], c["k"], c["v"], c["q2"], c["k2"], g_slices, c["dO"], c["beta"],
                         c["h0"], _np(dht), use_delta=use_delta)
    return ro, rht, rg


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
@pytest.mark.parametrize("dk,dv,E", [(32, 64, 32), (64, 128, 32), (64, 64, 16)])
def test_many_slices(dtype, dk, dv, E):
    """E = 16 and 32 with d_k = 32 / 64 (the paper's iso-state variants)."""
    x = inputs.chunk_inputs(1, 130, 2, dk, dv, E, dtype=dtype, with_beta=True, h0_std=0.1,
                            backward=True, device="cuda", seed=dk + E)
    o, ht, grads = run_both(x, True)
    ro, rht, rg = oracle_both(x, True, _np(x["g"]))
    rel = 0.01 if dtype == "bf16" else None
    close("o", o, ro, TOL[dtype], rel)
    close("ht", ht, rht, TOL[dtype], rel)
    for n in rg:
        close(n, grads[n], rg[n], TOL[dtype], rel)


@pytest.mark.parametrize("use_delta", [True, False])
@pytest.mark.parametrize("dtype,dk,dv,E", [("bf16", 128, 128, 4), ("fp32", 32, 32, 4),
                                           ("bf16", 128, 64, 8)])
def test_gate_per_head(use_delta, dtype, dk, dv, E):
    x = inputs.chunk_inputs(2, 150, 2, dk, dv, E, dtype=dtype, with_beta=True, h0_std=0.1,
                            backward=True, device="cuda", seed=3 * E + dk)
    x["g"] = x["g"][..., 0].contiguous()   # one log gate per head and token: [B,T,H]
    o, ht, grads = run_both(x, use_delta)
    assert grads["dg"].shape == x["g"].shape
    g_slices = np.repeat(_np(x["g"])[..., None], E, axis=-1)
    ro, rht, rg = oracle_both(x, use_delta, g_slices)
    rg["dg"] = rg["dg"].sum(axis=-1)
    rel = 0.01 if dtype == "bf16" else None
    close("o", o, ro, TOL[dtype], rel)
    close("ht", ht, rht, TOL[dtype], rel)
    for n in rg:
        close(n, grads[n], rg[n], TOL[dtype], rel)


@pytest.mark.parametrize("use_delta", [True, False])
def test_decode_many_slices(use_delta):
    B, H, dk, dv, E = 3, 2, 64, 64, 32
    gen = torch.Generator("cuda")
    gen.manual_seed(5)
    state = 0.1 * torch.randn(B, H, E, dk, dv, device="cuda", generator=gen)
    ref_state = _np(state)
    for step in range(3):
        s = inputs.decode_inputs(B, H, dk, dv, E, dtype="bf16", device="cuda", seed=10 + step)
        o = tla.tla_decode_step(state, s["q"], s["k"], s["v"], s["q2"], s["k2"], s["g"], s["beta"],
                                use_delta=use_delta)
        torch.cuda.synchronize()
        c = {n: _np(t) for n, t in s.items()}
        ro, ref_state = oracle.decode_step(ref_state, c["q"], c["k"], c["v"], c["q2"], c["k2"],
                                           c["g"], c["beta"], use_delta=use_delta)
        close("o", o, ro, TOL["bf16"])
        close("state", state, ref_state, TOL["bf16"])
