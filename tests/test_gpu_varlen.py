"""Packed variable-length documents (Appendix A, Kernels): the CUDA path through the C ABI
against the float64 oracle run document by document, each from its own initial state.

Tolerances as in test_gpu_parity (bf16 inputs): max|err| <= 2e-2 * RMS(oracle), gradients
also rel. L2 < 1%.  Packing equal-length documents must reproduce the batched call exactly.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_36529_gb300 import inputs, tla

pytestmark = pytest.mark.gpu

TOL = 2e-2


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__ as ge
    ge.build()
    assert torch.cuda.is_available()


def _np(t):
    return None if t is None else t.detach().double().cpu().numpy()


def close(name, got, ref, rel_l2=None):
    got = np.asarray(_np(got) if isinstance(got, torch.Tensor) else got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, (name, got.shape, ref.shape)
    assert np.isfinite(got).all(), name
    rms = float(np.sqrt(np.mean(ref ** 2)))
    if rms == 0.0:
        assert np.abs(got).max() <= 1e-6, name
        return
    err = float(np.abs(got - ref).max())
    assert err <= TOL * rms, f"{name}: max|err| {err:.3e} > {TOL} x RMS {rms:.3e}"
    if rel_l2 is not None:
        rl = float(np.linalg.norm(got - ref) / np.linalg.norm(ref))
        assert rl < rel_l2, f"{name}: rel L2 {rl:.3e}"


def packed(lens, H, dv, E, seed, backward=False, dk=128):
    x, cu = inputs.packed_inputs(lens, H, dk, dv, E, dtype="bf16", h0_std=0.1,
                                 backward=backward, device="cuda", seed=seed)
    return x, cu


def oracle_docs(x, cu, use_delta, dht=None):
    """Forward (and with dht given, backward) of every document on its own."""
    c = {n: _np(t) for n, t in x.items()}
    T, H, dv = c["v"].shape[1], c["v"].shape[2], c["v"].shape[3]
    o = np.zeros((1, T, H, dv))
    ht = np.zeros_like(c["h0"])
    grads = None
    if dht is not None:
        grads = {n: np.zeros_like(c[k]) for n, k in (("dq", "q"), ("dk", "k"), ("dv", "v"),
                                                    ("dq2", "q2"), ("dk2", "k2"), ("dg", "g"),
                                                    ("dbeta", "beta"), ("dh0", "h0"))}
    for d in range(len(cu) - 1):
        a, b = cu[d], cu[d + 1]
        if a == b:   # empty document: state and its gradient pass through
            ht[d] = c["h0"][d]
            if grads is not None:
                grads["dh0"][d] = dht[d]
            continue
        sl = {n: c[n][:, a:b] for n in ("q", "k", "v", "q2", "k2", "g", "beta")}
        od, hd = oracle.forward(sl["q"], sl["k"], sl["v"], sl["q2"], sl["k2"], sl["g"],
                                sl["beta"], c["h0"][d:d + 1], use_delta=use_delta)
        o[:, a:b] = od
        ht[d] = hd[0]
        if grads is not None:
            gd = oracle.backward(sl["q"], sl["k"], sl["v"], sl["q2"], sl["k2"], sl["g"],
                                 c["dO"][:, a:b], sl["beta"], c["h0"][d:d + 1], dht[d:d + 1],
                                 use_delta=use_delta)
            for n in ("dq", "dk", "dv", "dq2", "dk2", "dg", "dbeta"):
                grads[n][:, a:b] = gd[n]
            grads["dh0"][d] = gd["dh0"][0]
    return o, ht, grads


LENS = [[1, 63, 64, 65, 130, 7], [300], [0, 70, 0, 5, 64, 0]]


@pytest.mark.parametrize("use_delta", [True, False])
@pytest.mark.parametrize("lens", LENS)
@pytest.mark.parametrize("dv,E", [(128, 4), (64, 8)])
def test_packed_forward(use_delta, lens, dv, E):
    x, cu = packed(lens, 2, dv, E, seed=sum(lens) + dv + E)
    o, ht, _ = tla.tla_chunk_fwd(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"], x["beta"],
                                 x["h0"], use_delta=use_delta, cu_seqlens=cu)
    torch.cuda.synchronize()
    assert tla.tla_last_device_status() == 0
    ro, rht, _ = oracle_docs(x, cu, use_delta)
    close("o", o, ro, rel_l2=0.01)
    close("ht", ht, rht, rel_l2=0.01)


@pytest.mark.parametrize("use_delta", [True, False])
@pytest.mark.parametrize("lens", LENS)
def test_packed_backward(use_delta, lens):
    E, dv = 4, 128
    x, cu = packed(lens, 2, dv, E, seed=7 * sum(lens), backward=True)
    gen = torch.Generator("cuda")
    gen.manual_seed(len(lens))
    dht = 0.5 * torch.randn(len(lens), 2, E, 128, dv, device="cuda", generator=gen)
    _, _, ws = tla.tla_chunk_fwd(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"], x["beta"],
                                 x["h0"], use_delta=use_delta, save_for_bwd=True, cu_seqlens=cu)
    grads, _ = tla.tla_chunk_bwd(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"], x["dO"], ws,
                                 beta=x["beta"], h0=x["h0"], dht=dht, use_delta=use_delta,
                                 cu_seqlens=cu)
    torch.cuda.synchronize()
    assert tla.tla_last_device_status() == 0
    _, _, ref = oracle_docs(x, cu, use_delta, dht=_np(dht))
    assert set(ref) == set(grads)
    for n in ref:
        close(n, grads[n], ref[n], rel_l2=0.01)


@pytest.mark.parametrize("dk,dv,E", [(64, 128, 4), (128, 64, 12), (64, 64, 16)])
def test_packed_backward_shapes(dk, dv, E):
    """Packed documents with d_k = 64 (zero-padded key rows) and more than eight slices."""
    lens = [70, 0, 129, 64, 3]
    x, cu = packed(lens, 2, dv, E, seed=dk + E, backward=True, dk=dk)
    gen = torch.Generator("cuda")
    gen.manual_seed(dk * E)
    dht = 0.5 * torch.randn(len(lens), 2, E, dk, dv, device="cuda", generator=gen)
    o, ht, ws = tla.tla_chunk_fwd(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"], x["beta"],
                                  x["h0"], save_for_bwd=True, cu_seqlens=cu)
    grads, _ = tla.tla_chunk_bwd(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"], x["dO"], ws,
                                 beta=x["beta"], h0=x["h0"], dht=dht, cu_seqlens=cu)
    torch.cuda.synchronize()
    assert tla.tla_last_device_status() == 0
    ro, rht, ref = oracle_docs(x, cu, True, dht=_np(dht))
    close("o", o, ro, rel_l2=0.01)
    close("ht", ht, rht, rel_l2=0.01)
    for n in ref:
        close(n, grads[n], ref[n], rel_l2=0.01)


def test_packed_equal_lengths_match_batched_exactly():
    """Three documents of 130 tokens packed = a batch of three sequences, bit for bit."""
    B, T, H, dv, E = 3, 130, 2, 128, 4
    x = inputs.chunk_inputs(B, T, H, 128, dv, E, dtype="bf16", h0_std=0.1, backward=True,
                            device="cuda", seed=11)
    o_b, ht_b, ws_b = tla.tla_chunk_fwd(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"],
                                        x["beta"], x["h0"], save_for_bwd=True)
    g_b, _ = tla.tla_chunk_bwd(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"], x["dO"], ws_b,
                               beta=x["beta"], h0=x["h0"])
    p = {n: (t.reshape(1, B * T, *t.shape[2:]) if n not in ("h0",) and t is not None else t)
         for n, t in x.items()}
    cu = [0, T, 2 * T, 3 * T]
    o_p, ht_p, ws_p = tla.tla_chunk_fwd(p["q"], p["k"], p["v"], p["q2"], p["k2"], p["g"],
                                        p["beta"], p["h0"], save_for_bwd=True, cu_seqlens=cu)
    g_p, _ = tla.tla_chunk_bwd(p["q"], p["k"], p["v"], p["q2"], p["k2"], p["g"], p["dO"], ws_p,
                               beta=p["beta"], h0=p["h0"], cu_seqlens=cu)
    torch.cuda.synchronize()
    assert torch.equal(o_p.reshape(o_b.shape), o_b)
    assert torch.equal(ht_p, ht_b)
    for n in g_b:
        assert torch.equal(g_p[n].reshape(g_b[n].shape), g_b[n]), n


def test_packed_off_the_tensor_core_path_is_refused():
    x, cu = inputs.packed_inputs([10, 20], 2, 32, 32, 4, dtype="fp32", device="cuda", seed=1)
    with pytest.raises(tla.TlaError) as ei:
        tla.tla_chunk_fwd(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"], x["beta"], None,
                          cu_seqlens=cu)
    assert ei.value.status == -2
