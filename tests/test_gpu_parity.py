"""GPU parity: the CUDA path through the C ABI against the float64 oracle.

Tolerances (per output tensor, oracle as reference):
  fp32 inputs : max|err| <= 1e-4 * RMS(oracle)
  bf16 inputs : max|err| <= 2e-2 * RMS(oracle); gradients also rel. L2 < 1%
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


def close_rounded(name, got, ref, tol):
    """Results stored in bf16: allow the tolerance plus the output rounding (2^-8 |ref|)."""
    got = _np(got)
    ref = np.asarray(ref, dtype=np.float64)
    rms = float(np.sqrt(np.mean(ref ** 2)))
    excess = np.abs(got - ref) - (tol * rms + 2.0 ** -8 * np.abs(ref))
    assert np.isfinite(got).all() and excess.max() <= 0, f"{name}: exceeds by {excess.max():.3e}"


def run_fwd(x, use_delta, save=False):
    return tla.tla_chunk_fwd(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"], x["beta"], x["h0"],
                             use_delta=use_delta, save_for_bwd=save)


def oracle_fwd(x, use_delta):
    c = {n: _np(t) for n, t in x.items()}
    return oracle.forward(c["q"], c["k"], c["v"], c["q2"], c["k2"], c["g"], c["beta"], c["h0"],
                          use_delta=use_delta)


# --- the fp32 sGLA workload exactly as specified (B1 H2 T256 d32 E4, seed 0)

def test_sgla_fp32_workload_full():
    w = inputs.SGLA_FWD_FP32
    x = inputs.workload_inputs(w, device="cuda", seed=0)
    o, ht, _ = run_fwd(x, w.use_delta)
    torch.cuda.synchronize()
    ro, rht = oracle_fwd(x, w.use_delta)
    close("o", o, ro, TOL["fp32"])
    close("ht", ht, rht, TOL["fp32"])


# --- several chunks and ragged tails, both variants, both dtypes

@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
@pytest.mark.parametrize("use_delta", [True, False])
@pytest.mark.parametrize("T", [1, 63, 64, 65, 200])
def test_fwd_small(dtype, use_delta, T):
    x = inputs.chunk_inputs(2, T, 3, 64, 32, 3, dtype=dtype, with_beta=True, h0_std=0.2,
                            device="cuda", seed=T)
    o, ht, _ = run_fwd(x, use_delta)
    torch.cuda.synchronize()
    ro, rht = oracle_fwd(x, use_delta)
    close("o", o, ro, TOL[dtype])
    close("ht", ht, rht, TOL[dtype])


@pytest.mark.parametrize("dk,dv,E", [(16, 16, 1), (32, 64, 2), (64, 48, 5), (128, 128, 4),
                                     (48, 80, 16), (128, 128, 8), (128, 16, 16)])
def test_fwd_shapes(dk, dv, E):
    x = inputs.chunk_inputs(1, 150, 2, dk, dv, E, dtype="bf16", with_beta=True, h0_std=0.1,
                            device="cuda", seed=dk + dv + E)
    o, ht, _ = run_fwd(x, True)
    torch.cuda.synchronize()
    ro, rht = oracle_fwd(x, True)
    close("o", o, ro, TOL["bf16"])
    close("ht", ht, rht, TOL["bf16"])


@pytest.mark.parametrize("use_delta", [True, False])
@pytest.mark.parametrize("T,E", [(1, 4), (63, 1), (65, 8), (200, 4), (130, 16), (257, 6)])
def test_fwd_tensor_core_path(use_delta, T, E):
    """bf16, dk = 128: the tcgen05 recurrence (value blocks of 32 for E <= 4, else 16)."""
    x = inputs.chunk_inputs(2, T, 2, 128, 64, E, dtype="bf16", with_beta=True, h0_std=0.1,
                            device="cuda", seed=T * 31 + E)
    o, ht, _ = run_fwd(x, use_delta)
    torch.cuda.synchronize()
    assert tla.tla_last_device_status() == 0
    ro, rht = oracle_fwd(x, use_delta)
    close("o", o, ro, TOL["bf16"], rel_l2=0.01)
    close("ht", ht, rht, TOL["bf16"], rel_l2=0.01)


def test_fwd_sgla_no_beta_no_h0():
    x = inputs.chunk_inputs(2, 129, 2, 32, 32, 4, dtype="fp32", with_beta=False, device="cuda",
                            seed=5)
    o, ht, _ = run_fwd(x, False)
    torch.cuda.synchronize()
    ro, rht = oracle_fwd(x, False)
    close("o", o, ro, TOL["fp32"])
    close("ht", ht, rht, TOL["fp32"])


@pytest.mark.parametrize("total", [200.0, 600.0])
def test_fwd_extreme_gates(total):
    """Within-chunk decay of e^-200 and e^-600 in one slice (Appendix A, Numerical stability)."""
    x = inputs.chunk_inputs(1, 128, 2, 32, 32, 3, dtype="fp32", with_beta=True, h0_std=0.3,
                            device="cuda", seed=7)
    x["g"][..., 0] = -total / 64.0
    o, ht, _ = run_fwd(x, True)
    torch.cuda.synchronize()
    ro, rht = oracle_fwd(x, True)
    close("o", o, ro, TOL["fp32"])
    close("ht", ht, rht, TOL["fp32"])


@pytest.mark.parametrize("E", [4, 8])
@pytest.mark.parametrize("total", [200.0, 600.0])
def test_tensor_core_extreme_gates_fwd_bwd(E, total):
    """The same within-chunk decays (e^-200, e^-600 across one chunk in slice 0; slice 1
    decays by e^-600 in its first chunk only) through the tensor-core path: bf16 inputs,
    d_k = 128, prep, both recurrences and the chunk-gradient kernel.  Every product that
    sees the decay must stay finite and within the bf16 tolerance (Appendix A, Numerical
    stability: only non-positive exponents are ever formed)."""
    x = inputs.chunk_inputs(2, 200, 2, 128, 128, E, dtype="bf16", with_beta=True, h0_std=0.1,
                            backward=True, device="cuda", seed=int(total) + E)
    x["g"][..., 0] = -total / 64.0
    x["g"][:, :64, :, 1] = -600.0 / 64.0
    dht = 0.5 * torch.randn(2, 2, E, 128, 128, device="cuda",
                            generator=torch.Generator("cuda").manual_seed(E))
    o, ht, grads = run_bwd(x, True, dht)
    torch.cuda.synchronize()
    assert tla.tla_last_device_status() == 0
    ro, rht = oracle_fwd(x, True)
    close("o", o, ro, TOL["bf16"], rel_l2=0.01)
    close("ht", ht, rht, TOL["bf16"], rel_l2=0.01)
    ref = oracle_bwd(x, True, dht)
    assert set(ref) == set(grads)
    for n in ref:
        close(n, grads[n], ref[n], TOL["bf16"], rel_l2=0.01)


def test_bf16_outputs_within_tolerance_plus_rounding():
    x = inputs.chunk_inputs(2, 300, 3, 128, 128, 8, dtype="bf16", with_beta=True, h0_std=0.1,
                            backward=True, device="cuda", seed=17)
    o, ht, ws = tla.tla_chunk_fwd(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"], x["beta"],
                                  x["h0"], save_for_bwd=True, out_dtype=torch.bfloat16)
    grads, _ = tla.tla_chunk_bwd(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"], x["dO"], ws,
                                 beta=x["beta"], h0=x["h0"], out_dtype=torch.bfloat16)
    torch.cuda.synchronize()
    assert o.dtype == torch.bfloat16 and grads["dq"].dtype == torch.bfloat16
    ro, rht = oracle_fwd(x, True)
    close_rounded("o", o, ro, TOL["bf16"])
    close("ht", ht, rht, TOL["bf16"])
    ref = oracle_bwd(x, True, None)
    for n in ref:
        close_rounded(n, grads[n], ref[n], TOL["bf16"])


# --- backward

def run_bwd(x, use_delta, dht):
    o, ht, ws = run_fwd(x, use_delta, save=True)
    grads, _ = tla.tla_chunk_bwd(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"], x["dO"], ws,
                                 beta=x["beta"], h0=x["h0"], dht=dht, use_delta=use_delta)
    return o, ht, grads


def oracle_bwd(x, use_delta, dht):
    c = {n: _np(t) for n, t in x.items()}
    return oracle.backward(c["q"], c["k"], c["v"], c["q2"], c["k2"], c["g"], c["dO"], c["beta"],
                           c["h0"], _np(dht), use_delta=use_delta)


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
@pytest.mark.parametrize("use_delta", [True, False])
@pytest.mark.parametrize("T", [1, 65, 200])
def test_bwd_small(dtype, use_delta, T):
    x = inputs.chunk_inputs(2, T, 2, 32, 48, 3, dtype=dtype, with_beta=True, h0_std=0.2,
                            backward=True, device="cuda", seed=100 + T)
    dht = torch.randn(2, 2, 3, 32, 48, device="cuda",
                      generator=torch.Generator("cuda").manual_seed(T))
    _, _, grads = run_bwd(x, use_delta, dht)
    torch.cuda.synchronize()
    ref = oracle_bwd(x, use_delta, dht)
    assert set(ref) == set(grads)
    for n in ref:
        close(n, grads[n], ref[n], TOL[dtype], rel_l2=0.01 if dtype == "bf16" else None)


@pytest.mark.parametrize("use_delta", [True, False])
@pytest.mark.parametrize("T,E,dv", [(1, 4, 64), (64, 2, 64), (65, 4, 128), (200, 8, 64),
                                    (130, 1, 64), (90, 3, 64), (140, 6, 128), (150, 12, 128),
                                    (193, 16, 128)])
def test_bwd_tensor_core_path(use_delta, T, E, dv):
    """bf16, dk = 128: tcgen05 forward and backward recurrences (+ chunk gradients); every
    slice count the tensor-core path takes, E = 16 with its K dS' product in two halves."""
    x = inputs.chunk_inputs(2, T, 2, 128, dv, E, dtype="bf16", with_beta=True, h0_std=0.1,
                            backward=True, device="cuda", seed=1000 + T * 7 + E)
    dht = 0.5 * torch.randn(2, 2, E, 128, dv, device="cuda",
                            generator=torch.Generator("cuda").manual_seed(T + E))
    _, _, grads = run_bwd(x, use_delta, dht)
    torch.cuda.synchronize()
    assert tla.tla_last_device_status() == 0
    ref = oracle_bwd(x, use_delta, dht)
    assert set(ref) == set(grads)
    for n in ref:
        close(n, grads[n], ref[n], TOL["bf16"], rel_l2=0.01)


@pytest.mark.parametrize("use_delta", [True, False])
@pytest.mark.parametrize("T,E,dv", [(130, 4, 128), (200, 8, 64), (150, 16, 128), (64, 2, 64)])
def test_tensor_core_dk64(use_delta, T, E, dv):
    """d_k = 64 on the tensor-core kernels (key rows past 64 zero-filled by the copy engine):
    forward with h0 and final state, backward with dht and dh0, every output."""
    x = inputs.chunk_inputs(2, T, 2, 64, dv, E, dtype="bf16", with_beta=True, h0_std=0.1,
                            backward=True, device="cuda", seed=2000 + T + E)
    dht = 0.5 * torch.randn(2, 2, E, 64, dv, device="cuda",
                            generator=torch.Generator("cuda").manual_seed(T * E))
    o, ht, grads = run_bwd(x, use_delta, dht)
    torch.cuda.synchronize()
    assert tla.tla_last_device_status() == 0
    ro, rht = oracle_fwd(x, use_delta)
    close("o", o, ro, TOL["bf16"], rel_l2=0.01)
    close("ht", ht, rht, TOL["bf16"], rel_l2=0.01)
    ref = oracle_bwd(x, use_delta, dht)
    assert set(ref) == set(grads)
    for n in ref:
        close(n, grads[n], ref[n], TOL["bf16"], rel_l2=0.01)


def test_bwd_sgla_no_beta_no_h0():
    x = inputs.chunk_inputs(1, 150, 2, 32, 32, 4, dtype="fp32", with_beta=False, backward=True,
                            device="cuda", seed=11)
    _, _, grads = run_bwd(x, False, None)
    torch.cuda.synchronize()
    ref = oracle_bwd(x, False, None)
    assert set(ref) == set(grads)
    for n in ref:
        close(n, grads[n], ref[n], TOL["fp32"])


@pytest.mark.parametrize("dk,dv,E", [(128, 128, 4), (64, 32, 8), (16, 128, 1)])
def test_bwd_shapes(dk, dv, E):
    x = inputs.chunk_inputs(1, 130, 2, dk, dv, E, dtype="bf16", with_beta=True, h0_std=0.1,
                            backward=True, device="cuda", seed=dk * E)
    _, _, grads = run_bwd(x, True, None)
    torch.cuda.synchronize()
    ref = oracle_bwd(x, True, None)
    for n in ref:
        close(n, grads[n], ref[n], TOL["bf16"], rel_l2=0.01)


def test_bwd_deterministic():
    x = inputs.chunk_inputs(2, 190, 2, 64, 64, 4, dtype="bf16", with_beta=True, h0_std=0.1,
                            backward=True, device="cuda", seed=3)
    _, _, g1 = run_bwd(x, True, None)
    _, _, g2 = run_bwd(x, True, None)
    torch.cuda.synchronize()
    for n in g1:
        assert torch.equal(g1[n], g2[n]), n


# --- decode

@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
@pytest.mark.parametrize("use_delta", [True, False])
@pytest.mark.parametrize("dk,dv,E", [(128, 128, 8), (64, 48, 16), (16, 32, 1), (128, 128, 16)])
def test_decode_steps(dtype, use_delta, dk, dv, E):
    B, H = 3, 2
    gen = torch.Generator("cuda").manual_seed(dk + E)
    state = 0.1 * torch.randn(B, H, E, dk, dv, device="cuda", generator=gen)
    ref_state = _np(state)
    for step in range(4):
        d = inputs.decode_inputs(B, H, dk, dv, E, dtype=dtype, device="cuda", gen=gen)
        beta = d["beta"] if (use_delta or step % 2) else None
        o = tla.tla_decode_step(state, d["q"], d["k"], d["v"], d["q2"], d["k2"], d["g"], beta,
                                use_delta=use_delta)
        torch.cuda.synchronize()
        c = {n: _np(t) for n, t in d.items()}
        ro, ref_state = oracle.decode_step(ref_state, c["q"], c["k"], c["v"], c["q2"], c["k2"],
                                           c["g"], _np(beta), use_delta=use_delta)
        close(f"o step {step}", o, ro, TOL[dtype])
        close(f"state step {step}", state, ref_state, 1e-4)


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
@pytest.mark.parametrize("use_delta", [True, False])
def test_decode_many_heads(dtype, use_delta):
    """Many (b, h, 16-column) slabs, several waves of CTAs (dv = 48: three column blocks;
    E*dk = 512 rows), every output checked."""
    B, H, dk, dv, E = 40, 4, 128, 48, 4
    gen = torch.Generator("cuda").manual_seed(77)
    state = 0.1 * torch.randn(B, H, E, dk, dv, device="cuda", generator=gen)
    ref_state = _np(state)
    for step in range(3):
        d = inputs.decode_inputs(B, H, dk, dv, E, dtype=dtype, device="cuda", gen=gen)
        o = tla.tla_decode_step(state, d["q"], d["k"], d["v"], d["q2"], d["k2"], d["g"], d["beta"],
                                use_delta=use_delta)
        torch.cuda.synchronize()
        c = {n: _np(t) for n, t in d.items()}
        ro, ref_state = oracle.decode_step(ref_state, c["q"], c["k"], c["v"], c["q2"], c["k2"],
                                           c["g"], c["beta"], use_delta=use_delta)
        if dtype == "fp32":
            close(f"o step {step}", o, ro, TOL["fp32"])
        else:   # bf16-stored o: the tolerance plus its own rounding
            close_rounded(f"o step {step}", o, ro, TOL["bf16"])
        close(f"state step {step}", state, ref_state, 1e-4)


def test_decode_after_chunk_prefill_matches_token_recurrence():
    """Prefill by the chunk forward, then decode: equals the oracle's recurrence over all tokens."""
    x = inputs.chunk_inputs(2, 70, 2, 64, 64, 4, dtype="fp32", with_beta=True, device="cuda",
                            seed=21)
    _, ht, _ = run_fwd({n: (t[:, :64].contiguous() if t is not None and t.dim() >= 3 and t.shape[1] == 70
                            else t) for n, t in x.items()}, True)
    outs = []
    for t in range(64, 70):
        outs.append(tla.tla_decode_step(ht, *(x[n][:, t].contiguous() for n in
                                              ("q", "k", "v", "q2", "k2", "g")),
                                        x["beta"][:, t].contiguous()))
    torch.cuda.synchronize()
    ro, rht = oracle_fwd(x, True)
    close("decode o", torch.stack(outs, 1), ro[:, 64:], TOL["fp32"])
    close("final state", ht, rht, TOL["fp32"])


# --- full-size workloads in the launch configuration the benchmark times, sampled heads

def _sample_heads(x, bh_list, T=None):
    """Slice inputs down to the listed (b, h) pairs (as a batch of single-head problems)."""
    out = {}
    for n, t in x.items():
        if t is None:
            out[n] = None
        elif n == "h0":
            out[n] = torch.stack([t[b, h] for b, h in bh_list])[:, None]
        elif n == "beta":
            out[n] = torch.stack([t[b, :T, h] for b, h in bh_list])[:, :, None]
        else:
            out[n] = torch.stack([t[b, :T, h] for b, h in bh_list])[:, :, None]
    return out


@pytest.mark.parametrize("name", ["gdn_fwd_bf16_B4_H16_T4096_d128_E8",
                                  "gdn_fwd_bf16_B1_H32_T65536_d128_E16"])
def test_full_size_forward_sampled(name):
    """The two forward-only workloads as the benchmark launches them, every output of the
    sampled heads over the whole sequence (65,536 tokens for the long-context one, whose
    chain runs through 1024 chunks of the E = 16 recurrence) and their final states."""
    w = inputs.WORKLOADS[name]
    x = inputs.workload_inputs(w, device="cuda", seed=0)
    o, ht, _ = run_fwd(x, w.use_delta)
    torch.cuda.synchronize()
    assert tla.tla_last_device_status() == 0
    # heads are independent: the oracle runs only the sampled ones, one host thread each
    picks = [(0, 0), (w.B - 1, w.H - 1), (w.B // 2, w.H // 2), (0, w.H // 4)]
    xs = _sample_heads(x, picks)
    o_s = torch.stack([o[b, :, h] for b, h in picks]).cpu()
    ht_s = torch.stack([ht[b, h] for b, h in picks]).cpu()
    del o, ht, x
    ro, rht = oracle_fwd(xs, w.use_delta)
    for i, (b, h) in enumerate(picks):
        close(f"o b{b}h{h}", o_s[i], ro[i, :, 0], TOL[w.dtype], rel_l2=0.01)
        close(f"ht b{b}h{h}", ht_s[i], rht[i, 0], TOL[w.dtype], rel_l2=0.01)
        # the end of the sequence on its own: the error must not grow along the chain
        close(f"o[-4096:] b{b}h{h}", o_s[i, -4096:], ro[i, -4096:, 0], TOL[w.dtype])


@pytest.mark.parametrize("out_dtype", [torch.float32, torch.bfloat16])
def test_full_size_fwd_bwd_sampled(out_dtype):
    """The headline workload as the benchmark launches it (bf16 o and input gradients; fp32
    too), two sampled heads against the oracle."""
    w = inputs.GDN_FWDBWD_BF16
    x = inputs.workload_inputs(w, device="cuda", seed=0)
    o, _, ws = tla.tla_chunk_fwd(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"], x["beta"],
                                 None, use_delta=True, save_for_bwd=True, want_ht=False,
                                 out_dtype=out_dtype)
    grads, _ = tla.tla_chunk_bwd(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"], x["dO"], ws,
                                 beta=x["beta"], use_delta=True, out_dtype=out_dtype)
    torch.cuda.synchronize()
    del ws
    picks = [(0, 0), (w.B - 1, w.H - 1)]
    xs = _sample_heads(x, picks)
    ro, _ = oracle_fwd(xs, True)
    ref = oracle_bwd(xs, True, None)
    bf16_out = out_dtype == torch.bfloat16
    for i, (b, h) in enumerate(picks):
        if bf16_out:   # bf16-stored results: the tolerance plus their own rounding
            close_rounded(f"o b{b}h{h}", o[b, :, h], ro[i, :, 0], TOL["bf16"])
        else:
            close(f"o b{b}h{h}", o[b, :, h], ro[i, :, 0], TOL["bf16"])
        for n in ("dq", "dk", "dv", "dq2", "dk2", "dg"):
            got, r = grads[n][b, :, h], ref[n][i, :, 0]
            if bf16_out and n != "dg":
                close_rounded(f"{n} b{b}h{h}", got, r, TOL["bf16"])
                close(f"{n} b{b}h{h} rel L2", got, r, 1.0, rel_l2=0.01)
            else:
                close(f"{n} b{b}h{h}", got, r, TOL["bf16"], rel_l2=0.01)
        close(f"dbeta b{b}h{h}", grads["dbeta"][b, :, h], ref["dbeta"][i, :, 0], TOL["bf16"],
              rel_l2=0.01)


def test_full_size_decode_sampled():
    w = inputs.DECODE
    gen = torch.Generator("cuda").manual_seed(0)
    state = 0.05 * torch.randn(w.B, w.H, w.E, w.dk, w.dv, device="cuda", generator=gen)
    picks = [(0, 0), (w.B - 1, w.H - 1), (w.B // 2, 5)]
    ref = np.stack([_np(state[b, h]) for b, h in picks])[:, None]
    for step in range(3):
        d = inputs.decode_inputs(w.B, w.H, w.dk, w.dv, w.E, device="cuda", gen=gen)
        o = tla.tla_decode_step(state, d["q"], d["k"], d["v"], d["q2"], d["k2"], d["g"], d["beta"])
        torch.cuda.synchronize()
        c = {n: np.stack([_np(t[b, h]) for b, h in picks])[:, None] for n, t in d.items()}
        ro, ref = oracle.decode_step(ref, c["q"], c["k"], c["v"], c["q2"], c["k2"], c["g"],
                                     c["beta"])
        for i, (b, h) in enumerate(picks):
            close(f"o step{step} b{b}h{h}", o[b, h], ro[i, 0], TOL["fp32"])
            close(f"state step{step} b{b}h{h}", state[b, h], ref[i, 0], 1e-4)


@pytest.mark.parametrize("use_delta", [False, True])
def test_full_size_decode_after_prefill(use_delta):
    """The decode workload as the benchmark runs it: the fp32 state [256,32,8,128,128] filled
    by a 512-token chunked prefill (tensor-core forward, bf16 inputs), then 100 consecutive
    decode steps with bf16 inputs and outputs, for sGLA and GDN.  Sampled heads follow the
    oracle's token recurrence over all 612 tokens: o at every step, the state every 25 steps."""
    w = inputs.DECODE
    gen = torch.Generator("cuda").manual_seed(1000 + int(use_delta))
    state = torch.empty(w.B, w.H, w.E, w.dk, w.dv, dtype=torch.float32, device="cuda")
    pre = inputs.chunk_inputs(w.B, w.prefill, w.H, w.dk, w.dv, w.E, dtype="bf16",
                              with_beta=True, device="cuda", gen=gen)
    tla.tla_chunk_fwd(pre["q"], pre["k"], pre["v"], pre["q2"], pre["k2"], pre["g"], pre["beta"],
                      None, use_delta=use_delta, ht=state)
    torch.cuda.synchronize()
    assert tla.tla_last_device_status() == 0
    picks = [(0, 0), (w.B - 1, w.H - 1), (w.B // 2, 5), (37, 17)]
    _, ref = oracle_fwd(_sample_heads(pre, picks), use_delta)
    del pre
    close("state after prefill", torch.stack([state[b, h] for b, h in picks])[:, None], ref,
          TOL["bf16"], rel_l2=0.01)
    o = torch.empty(w.B, w.H, w.dv, dtype=torch.bfloat16, device="cuda")
    for step in range(w.steps):
        d = inputs.decode_inputs(w.B, w.H, w.dk, w.dv, w.E, dtype="bf16", device="cuda", gen=gen)
        tla.tla_decode_step(state, d["q"], d["k"], d["v"], d["q2"], d["k2"], d["g"], d["beta"],
                            use_delta=use_delta, o=o)
        c = {n: np.stack([_np(t[b, h]) for b, h in picks])[:, None] for n, t in d.items()}
        ro, ref = oracle.decode_step(ref, c["q"], c["k"], c["v"], c["q2"], c["k2"], c["g"],
                                     c["beta"], use_delta=use_delta)
        got = torch.stack([o[b, h] for b, h in picks])[:, None]
        close_rounded(f"o step {step}", got, ro, TOL["bf16"])
        if step % 25 == 24:
            close(f"state step {step}", torch.stack([state[b, h] for b, h in picks])[:, None],
                  ref, TOL["bf16"], rel_l2=0.01)
    assert tla.tla_last_device_status() == 0
