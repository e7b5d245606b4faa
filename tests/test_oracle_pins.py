"""Pins of the float64 oracle against facts the paper and the mathematics fix.

None of these tests re-types the oracle's own loop: each compares it with an
independent formulation (a textbook special case, the materialised attention
sum, the flattened joint-key matrix form, a hand-worked example, invariants,
finite differences, autograd of a separately written form).
"""
import json
import os

import numpy as np
import pytest
import torch

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def rnd(seed, B=1, T=37, H=2, dk=4, dv=3, E=3, unit=True, gate_scale=0.3):
    rng = np.random.default_rng(seed)

    def u(*s):
        x = rng.normal(size=s)
        return x / np.linalg.norm(x, axis=-1, keepdims=True) if unit else x

    d = dict(q=u(B, T, H, dk), k=u(B, T, H, dk), v=rng.normal(size=(B, T, H, dv)),
             q2=u(B, T, H, E), k2=u(B, T, H, E),
             g=-gate_scale * rng.random((B, T, H, E)),
             beta=1.0 / (1.0 + np.exp(-rng.normal(size=(B, T, H)))),
             h0=0.5 * rng.normal(size=(B, H, E, dk, dv)))
    return d


# --- (i) E = 1 with q' = k' = 1 is ordinary Gated DeltaNet / gated linear attention (Section 2.2, Eq. la3; Appendix D)

def textbook_gdn(q, k, v, alpha, beta, S0, delta):
    """Matrix-state Gated DeltaNet (delta=True) or scalar-gated LA, one head."""
    S = S0.copy()
    out = []
    for t in range(q.shape[0]):
        S = alpha[t] * S
        if delta:
            S = S + beta[t] * np.outer(k[t], v[t] - S.T @ k[t])
        else:
            S = S + beta[t] * np.outer(k[t], v[t])
        out.append(S.T @ q[t])
    return np.array(out), S


@pytest.mark.parametrize("delta", [True, False])
def test_e1_reduces_to_matrix_state(delta):
    d = rnd(1, E=1, H=2)
    d["q2"][:] = 1.0
    d["k2"][:] = 1.0
    o, ht = oracle.forward(d["q"], d["k"], d["v"], d["q2"], d["k2"], d["g"], d["beta"], d["h0"],
                           use_delta=delta)
    for h in range(2):
        oo, S = textbook_gdn(d["q"][0, :, h], d["k"][0, :, h], d["v"][0, :, h],
                             np.exp(d["g"][0, :, h, 0]), d["beta"][0, :, h], d["h0"][0, h, 0], delta)
        np.testing.assert_allclose(o[0, :, h], oo, rtol=0, atol=1e-12)
        np.testing.assert_allclose(ht[0, h, 0], S, rtol=0, atol=1e-12)


# --- (ii) without the delta rule the output is the materialised gated attention sum (Eq. la3 with Eq. forget3)

def test_materialised_sum_no_delta():
    d = rnd(2, T=29)
    o, _ = oracle.forward(d["q"], d["k"], d["v"], d["q2"], d["k2"], d["g"], d["beta"], d["h0"],
                          use_delta=False)
    B, T, H, dk = d["q"].shape
    Gg = np.cumsum(d["g"], axis=1)  # global inclusive log-decay
    ref = np.zeros_like(o)
    for h in range(H):
        for t in range(T):
            acc = np.zeros(d["v"].shape[-1])
            for e in range(d["q2"].shape[-1]):
                acc += d["q2"][0, t, h, e] * np.exp(Gg[0, t, h, e]) * (d["h0"][0, h, e].T @ d["q"][0, t, h])
            for s in range(t + 1):
                qk = d["q"][0, t, h] @ d["k"][0, s, h]
                w = sum(d["q2"][0, t, h, e] * d["k2"][0, s, h, e] * np.exp(Gg[0, t, h, e] - Gg[0, s, h, e])
                        for e in range(d["q2"].shape[-1]))
                acc += qk * w * d["beta"][0, s, h] * d["v"][0, s, h]
            ref[0, t, h] = acc
    np.testing.assert_allclose(o, ref, rtol=0, atol=1e-12)


# --- (iii) with the delta rule the recurrence is Gated DeltaNet on the joint key kappa = k (x) k' (Eq. gdn3flat)

def flat_gdn(q, k, v, q2, k2, alpha, beta, S0, delta=True):
    """Eq. gdn3flat: S = (I - beta kappa kappa^T) D S + beta kappa v^T, o = S^T (q (x) q').

    The flattened state row index is e*dk + i, so kappa = kron(k', k)."""
    E, dk, dv = S0.shape
    S = S0.reshape(E * dk, dv).copy()
    out = []
    for t in range(q.shape[0]):
        kap = np.kron(k2[t], k[t])
        qq = np.kron(q2[t], q[t])
        D = np.diag(np.repeat(alpha[t], dk))
        if delta:
            S = (np.eye(E * dk) - beta[t] * np.outer(kap, kap)) @ D @ S + beta[t] * np.outer(kap, v[t])
        else:
            S = D @ S + beta[t] * np.outer(kap, v[t])
        out.append(S.T @ qq)
    return np.array(out), S.reshape(E, dk, dv)


@pytest.mark.parametrize("delta", [True, False])
def test_flattened_joint_key(delta):
    d = rnd(3, T=41)
    o, ht = oracle.forward(d["q"], d["k"], d["v"], d["q2"], d["k2"], d["g"], d["beta"], d["h0"],
                           use_delta=delta)
    for h in range(2):
        oo, S = flat_gdn(d["q"][0, :, h], d["k"][0, :, h], d["v"][0, :, h], d["q2"][0, :, h],
                         d["k2"][0, :, h], np.exp(d["g"][0, :, h]), d["beta"][0, :, h], d["h0"][0, h],
                         delta)
        np.testing.assert_allclose(o[0, :, h], oo, rtol=0, atol=1e-12)
        np.testing.assert_allclose(ht[0, h], S, rtol=0, atol=1e-12)


# --- (iv) the chunkwise form (Appendix A, Eq. joint-chunk) reaches the token recurrence's result

@pytest.mark.parametrize("delta", [True, False])
@pytest.mark.parametrize("T,C", [(200, 64), (64, 64), (1, 64), (63, 64), (65, 64), (37, 8)])
def test_chunk_equals_token(delta, T, C):
    d = rnd(4, T=T, dk=5, dv=4, E=3)
    o, ht = oracle.forward(d["q"], d["k"], d["v"], d["q2"], d["k2"], d["g"], d["beta"], d["h0"],
                           use_delta=delta)
    oc, hc = oracle.chunk_forward(d["q"], d["k"], d["v"], d["q2"], d["k2"], d["g"], d["beta"],
                                  d["h0"], use_delta=delta, chunk=C)
    np.testing.assert_allclose(oc, o, rtol=0, atol=1e-11)
    np.testing.assert_allclose(hc, ht, rtol=0, atol=1e-11)


def test_chunk_equals_token_no_beta_no_h0():
    d = rnd(5, T=130)
    o, ht = oracle.forward(d["q"], d["k"], d["v"], d["q2"], d["k2"], d["g"], None, None, use_delta=False)
    oc, hc = oracle.chunk_forward(d["q"], d["k"], d["v"], d["q2"], d["k2"], d["g"], None, None,
                                  use_delta=False)
    np.testing.assert_allclose(oc, o, rtol=0, atol=1e-11)
    np.testing.assert_allclose(hc, ht, rtol=0, atol=1e-11)


# --- extreme within-chunk decay (Appendix A, "Numerical stability": e^-200 and e^-600 per chunk)

@pytest.mark.parametrize("total", [200.0, 600.0])
def test_extreme_gates_chunk_form(total):
    d = rnd(6, T=128, dk=4, dv=3, E=3)
    d["g"][..., 0] = -total / 64.0   # slice 0 decays by e^-total across one chunk
    o, ht = oracle.forward(d["q"], d["k"], d["v"], d["q2"], d["k2"], d["g"], d["beta"], d["h0"])
    oc, hc = oracle.chunk_forward(d["q"], d["k"], d["v"], d["q2"], d["k2"], d["g"], d["beta"], d["h0"])
    assert np.isfinite(oc).all() and np.isfinite(hc).all()
    np.testing.assert_allclose(oc, o, rtol=0, atol=1e-11)
    np.testing.assert_allclose(hc, ht, rtol=0, atol=1e-11)


# --- (v) delta rule: after the write, the read at the just-written unit joint key is (1-beta) kappa^T Shat + beta v

def test_delta_rule_read_at_written_key():
    d = rnd(7, T=20, dk=4, dv=3, E=3)
    o1, h_prev = oracle.forward(*(d[n][:, :-1] for n in ("q", "k", "v", "q2", "k2", "g")),
                                d["beta"][:, :-1], d["h0"])
    last = {n: d[n][:, -1:] for n in ("k", "v", "k2", "g", "beta")}
    # read the final state at the last token's joint key, through the oracle's own read:
    for beta_val in (1.0, 0.3):
        beta = np.full_like(last["beta"], beta_val)
        _, h_T = oracle.forward(last["k"], last["k"], last["v"], last["k2"], last["k2"], last["g"],
                                beta, h_prev)
        # append a read-only token: zero key writes nothing; queries = the written joint key
        zero_k = np.zeros_like(last["k"])
        o_read, _ = oracle.forward(last["k"], zero_k, last["v"], last["k2"], last["k2"],
                                   np.zeros_like(last["g"]), beta, h_T)
        alpha = np.exp(last["g"][0, 0])            # [H,E]
        for h in range(h_prev.shape[1]):
            kap = np.kron(last["k2"][0, 0, h], last["k"][0, 0, h])
            Shat = (h_prev[0, h] * alpha[h][:, None, None]).reshape(-1, h_prev.shape[-1])
            expect = (1 - beta_val) * (Shat.T @ kap) + beta_val * last["v"][0, 0, h]
            np.testing.assert_allclose(o_read[0, 0, h], expect, rtol=0, atol=1e-12)
            if beta_val == 1.0:
                np.testing.assert_allclose(o_read[0, 0, h], last["v"][0, 0, h], rtol=0, atol=1e-12)


# --- (vi) capacity: with orthonormal roles the state stores dk*E associations exactly (Section 2.2)

def test_capacity_orthonormal_roles():
    dk, dv, E = 4, 5, 3
    n = dk * E
    rng = np.random.default_rng(8)
    q = np.zeros((1, 2 * n, 1, dk)); k = np.zeros_like(q)
    q2 = np.zeros((1, 2 * n, 1, E)); k2 = np.zeros_like(q2)
    v = rng.normal(size=(1, 2 * n, 1, dv))
    vals = v[:, :n].copy()
    for t in range(n):
        i, e = t % dk, t // dk
        k[0, t, 0, i] = 1.0; k2[0, t, 0, e] = 1.0   # write phase
        q[0, n + t, 0, i] = 1.0; q2[0, n + t, 0, e] = 1.0  # read phase, zero key => no write
    g = np.zeros((1, 2 * n, 1, E))
    for delta in (False, True):
        o, _ = oracle.forward(q, k, v, q2, k2, g, None, None, use_delta=delta)
        np.testing.assert_allclose(o[:, n:], vals, rtol=0, atol=1e-13)
    # with dk*E + 1 associations the first one is overwritten (delta) or mixed (no delta)
    # is not asserted; capacity exactly dk*E is the claim.


# --- (vii) hand-worked single token with a non-zero initial state

def test_t1_hand_worked():
    with open(os.path.join(GOLDEN, "t1_closed_form.json")) as f:
        gold = json.load(f)
    x = gold["inputs"]
    sh = lambda a, *s: np.array(a, dtype=np.float64).reshape(*s)
    args = dict(q=sh(x["q"], 1, 1, 1, 2), k=sh(x["k"], 1, 1, 1, 2), v=sh(x["v"], 1, 1, 1, 2),
                q2=sh(x["q2"], 1, 1, 1, 2), k2=sh(x["k2"], 1, 1, 1, 2),
                g=np.log(sh(x["alpha"], 1, 1, 1, 2)), beta=sh([x["beta"]], 1, 1, 1),
                h0=sh(x["h0"], 1, 1, 2, 2, 2))
    for name, delta in (("delta", True), ("sgla", False)):
        o, ht = oracle.forward(**args, use_delta=delta)
        np.testing.assert_allclose(o.reshape(-1), gold["expected"][name]["o"], atol=1e-12)
        np.testing.assert_allclose(ht.reshape(2, 2, 2), gold["expected"][name]["ht"], atol=1e-12)
        oc, hc = oracle.chunk_forward(**args, use_delta=delta)
        np.testing.assert_allclose(oc.reshape(-1), gold["expected"][name]["o"], atol=1e-12)


# --- decode step is one token of the recurrence

@pytest.mark.parametrize("delta", [True, False])
def test_decode_steps_equal_forward(delta):
    d = rnd(9, T=6, H=3)
    o, ht = oracle.forward(d["q"], d["k"], d["v"], d["q2"], d["k2"], d["g"], d["beta"], d["h0"],
                           use_delta=delta)
    st = d["h0"].copy()
    for t in range(6):
        od, st = oracle.decode_step(st, *(d[n][:, t] for n in ("q", "k", "v", "q2", "k2", "g")),
                                    d["beta"][:, t], use_delta=delta)
        np.testing.assert_allclose(od, o[:, t], rtol=0, atol=1e-13)
    np.testing.assert_allclose(st, ht, rtol=0, atol=1e-13)


# --- backward: central finite differences of L = <o, dO> + <ht, dht>

def _loss(d, dO, dht, delta):
    o, ht = oracle.forward(d["q"], d["k"], d["v"], d["q2"], d["k2"], d["g"], d.get("beta"),
                           d.get("h0"), use_delta=delta)
    return float((o * dO).sum() + (ht * dht).sum())


@pytest.mark.parametrize("delta", [True, False])
def test_backward_finite_differences(delta):
    d = rnd(10, B=1, T=70, H=2, dk=3, dv=2, E=2)   # T spans the oracle's 64-token checkpoint segment
    rng = np.random.default_rng(11)
    dO = rng.normal(size=d["v"].shape)
    dht = rng.normal(size=d["h0"].shape)
    gr = oracle.backward(d["q"], d["k"], d["v"], d["q2"], d["k2"], d["g"], dO, d["beta"], d["h0"],
                         dht, use_delta=delta)
    eps = 1e-6
    names = {"q": "dq", "k": "dk", "v": "dv", "q2": "dq2", "k2": "dk2", "g": "dg",
             "beta": "dbeta", "h0": "dh0"}
    for x, gname in names.items():
        flat = d[x].reshape(-1)
        idx = rng.choice(flat.size, size=min(flat.size, 40), replace=False)
        for i in idx:
            keep = flat[i]
            flat[i] = keep + eps
            lp = _loss(d, dO, dht, delta)
            flat[i] = keep - eps
            lm = _loss(d, dO, dht, delta)
            flat[i] = keep
            fd = (lp - lm) / (2 * eps)
            an = gr[gname].reshape(-1)[i]
            assert abs(fd - an) <= 1e-6 * max(1.0, abs(fd)), (x, i, fd, an)


# --- backward: autograd of the independently written flattened form (Eq. gdn3flat) in torch

@pytest.mark.parametrize("delta", [True, False])
def test_backward_vs_autograd_flat(delta):
    d = rnd(12, B=2, T=67, H=1, dk=3, dv=4, E=2)
    rng = np.random.default_rng(13)
    dO = rng.normal(size=d["v"].shape)
    dht = rng.normal(size=d["h0"].shape)
    gr = oracle.backward(d["q"], d["k"], d["v"], d["q2"], d["k2"], d["g"], dO, d["beta"], d["h0"],
                         dht, use_delta=delta)
    t = {n: torch.tensor(a, dtype=torch.float64, requires_grad=True) for n, a in d.items()}
    B, T, H, dk = d["q"].shape
    E, dv = d["q2"].shape[-1], d["v"].shape[-1]
    loss = 0.0
    for b in range(B):
        S = t["h0"][b, 0].reshape(E * dk, dv)
        for s in range(T):
            kap = torch.kron(t["k2"][b, s, 0], t["k"][b, s, 0])
            qq = torch.kron(t["q2"][b, s, 0], t["q"][b, s, 0])
            D = torch.repeat_interleave(torch.exp(t["g"][b, s, 0]), dk)
            bt = t["beta"][b, s, 0]
            S = D[:, None] * S
            if delta:
                S = S - bt * torch.outer(kap, kap @ S) + bt * torch.outer(kap, t["v"][b, s, 0])
            else:
                S = S + bt * torch.outer(kap, t["v"][b, s, 0])
            loss = loss + (S.T @ qq) @ torch.tensor(dO[b, s, 0])
        loss = loss + (S.reshape(E, dk, dv) * torch.tensor(dht[b, 0])).sum()
    loss.backward()
    names = {"q": "dq", "k": "dk", "v": "dv", "q2": "dq2", "k2": "dk2", "g": "dg",
             "beta": "dbeta", "h0": "dh0"}
    for x, gname in names.items():
        np.testing.assert_allclose(gr[gname], t[x].grad.numpy(), rtol=1e-10, atol=1e-10,
                                   err_msg=x)


# --- layer input path and output gate (Algorithm 2; Appendix A, Input projections)

def _layer_inputs(seed, B=2, T=37, H=2, dk=8, dv=16, E=3, K=4):
    rng = np.random.default_rng(seed)
    C = 2 * dk + dv + 2 * E
    return dict(P=rng.standard_normal((B, T, H, C)), conv_w=0.5 * rng.standard_normal((H, C, K)),
                gate_in=rng.standard_normal((B, T, H, E)), gate_bias=rng.standard_normal((H, E)),
                A_log=0.3 * rng.standard_normal((H, E)), beta_in=rng.standard_normal((B, T, H))), \
        (dk, dv, E)


def _torch_prologue(x, dk, dv, E, eps=1e-6):
    """The same layer written with library routines: a grouped F.conv1d over a left-padded
    sequence (causal depthwise convolution), F.silu / F.softplus, torch reductions."""
    import torch.nn.functional as F
    P, w = x["P"], x["conv_w"]
    B, T, H, C = P.shape
    K = w.shape[-1]
    seq = P.permute(0, 2, 3, 1).reshape(B, H * C, T)
    a = F.conv1d(F.pad(seq, (K - 1, 0)), w.reshape(H * C, 1, K), groups=H * C)
    a = a.reshape(B, H, C, T).permute(0, 3, 1, 2)
    parts = torch.split(a, [dk, dk, dv, E, E], dim=-1)

    def unit(y):
        return y / torch.sqrt((y * y).sum(-1, keepdim=True) + eps)

    out = {"q": unit(F.silu(parts[0])), "k": unit(F.silu(parts[1])), "v": F.silu(parts[2]),
           "q2": unit(F.softplus(parts[3])), "k2": unit(F.softplus(parts[4])),
           "g": -torch.exp(x["A_log"]) * F.softplus(x["gate_in"] + x["gate_bias"]),
           "beta": torch.sigmoid(x["beta_in"])}
    return out


def test_layer_prologue_matches_library_form():
    x, (dk, dv, E) = _layer_inputs(1)
    ref = _torch_prologue({n: torch.tensor(a) for n, a in x.items()}, dk, dv, E)
    got = oracle.prologue(**x, dk=dk, dv=dv, E=E)
    for n in ref:
        np.testing.assert_allclose(got[n], ref[n].numpy(), rtol=0, atol=1e-12, err_msg=n)
    for n in ("q", "k", "q2", "k2"):   # unit vectors up to eps
        np.testing.assert_allclose(np.linalg.norm(got[n], axis=-1), 1.0, atol=1e-4)


def test_layer_prologue_is_causal():
    x, (dk, dv, E) = _layer_inputs(2)
    base = oracle.prologue(**x, dk=dk, dv=dv, E=E)
    y = dict(x)
    y["P"] = x["P"].copy()
    y["P"][:, 20:] += 3.0    # change every projection from token 20 on
    moved = oracle.prologue(**y, dk=dk, dv=dv, E=E)
    for n in ("q", "k", "v", "q2", "k2"):
        np.testing.assert_array_equal(moved[n][:, :20], base[n][:, :20])
        assert np.abs(moved[n][:, 20:] - base[n][:, 20:]).max() > 1e-3


def test_layer_prologue_backward_matches_autograd():
    x, (dk, dv, E) = _layer_inputs(3)
    tx = {n: torch.tensor(a, requires_grad=True) for n, a in x.items()}
    out = _torch_prologue(tx, dk, dv, E)
    rng = np.random.default_rng(4)
    cot = {n: rng.standard_normal(tuple(t.shape)) for n, t in out.items()}
    sum((out[n] * torch.tensor(cot[n])).sum() for n in out).backward()
    grads = {"d" + n: cot[n] for n in ("q", "k", "v", "q2", "k2", "g")}
    grads["dbeta"] = cot["beta"]
    got = oracle.prologue_backward(**x, grads=grads, dk=dk, dv=dv, E=E)
    pairs = {"dP": "P", "dconv_w": "conv_w", "dgate_in": "gate_in", "dgate_bias": "gate_bias",
             "dA_log": "A_log", "dbeta_in": "beta_in"}
    for gname, xname in pairs.items():
        np.testing.assert_allclose(got[gname], tx[xname].grad.numpy(), rtol=1e-9, atol=1e-10,
                                   err_msg=gname)


def test_output_gate_matches_library_form_and_autograd():
    rng = np.random.default_rng(5)
    o, z = rng.standard_normal((2, 9, 3, 32)), rng.standard_normal((2, 9, 3, 32))
    w = 1.0 + 0.1 * rng.standard_normal(32)
    to, tz, tw = (torch.tensor(a, requires_grad=True) for a in (o, z, w))
    ref = torch.nn.functional.rms_norm(to, (32,), tw, eps=1e-6) * torch.sigmoid(tz)
    np.testing.assert_allclose(oracle.gate_norm(o, z, w), ref.detach().numpy(), atol=1e-12)
    dy = rng.standard_normal(o.shape)
    (ref * torch.tensor(dy)).sum().backward()
    got = oracle.gate_norm_backward(o, z, w, dy)
    for gname, t in (("do", to), ("dz", tz), ("dw_norm", tw)):
        np.testing.assert_allclose(got[gname], t.grad.numpy(), rtol=1e-9, atol=1e-10, err_msg=gname)


def test_projection_is_the_per_channel_sum():
    """Input projection of Algorithm 2 (Appendix A, Input projections): every entry of
    P[b,t,h,c] is the explicit sum over the model width of u[b,t,i] W[h C + c, i], head h's
    rows of W in the order [q|k|v|q'|k'] (brute force on a tiny case)."""
    rng = np.random.default_rng(3)
    B, T, H, C, Dm = 2, 3, 2, 5, 7
    u = rng.standard_normal((B, T, Dm))
    W = rng.standard_normal((H * C, Dm))
    P = oracle.projection(u, W, H)
    assert P.shape == (B, T, H, C)
    for b in range(B):
        for t in range(T):
            for h in range(H):
                for c in range(C):
                    ref = 0.0
                    for i in range(Dm):
                        ref += u[b, t, i] * W[h * C + c, i]
                    assert abs(P[b, t, h, c] - ref) <= 1e-12 * (1 + abs(ref))
