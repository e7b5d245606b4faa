"""The kernels under torch.autograd: gradients through the binding against the float64
oracle's backward, and a short MQAR training run (Section 2.3, Appendix C) that must learn."""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2609_36529_gb300 import inputs
from paper_2609_36529_gb300.autograd import triadic_linear_attention

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__ as ge
    ge.build()
    assert torch.cuda.is_available()


def _np(t):
    return None if t is None else t.detach().double().cpu().numpy()


@pytest.mark.parametrize("use_delta", [True, False])
def test_autograd_gradients_match_oracle(use_delta):
    x = inputs.chunk_inputs(2, 70, 2, 16, 16, 4, dtype="fp32", with_beta=True, h0_std=0.1,
                            backward=True, device="cuda", seed=4)
    names = ("q", "k", "v", "q2", "k2", "g", "beta", "h0")
    leaf = {n: x[n].clone().requires_grad_() for n in names}
    o, ht = triadic_linear_attention(*(leaf[n] for n in names), use_delta=use_delta)
    gen = torch.Generator("cuda").manual_seed(9)
    wh = torch.randn(ht.shape, device="cuda", generator=gen)
    ((o * x["dO"]).sum() + (ht * wh).sum()).backward()
    c = {n: _np(x[n]) for n in names}
    ro, rht = oracle.forward(*(c[n] for n in names), use_delta=use_delta)
    ref = oracle.backward(c["q"], c["k"], c["v"], c["q2"], c["k2"], c["g"], _np(x["dO"]),
                          c["beta"], c["h0"], _np(wh), use_delta=use_delta)
    for name, got, want in [("o", o, ro), ("ht", ht, rht)] + \
            [("d" + n, leaf[n].grad, ref["d" + n]) for n in names]:
        got = _np(got)
        rms = float(np.sqrt(np.mean(want ** 2)))
        assert np.isfinite(got).all(), name
        assert float(np.abs(got - want).max()) <= 1e-4 * rms, name


def test_mqar_model_memorises_a_batch():
    """The reduced MQAR model trained on one fixed batch through the kernels' backward:
    the loss must fall far below chance (ln 256 = 5.5) -- the gradients flow end to end."""
    import mqar
    first, last, acc = mqar.train(E=4, N=32, steps=120, batch=16, n_keys=256, n_vals=256,
                                  lr=3e-3, fixed_batch=True)
    assert math.isfinite(first) and math.isfinite(last)
    assert last < 0.5 * first, (first, last)
    assert 0.0 <= acc <= 1.0
