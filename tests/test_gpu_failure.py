"""Failure detection on the GPU without a fault: a bounded device-side wait that nothing
satisfies gives up after its limit, the status word reports TLA_ERR_TIMEOUT once, and the
context keeps running the path (a forward through the tensor-core kernels then matches
the oracle)."""
import time

import numpy as np
import pytest
import torch

import oracle
from paper_2609_36529_gb300 import inputs, tla

pytestmark = pytest.mark.gpu

TLA_ERR_TIMEOUT = -4


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__ as ge
    ge.build()
    assert torch.cuda.is_available()


def test_bounded_wait_expires_and_is_reported_once():
    assert tla.tla_last_device_status() == 0
    t0 = time.perf_counter()
    tla.tla_selftest_bounded_wait(5_000_000)          # 5 ms limit
    status = tla.tla_last_device_status()             # synchronises the stream
    elapsed = time.perf_counter() - t0
    assert status == TLA_ERR_TIMEOUT
    assert elapsed >= 0.004                           # the wait ran to its limit
    assert elapsed < 5.0                              # and no further
    assert tla.tla_last_device_status() == 0          # the record is cleared on read


def test_context_usable_after_an_expired_wait():
    tla.tla_selftest_bounded_wait(1_000_000)
    assert tla.tla_last_device_status() == TLA_ERR_TIMEOUT
    x = inputs.chunk_inputs(1, 130, 2, 128, 64, 4, dtype="bf16", with_beta=True, h0_std=0.1,
                            device="cuda", seed=5)
    o, ht, _ = tla.tla_chunk_fwd(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"], x["beta"],
                                 x["h0"], use_delta=True, want_ht=True)
    torch.cuda.synchronize()
    assert tla.tla_last_device_status() == 0
    c = {n: (None if t is None else t.double().cpu().numpy()) for n, t in x.items()}
    ro, rht = oracle.forward(c["q"], c["k"], c["v"], c["q2"], c["k2"], c["g"], c["beta"], c["h0"],
                             use_delta=True)
    for got, ref in ((o, ro), (ht, rht)):
        got = got.double().cpu().numpy()
        rms = float(np.sqrt(np.mean(ref ** 2)))
        assert float(np.abs(got - ref).max()) <= 2e-2 * rms


def test_selftest_rejects_limits_out_of_range():
    with pytest.raises(tla.TlaError):
        tla.tla_selftest_bounded_wait(0)
    with pytest.raises(tla.TlaError):
        tla.tla_selftest_bounded_wait(2_000_000_000)
