"""GPU test of tla_chunk_fwd_noalloc, the forward that allocates nothing.

Callers that cannot allocate device memory (a host runtime owning all device
memory, a serving process that forbids allocation after start-up) use this
entry point; its workspace is a fixed buffer inside the library.  It must give
the same results as tla_chunk_fwd with a caller-provided workspace, call after
call (the buffer keeps the previous call's contents).  This file is collected
last so a stop-at-first-failure run has already run every other test.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2609_36529_gb300 import inputs, tla

pytestmark = pytest.mark.gpu

TOL = {"fp32": 1e-4, "bf16": 2e-2}


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__ as ge
    ge.build_library()
    assert torch.cuda.is_available()


def _close(got, ref, tol):
    got = got.double().cpu().numpy()
    ref = ref.double().cpu().numpy()
    rms = float(np.sqrt(np.mean(ref ** 2)))
    assert np.isfinite(got).all()
    assert float(np.abs(got - ref).max()) <= tol * rms


@pytest.mark.parametrize("dtype,dk,E,use_delta", [("bf16", 128, 4, True), ("fp32", 64, 3, False)])
def test_noalloc_matches_workspace_forward_twice(dtype, dk, E, use_delta):
    L = tla.lib()
    for call in range(2):   # two calls in a row on different inputs
        x = inputs.chunk_inputs(2, 300 + 37 * call, 3, dk, 64, E, dtype=dtype, with_beta=True,
                                h0_std=0.1, device="cuda", seed=50 + call)
        o_ref, ht_ref, _ = tla.tla_chunk_fwd(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"],
                                             x["beta"], x["h0"], use_delta=use_delta)
        o = torch.empty_like(o_ref)
        ht = torch.empty_like(ht_ref)
        p = tla.make_problem(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"], x["beta"],
                             x["h0"], o, ht, use_delta)
        need = L.tla_fwd_workspace_bytes(ctypes.byref(p), 0)
        assert 0 < need <= L.tla_noalloc_scratch_bytes()
        st = L.tla_chunk_fwd_noalloc(ctypes.byref(p),
                                     ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
        assert st == 0, tla.STATUS.get(st, st)
        torch.cuda.synchronize()
        assert tla.tla_last_device_status() == 0
        _close(o, o_ref, TOL[dtype])
        _close(ht, ht_ref, TOL[dtype])
