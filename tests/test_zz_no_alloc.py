"""GPU test of tla_chunk_fwd_noalloc, the forward that allocates nothing.

Callers that cannot allocate device memory (a host runtime owning all device
memory, a serving process that forbids allocation after start-up) use this
entry point; its workspace is a fixed buffer inside the library.  The same
kernels run on the same inputs as tla_chunk_fwd with a caller-provided
workspace, so the results must be bit-identical, call after call (the buffer
keeps the previous call's contents).  This file is collected last so a
stop-at-first-failure run has already run every other test.
"""
import ctypes

import pytest
import torch

from paper_2609_36529_gb300 import inputs, tla

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__ as ge
    ge.build_library()
    assert torch.cuda.is_available()


def _noalloc_abi(x, o, ht, use_delta, cu_seqlens=None):
    """Call the entry point straight through the C ABI."""
    L = tla.lib()
    p = tla.make_problem(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"], x["beta"],
                         x["h0"], o, ht, use_delta, cu_seqlens=cu_seqlens)
    need = L.tla_fwd_workspace_bytes(ctypes.byref(p), 0)
    assert 0 < need <= L.tla_noalloc_scratch_bytes()
    return L.tla_chunk_fwd_noalloc(ctypes.byref(p),
                                   ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))


@pytest.mark.parametrize("dtype,dk,E,use_delta", [("bf16", 128, 4, True), ("fp32", 64, 3, False)])
def test_noalloc_matches_workspace_forward_twice(dtype, dk, E, use_delta):
    for call in range(2):   # two calls in a row on different inputs
        x = inputs.chunk_inputs(2, 300 + 37 * call, 3, dk, 64, E, dtype=dtype, with_beta=True,
                                h0_std=0.1, device="cuda", seed=50 + call)
        o_ref, ht_ref, _ = tla.tla_chunk_fwd(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"],
                                             x["beta"], x["h0"], use_delta=use_delta)
        o = torch.empty_like(o_ref)
        ht = torch.empty_like(ht_ref)
        st = _noalloc_abi(x, o, ht, use_delta)
        assert st == 0, tla.STATUS.get(st, st)
        torch.cuda.synchronize()
        assert tla.tla_last_device_status() == 0
        assert torch.equal(o, o_ref)
        assert torch.equal(ht, ht_ref)


def test_noalloc_wrapper_defaults_and_packed_documents():
    """The Python wrapper (same defaults as tla_chunk_fwd: final state returned, o in the
    requested dtype) and a packed-document call through the C ABI, twice each."""
    for call in range(2):
        x = inputs.chunk_inputs(1, 260, 2, 128, 128, 4, dtype="bf16", with_beta=True,
                                h0_std=0.1, device="cuda", seed=70 + call)
        o_ref, ht_ref, _ = tla.tla_chunk_fwd(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"],
                                             x["beta"], x["h0"], out_dtype=torch.bfloat16)
        o, ht = tla.tla_chunk_fwd_noalloc(x["q"], x["k"], x["v"], x["q2"], x["k2"], x["g"],
                                          x["beta"], x["h0"], out_dtype=torch.bfloat16)
        torch.cuda.synchronize()
        assert ht is not None and o.dtype == torch.bfloat16
        assert torch.equal(o, o_ref) and torch.equal(ht, ht_ref)

        lens = [70, 0, 129 + call, 64, 200 - call]
        xp, cu = inputs.packed_inputs(lens, 2, 128, 128, 4, dtype="bf16", h0_std=0.1,
                                      device="cuda", seed=80 + call)
        o_ref, ht_ref, _ = tla.tla_chunk_fwd(xp["q"], xp["k"], xp["v"], xp["q2"], xp["k2"],
                                             xp["g"], xp["beta"], xp["h0"], cu_seqlens=cu)
        o = torch.empty_like(o_ref)
        ht = torch.empty_like(ht_ref)
        st = _noalloc_abi(xp, o, ht, True, cu_seqlens=cu)
        assert st == 0, tla.STATUS.get(st, st)
        torch.cuda.synchronize()
        assert tla.tla_last_device_status() == 0
        assert torch.equal(o, o_ref) and torch.equal(ht, ht_ref)
