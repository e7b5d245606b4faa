"""Host-side checks of the C-ABI library (no GPU needed, no compute calls)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def header_functions():
    src = open(os.path.join(ROOT, "include", "tla.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(tla_[a-z0-9_]+)\s*\(", src)))


@pytest.fixture(scope="module")
def tla():
    import __graft_entry__ as ge
    ge.build_library()
    from paper_2609_36529_gb300 import tla as t
    return t


def test_library_exports_every_declared_symbol(tla):
    L = tla.lib()
    names = header_functions()
    assert {"tla_chunk_fwd", "tla_chunk_bwd", "tla_decode_step"} <= set(names)
    for n in names:
        assert hasattr(L, n), n
    assert set(tla.EXPORTED) <= set(names)


def test_status_strings(tla):
    for code, name in tla.STATUS.items():
        assert tla.lib().tla_status_string(code).decode() == name
    assert tla.tla_version().startswith("tla")


def _problem(tla, **kw):
    p = tla.tla_problem()
    p.B, p.T, p.H, p.dk, p.dv, p.E, p.chunk, p.dtype, p.use_delta = 2, 100, 3, 64, 32, 4, 64, 0, 1
    p.out_dtype = 1
    fake = ctypes.c_void_p(0x1000)
    for n in ("q", "k", "v", "q2", "k2", "g", "beta", "o"):
        setattr(p, n, fake)
    for n, v in kw.items():
        setattr(p, n, v)
    return p


def test_host_validation_rejects_before_launch(tla):
    L = tla.lib()
    cases = [
        (dict(chunk=32), -2), (dict(dk=20), -2), (dict(dv=256), -2), (dict(E=33), -2),
        (dict(E=17, dk=128), -2), (dict(gate_per_head=2), -1),
        (dict(E=0), -1), (dict(T=0), -1), (dict(dtype=7), -1), (dict(use_delta=2), -1),
        (dict(out_dtype=3), -1),
        (dict(q=None), -1), (dict(beta=None), -1), (dict(o=None), -1),
    ]
    for kw, want in cases:
        p = _problem(tla, **kw)
        assert L.tla_chunk_fwd(ctypes.byref(p), None, 0, 0, None) == want, kw
        assert L.tla_fwd_workspace_bytes(ctypes.byref(p), 0) == 0
    # valid problem, missing or short workspace: rejected before any launch
    p = _problem(tla)
    need = L.tla_fwd_workspace_bytes(ctypes.byref(p), 1)
    assert need > 0 and need % 256 == 0
    assert L.tla_chunk_fwd(ctypes.byref(p), None, need, 1, None) == -5
    assert L.tla_chunk_fwd(ctypes.byref(p), ctypes.c_void_p(0x100000), need - 1, 1, None) == -5
    assert L.tla_chunk_fwd(ctypes.byref(p), ctypes.c_void_p(0x100010), need, 1, None) == -5
    # sGLA may omit beta
    p = _problem(tla, use_delta=0, beta=None)
    assert L.tla_fwd_workspace_bytes(ctypes.byref(p), 0) > 0


def test_host_validation_bwd_and_decode(tla):
    L = tla.lib()
    p = _problem(tla)
    f = ctypes.c_void_p(0x1000)
    # dbeta must be given iff beta is
    assert L.tla_chunk_bwd(ctypes.byref(p), f, 1 << 40, f, None, f, f, f, f, f, None, f, None,
                           f, 1 << 40, None) == -1
    # h0 absent => dh0 must be NULL
    assert L.tla_chunk_bwd(ctypes.byref(p), f, 1 << 40, f, None, f, f, f, f, f, f, f, f,
                           f, 1 << 40, None) == -1
    # short forward workspace
    assert L.tla_chunk_bwd(ctypes.byref(p), None, 0, f, None, f, f, f, f, f, f, f, None,
                           f, 1 << 40, None) == -5
    # decode: misaligned state, unsupported dims, missing beta with the delta rule
    assert L.tla_decode_step(2, 2, 64, 64, 4, 1, 0, f, f, f, f, f, f, f, ctypes.c_void_p(0x1004),
                             f, None) == -1
    assert L.tla_decode_step(2, 2, 64, 200, 4, 1, 0, f, f, f, f, f, f, f, f, f, None) == -2
    assert L.tla_decode_step(2, 2, 64, 64, 33, 1, 0, f, f, f, f, f, f, f, f, f, None) == -2
    assert L.tla_decode_step(2, 2, 128, 64, 32, 1, 0, f, f, f, f, f, f, f, f, f, None) == -2
    assert L.tla_decode_step(2, 2, 64, 64, 4, 1, 0, f, f, f, f, f, f, None, f, f, None) == -1


def test_workspace_sizes_grow_with_saving(tla):
    L = tla.lib()
    p = _problem(tla)
    a = L.tla_fwd_workspace_bytes(ctypes.byref(p), 0)
    b = L.tla_fwd_workspace_bytes(ctypes.byref(p), 1)
    assert b > a > 0
    assert L.tla_bwd_workspace_bytes(ctypes.byref(p)) > 0


def test_noalloc_entry_rejects_on_host(tla):
    """The no-allocation forward rejects bad or oversized problems before any launch."""
    L = tla.lib()
    cap = L.tla_noalloc_scratch_bytes()
    assert cap == 64 << 20
    p = _problem(tla, chunk=32)
    assert L.tla_chunk_fwd_noalloc(ctypes.byref(p), None) == -2
    p = _problem(tla, B=64, T=8192, H=16, dk=128, dv=128)   # workspace far above the buffer
    assert L.tla_fwd_workspace_bytes(ctypes.byref(p), 0) > cap
    assert L.tla_chunk_fwd_noalloc(ctypes.byref(p), None) == -5


def test_packed_documents_validation(tla):
    """cu_seqlens (Appendix A, Kernels: packed documents) is checked on the host."""
    L = tla.lib()

    def packed(cu, **kw):
        args = dict(B=1, T=cu[-1])
        args.update(kw)
        p = _problem(tla, **args)
        arr = (ctypes.c_int * len(cu))(*cu)
        p._keep = arr
        p.cu_seqlens = ctypes.cast(arr, ctypes.POINTER(ctypes.c_int))
        p.n_docs = len(cu) - 1
        return p

    ok = packed([0, 10, 10, 100])   # an empty document is allowed
    need = L.tla_fwd_workspace_bytes(ctypes.byref(ok), 1)
    assert need > 0 and need % 256 == 0
    # each document starts its own chunks: 1 + 0 + 2 chunks instead of 2 for 100 tokens
    plain = _problem(tla, B=1, T=100)
    assert need > L.tla_fwd_workspace_bytes(ctypes.byref(plain), 1)
    bad = [packed([1, 10, 100]), packed([0, 50, 40, 100]), packed([0, 10, 99], T=100),
           packed([0, 100], B=2)]
    for p in bad:
        assert L.tla_fwd_workspace_bytes(ctypes.byref(p), 1) == 0
        assert L.tla_chunk_fwd(ctypes.byref(p), None, 0, 0, None) == -1
    p = packed([0, 100])
    p.n_docs = 0
    assert L.tla_chunk_fwd(ctypes.byref(p), None, 0, 0, None) == -1
    # packed documents run on the tensor-core path only (d_k = 64 or 128; here d_k = 32):
    # refused before a launch
    small = packed([0, 10, 10, 100], dk=32)
    need32 = L.tla_fwd_workspace_bytes(ctypes.byref(small), 1)
    assert L.tla_chunk_fwd(ctypes.byref(small), ctypes.c_void_p(0x100000), need32, 1, None) == -2


def test_layer_io_validation(tla):
    """Input prologue and output gate (Algorithm 2): argument checks before any launch."""
    L = tla.lib()
    f = ctypes.c_void_p(0x1000)

    def prologue(**kw):
        a = tla.tla_prologue_args()
        a.B, a.T, a.H, a.dk, a.dv, a.E, a.K, a.dtype, a.eps = 2, 100, 3, 64, 64, 4, 4, 0, 1e-6
        for n in ("P", "conv_w", "gate_in", "gate_bias", "A_log", "beta_in", "q", "k", "v",
                  "q2", "k2", "g", "beta"):
            setattr(a, n, f)
        for n, v in kw.items():
            setattr(a, n, v)
        return a

    for kw, want in [(dict(K=5), -2), (dict(K=0), -1), (dict(E=33), -2), (dict(dk=20), -2),
                     (dict(beta=None), -1), (dict(P=None), -1), (dict(eps=0.0), -1),
                     (dict(dtype=5), -1), (dict(q=ctypes.c_void_p(0x1004)), -1)]:
        assert L.tla_layer_prologue(ctypes.byref(prologue(**kw)), None) == want, kw
    ok = prologue()
    need = L.tla_layer_prologue_bwd_workspace_bytes(ctypes.byref(ok))
    assert need > 0 and need % 256 == 0
    args = [f] * 14
    assert L.tla_layer_prologue_bwd(ctypes.byref(ok), 1, *args[:13], None, need, None) == -5
    assert L.tla_layer_prologue_bwd(ctypes.byref(ok), 3, *args, need, None) == -1

    def gate(**kw):
        a = tla.tla_gate_args()
        a.B, a.T, a.H, a.dv, a.o_dtype, a.dtype, a.eps = 2, 10, 3, 64, 1, 0, 1e-6
        for n in ("o", "z", "w_norm", "y"):
            setattr(a, n, f)
        for n, v in kw.items():
            setattr(a, n, v)
        return a

    for kw, want in [(dict(dv=20), -2), (dict(o=None), -1), (dict(o_dtype=9), -1),
                     (dict(eps=-1.0), -1)]:
        assert L.tla_output_gate(ctypes.byref(gate(**kw)), None) == want, kw
    g = gate()
    need = L.tla_output_gate_bwd_workspace_bytes(ctypes.byref(g))
    assert need > 0
    assert L.tla_output_gate_bwd(ctypes.byref(g), f, f, f, f, None, need, None) == -5


def test_selftest_limit_checked_on_host(tla):
    L = tla.lib()
    for bad in (0, 1_000_000_001, 2 ** 63):
        assert L.tla_selftest_bounded_wait(bad, None) == -1


def test_projection_validation(tla):
    """Fused input projection (Algorithm 2): argument checks before any launch."""
    L = tla.lib()
    f = ctypes.c_void_p(0x1000)

    def args(**kw):
        a = tla.tla_projection_args()
        a.B, a.T, a.H, a.dk, a.dv, a.E, a.K, a.Dm, a.eps = 2, 100, 3, 128, 128, 4, 4, 256, 1e-6
        for n in ("u", "W", "conv_w", "gate_in", "gate_bias", "A_log", "q", "k", "v", "q2", "k2",
                  "g"):
            setattr(a, n, f)
        for n, v in kw.items():
            setattr(a, n, v)
        return a

    cases = [(dict(dk=96), -2), (dict(dv=32), -2), (dict(E=17), -2), (dict(Dm=100), -2),
             (dict(K=5), -1), (dict(K=0), -1), (dict(eps=0.0), -1), (dict(u=None), -1),
             (dict(beta_in=f), -1), (dict(q=ctypes.c_void_p(0x1004)), -1), (dict(T=0), -1)]
    for kw, want in cases:
        assert L.tla_layer_projection(ctypes.byref(args(**kw)), None) == want, kw
