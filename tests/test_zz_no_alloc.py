"""gradlev_forward_scan_noalloc: the forward scan for callers that cannot allocate.

Callers behind a fixed "inputs, outputs, stream" interface, or whose device
memory is budgeted once at start-up, have no workspace to pass; this entry
point keeps the kernel's scratch in a fixed array inside the library.  The test
calls it through the C ABI twice in a row, on different inputs that both need
the segment look-back scratch, and checks each result against the ordinary
entry point (which uses a caller workspace) within the bf16 tolerance of the
parity tests.  This file is collected last, so a failure here comes after every
other test has run; it also passes alone in a fresh process, where its first
call performs the per-device set-up.
"""
import ctypes

import numpy as np
import pytest
import torch

import workloads as W
from parity_util import TOL, rel_l2

gl = pytest.importorskip("paper_2609_34174_gb300")
from paper_2609_34174_gb300 import _binding as B  # noqa: E402

pytestmark = pytest.mark.gpu


def _noalloc_fn():
    lib = B.load_library()
    fn = lib.gradlev_forward_scan_noalloc
    Tp = ctypes.POINTER(B._Tensor)
    fn.argtypes = [ctypes.POINTER(B._Desc), Tp, Tp, ctypes.c_void_p, ctypes.c_float, ctypes.c_int,
                   Tp, Tp, ctypes.c_void_p]
    fn.restype = ctypes.c_int
    return lib, fn


def _call_noalloc(fn, x, g_hat, W0, eta, y):
    x5, g5, y5 = B._as5(x), B._as5(g_hat), B._as5(y)
    L, Bb, T, H, d_in = x5.shape
    desc = B._Desc(L, Bb, T, H, d_in, g5.shape[4], 1, 0)
    tx, tg, ty = B._tensor(x5), B._tensor(g5), B._tensor(y5)
    stream = torch.cuda.current_stream().cuda_stream
    return fn(ctypes.byref(desc), ctypes.byref(tx), ctypes.byref(tg),
              ctypes.c_void_p(W0.data_ptr()), float(eta), 0, ctypes.byref(ty), None,
              ctypes.c_void_p(stream))


def test_noalloc_matches_workspace_entry_point_twice():
    lib, fn = _noalloc_fn()
    base = W.workload("c4").resized(B=1, H=2, T=3000)
    # the shape needs the look-back scratch, and it fits the fixed array
    d = B._Desc(base.L, base.B, base.T, base.H, base.d_in, base.d_out, 1, 0)
    need = lib.gradlev_workspace_bytes(ctypes.byref(d))
    assert 4096 < need <= (4 << 20)
    for call, seed_shift in enumerate((0, 7)):
        wl = base.resized(seed=base.seed + seed_shift)
        inp = {k: (v.cuda() if isinstance(v, torch.Tensor) else v)
               for k, v in W.make_linear(wl).items()}
        y_ref = gl.forward_scan(inp["x"], inp["g_hat"], inp["W0"], wl.eta)
        y_new = torch.full_like(y_ref, float("nan"))
        rc = _call_noalloc(fn, inp["x"], inp["g_hat"], inp["W0"].contiguous(), wl.eta, y_new)
        assert rc == 0, f"call {call}: status {rc}"
        torch.cuda.synchronize()
        a = y_new.double().cpu().numpy()
        b = y_ref.double().cpu().numpy()
        assert np.isfinite(a).all(), f"call {call}: non-finite output"
        err = rel_l2(a, b)
        assert err <= TOL["bf16"], f"call {call}: rel-L2 {err:.3e}"


def test_noalloc_rejects_shapes_beyond_the_array():
    lib, fn = _noalloc_fn()
    # long context over few heads needs tens of MB of look-back scratch: too big
    wl = W.workload("c4")
    d = B._Desc(wl.L, wl.B, wl.T, wl.H, wl.d_in, wl.d_out, 1, 0)
    assert lib.gradlev_workspace_bytes(ctypes.byref(d)) > (4 << 20)
    small = torch.zeros((1, 1, 8, 1, 64), dtype=torch.bfloat16, device="cuda")
    desc = B._Desc(wl.L, wl.B, wl.T, wl.H, wl.d_in, wl.d_out, 1, 0)
    t = B._tensor(small)
    w0 = torch.zeros((64, 64), dtype=torch.float32, device="cuda")
    rc = fn(ctypes.byref(desc), ctypes.byref(t), ctypes.byref(t), ctypes.c_void_p(w0.data_ptr()),
            0.1, 0, ctypes.byref(t), None, None)
    assert rc == -5
