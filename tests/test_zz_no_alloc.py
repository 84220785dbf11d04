"""gradlev_forward_scan_noalloc: the forward scan for callers that cannot allocate.

Callers behind a fixed "inputs, outputs, stream" interface, or whose device
memory is budgeted once at start-up, have no workspace to pass; this entry
point keeps the kernel's scratch in a fixed array inside the library.  The tests
call it through the C ABI, on each kernel path that uses the array (the 64-wide
chunk kernel with its segment look-back, the wide-layer passes, the fp32
CUDA-core kernel), twice in a row on different inputs, and check each result
against the ordinary entry point (which uses a caller workspace) and against the
fp64 oracle, with the bounds of the other parity tests.  A timed-out wait on this
path is injected from the host and read back through
gradlev_forward_scan_noalloc_status.

This file is collected last, so a failure here comes after every other test has
run; it also passes alone in a fresh process, where its first call performs the
per-device set-up.
"""
import ctypes

import numpy as np
import pytest
import torch

import workloads as W
from parity_util import all_units, assert_parity, gpu_units, oracle_linear

gl = pytest.importorskip("paper_2609_34174_gb300")
from paper_2609_34174_gb300 import _binding as B  # noqa: E402

pytestmark = pytest.mark.gpu

SCRATCH_BYTES = 4 << 20
GRADLEV_ERR_TIMEOUT = -4
GRADLEV_ERR_WORKSPACE = -5


def _lib():
    lib = B.load_library()
    Tp = ctypes.POINTER(B._Tensor)
    lib.gradlev_forward_scan_noalloc.argtypes = [ctypes.POINTER(B._Desc), Tp, Tp, ctypes.c_void_p,
                                                 ctypes.c_float, ctypes.c_int, Tp, Tp,
                                                 ctypes.c_void_p]
    lib.gradlev_forward_scan_noalloc.restype = ctypes.c_int
    lib.gradlev_forward_scan_noalloc_status.argtypes = [ctypes.c_void_p]
    lib.gradlev_forward_scan_noalloc_status.restype = ctypes.c_int
    return lib


def _stream():
    return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)


def _call_noalloc(lib, x, g_hat, W0, eta, y):
    x5, g5, y5 = B._as5(x), B._as5(g_hat), B._as5(y)
    L, Bb, T, H, d_in = x5.shape
    dtype = 1 if x.dtype == torch.bfloat16 else 0
    desc = B._Desc(L, Bb, T, H, d_in, g5.shape[4], dtype, 0)
    tx, tg, ty = B._tensor(x5), B._tensor(g5), B._tensor(y5)
    return lib.gradlev_forward_scan_noalloc(ctypes.byref(desc), ctypes.byref(tx),
                                            ctypes.byref(tg), ctypes.c_void_p(W0.data_ptr()),
                                            float(eta), 0, ctypes.byref(ty), None, _stream())


CASES = {
    # 64-wide heads over several segments: the chunk kernel's ticket, look-back
    # flags and segment aggregates all live in the array
    "chunk-segmented": ("c4", dict(B=1, H=2, T=3000)),
    # d_in = 256: the wide-layer passes, whose segment states and score tiles are
    # TMA tensor maps over the array
    "wide-256x64": ("c2", dict(B=1, H=1, T=1000, d_in=256, d_out=64, w_std=1 / 16)),
    # fp32: the CUDA-core kernel (only the status words are cleared)
    "fp32-c1": ("c1", dict()),
}


@pytest.mark.parametrize("case", sorted(CASES))
def test_noalloc_matches_workspace_entry_point_and_oracle_twice(case):
    lib = _lib()
    key, kw = CASES[case]
    base = W.workload(key).resized(**kw)
    d = B._Desc(base.L, base.B, base.T, base.H, base.d_in, base.d_out,
                1 if base.dtype == "bf16" else 0, 0)
    assert 0 < lib.gradlev_workspace_bytes(ctypes.byref(d))
    dkey = "f32" if base.dtype == "f32" else "bf16"
    for call, seed_shift in enumerate((0, 7)):
        wl = base.resized(seed=base.seed + seed_shift)
        inputs = W.make_linear(wl)
        inp = {k: (v.cuda() if isinstance(v, torch.Tensor) else v) for k, v in inputs.items()}
        y_ref = gl.forward_scan(inp["x"], inp["g_hat"], inp["W0"], wl.eta)
        y_new = torch.full_like(y_ref, float("nan"))
        rc = _call_noalloc(lib, inp["x"], inp["g_hat"], inp["W0"].contiguous(), wl.eta, y_new)
        assert rc == 0, f"call {call}: status {rc}"
        assert lib.gradlev_forward_scan_noalloc_status(_stream()) == 0
        torch.cuda.synchronize()
        units = all_units(wl)
        a = gpu_units(y_new, units)
        assert_parity(f"{case} call {call} vs workspace entry point", a, gpu_units(y_ref, units),
                      dkey)
        yr, _ = oracle_linear(inputs, units, wl.eta, costate=False)
        assert_parity(f"{case} call {call} vs oracle", a, yr, dkey)


def test_noalloc_rejects_shapes_beyond_the_array():
    lib = _lib()
    # long context over few heads needs tens of MB of look-back scratch: too big
    wl = W.workload("c4")
    d = B._Desc(wl.L, wl.B, wl.T, wl.H, wl.d_in, wl.d_out, 1, 0)
    assert lib.gradlev_workspace_bytes(ctypes.byref(d)) > SCRATCH_BYTES
    small = torch.zeros((1, 1, 8, 1, 64), dtype=torch.bfloat16, device="cuda")
    t = B._tensor(small)
    w0 = torch.zeros((64, 64), dtype=torch.float32, device="cuda")
    rc = lib.gradlev_forward_scan_noalloc(ctypes.byref(d), ctypes.byref(t), ctypes.byref(t),
                                          ctypes.c_void_p(w0.data_ptr()), 0.1, 0,
                                          ctypes.byref(t), None, None)
    assert rc == GRADLEV_ERR_WORKSPACE


def test_noalloc_timeout_is_reported_and_next_call_is_correct(monkeypatch):
    """Host-side fault injection (no GPU fault): segment 0 of the first unit never
    publishes its look-back flag and the successor's wait is cut to 50 ms; the
    kernel records the error in the array's status word and returns, and the
    status call reports it.  The next call clears the word and is correct."""
    lib = _lib()
    wl = W.workload("c4").resized(B=1, H=2, T=3000)
    inputs = W.make_linear(wl)
    inp = {k: (v.cuda() if isinstance(v, torch.Tensor) else v) for k, v in inputs.items()}
    y = torch.empty_like(inp["g_hat"])
    monkeypatch.setenv("GRADLEV_TEST_SKIP_PUBLISH", "0")
    monkeypatch.setenv("GRADLEV_TEST_LOOKBACK_LIMIT_MS", "50")
    assert _call_noalloc(lib, inp["x"], inp["g_hat"], inp["W0"], wl.eta, y) == 0
    assert lib.gradlev_forward_scan_noalloc_status(_stream()) == GRADLEV_ERR_TIMEOUT
    monkeypatch.delenv("GRADLEV_TEST_SKIP_PUBLISH")
    monkeypatch.delenv("GRADLEV_TEST_LOOKBACK_LIMIT_MS")
    assert _call_noalloc(lib, inp["x"], inp["g_hat"], inp["W0"], wl.eta, y) == 0
    assert lib.gradlev_forward_scan_noalloc_status(_stream()) == 0
    units = all_units(wl)
    yr, _ = oracle_linear(inputs, units, wl.eta, costate=False)
    assert_parity("after the timeout", gpu_units(y, units), yr, "bf16")
