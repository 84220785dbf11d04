"""The C ABI without a GPU: the library builds for sm_103a, loads, exports every
symbol include/gradlev.h declares, and rejects bad arguments on the host before
any CUDA call."""
import ctypes
import os
import re
import subprocess

import pytest

from paper_2609_34174_gb300 import _binding as B
from paper_2609_34174_gb300 import build as libbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "gradlev.h")


def _declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(gradlev_[a-z_0-9]+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    libbuild.build()
    return B.load_library()


def test_header_declares_the_boundary():
    names = _declared_functions()
    for required in ("gradlev_forward_scan", "gradlev_costate_scan", "gradlev_workspace_bytes",
                     "gradlev_workspace_status", "gradlev_status_string"):
        assert required in names


def test_library_exports_every_declared_symbol(lib):
    names = _declared_functions()
    out = subprocess.run(["nm", "-D", "--defined-only", libbuild.LIB], capture_output=True,
                         text=True, check=True).stdout
    exported = set(re.findall(r"\bT\s+(gradlev_\w+)", out))
    missing = [n for n in names if n not in exported]
    assert not missing, f"declared but not exported: {missing}"
    for n in names:
        assert hasattr(lib, n)


def test_abi_version_and_status_strings(lib):
    assert lib.gradlev_abi_version() == 1
    for code in (0, -1, -2, -3, -4, -5):
        assert lib.gradlev_status_string(code)
    assert lib.gradlev_status_string(-99) == b"unknown status"


def _desc(**kw):
    base = dict(L=1, B=1, T=16, H=1, d_in=64, d_out=64, dtype=1, reserved=0)
    base.update(kw)
    return B._Desc(base["L"], base["B"], base["T"], base["H"], base["d_in"], base["d_out"],
                   base["dtype"], base["reserved"])


def _t(ptr=0x1000):
    t = B._Tensor()
    t.data = ptr
    return t


@pytest.mark.parametrize("bad", [dict(L=0), dict(B=-1), dict(T=-5), dict(d_in=0), dict(dtype=7),
                                 dict(reserved=3)])
def test_bad_descriptor_rejected(lib, bad):
    d = _desc(**bad)
    x, g, y = _t(), _t(), _t()
    rc = lib.gradlev_forward_scan(ctypes.byref(d), ctypes.byref(x), ctypes.byref(g),
                                  ctypes.c_void_p(0x2000), 0.1, 0, ctypes.byref(y), None, None, 0,
                                  None)
    assert rc == -1
    assert lib.gradlev_workspace_bytes(ctypes.byref(d)) == 0


def test_null_and_nonfinite_rejected(lib):
    d = _desc()
    x, g, y = _t(), _t(), _t()
    null = _t(0)
    # null descriptor
    assert lib.gradlev_forward_scan(None, ctypes.byref(x), ctypes.byref(g), ctypes.c_void_p(0x2000),
                                    0.1, 0, ctypes.byref(y), None, None, 0, None) == -1
    # null required tensor
    assert lib.gradlev_forward_scan(ctypes.byref(d), ctypes.byref(null), ctypes.byref(g),
                                    ctypes.c_void_p(0x2000), 0.1, 0, ctypes.byref(y), None, None, 0,
                                    None) == -1
    # null W0
    assert lib.gradlev_forward_scan(ctypes.byref(d), ctypes.byref(x), ctypes.byref(g), None, 0.1, 0,
                                    ctypes.byref(y), None, None, 0, None) == -1
    # non-finite eta
    assert lib.gradlev_forward_scan(ctypes.byref(d), ctypes.byref(x), ctypes.byref(g),
                                    ctypes.c_void_p(0x2000), float("nan"), 0, ctypes.byref(y), None,
                                    None, 0, None) == -1
    # activation out of range
    assert lib.gradlev_forward_scan(ctypes.byref(d), ctypes.byref(x), ctypes.byref(g),
                                    ctypes.c_void_p(0x2000), 0.1, 9, ctypes.byref(y), None, None, 0,
                                    None) == -1
    # act_out requested without an activation
    a = _t()
    assert lib.gradlev_forward_scan(ctypes.byref(d), ctypes.byref(x), ctypes.byref(g),
                                    ctypes.c_void_p(0x2000), 0.1, 0, ctypes.byref(y), ctypes.byref(a),
                                    None, 0, None) == -1
    # costate: missing g_out, and z without an activation
    gi = _t()
    assert lib.gradlev_costate_scan(ctypes.byref(d), ctypes.byref(x), ctypes.byref(g),
                                    ctypes.c_void_p(0x2000), 0.1, ctypes.byref(null), 0, None,
                                    ctypes.byref(gi), None, 0, None) == -1
    z = _t()
    go = _t()
    assert lib.gradlev_costate_scan(ctypes.byref(d), ctypes.byref(x), ctypes.byref(g),
                                    ctypes.c_void_p(0x2000), 0.1, ctypes.byref(go), 0,
                                    ctypes.byref(z), ctypes.byref(gi), None, 0, None) == -1


def test_bad_strides_rejected(lib):
    d = _desc(B=2, H=2)
    x = _t()
    x.stride[0], x.stride[1], x.stride[2], x.stride[3] = 0, 0, 64, 64   # B stride 0 with B=2
    g, y = _t(), _t()
    assert lib.gradlev_forward_scan(ctypes.byref(d), ctypes.byref(x), ctypes.byref(g),
                                    ctypes.c_void_p(0x2000), 0.1, 0, ctypes.byref(y), None, None, 0,
                                    None) == -1
    x.stride[0], x.stride[1], x.stride[2], x.stride[3] = 4096, 2048, 64, 32  # heads overlap
    assert lib.gradlev_forward_scan(ctypes.byref(d), ctypes.byref(x), ctypes.byref(g),
                                    ctypes.c_void_p(0x2000), 0.1, 0, ctypes.byref(y), None, None, 0,
                                    None) == -1


def test_workspace_bytes_cover_the_segment_carry(lib):
    # long sequences with few units need the look-back workspace; many units need none
    long_ctx = _desc(B=2, H=16, T=32768)
    many = _desc(L=12, B=8, H=12, T=8192)
    wl = lib.gradlev_workspace_bytes(ctypes.byref(long_ctx))
    wm = lib.gradlev_workspace_bytes(ctypes.byref(many))
    assert wl > 1 << 20
    assert 256 <= wm < 1 << 20
    assert wl % 256 == 0 or wl > 0


def test_decode_arguments_rejected_before_launch(lib):
    d = _desc(T=1)
    x, g, y = _t(), _t(), _t()
    delta, W0, eta = ctypes.c_void_p(0x4000), ctypes.c_void_p(0x8000), ctypes.c_void_p(0x9000)
    # a decode call covers exactly one token per unit
    d2 = _desc(T=2)
    assert lib.gradlev_decode_read(ctypes.byref(d2), ctypes.byref(x), W0, delta, 0,
                                   ctypes.byref(y), None, None) == -1
    # missing Delta
    assert lib.gradlev_decode_read(ctypes.byref(d), ctypes.byref(x), W0, None, 0,
                                   ctypes.byref(y), None, None) == -1
    # d_in not a multiple of 4
    d3 = _desc(T=1, d_in=6)
    assert lib.gradlev_decode_write(ctypes.byref(d3), ctypes.byref(x), ctypes.byref(g), W0, delta,
                                    eta, None, 0, None, None, None, 0, None) == -2
    # activation out of range
    assert lib.gradlev_decode_write(ctypes.byref(d), ctypes.byref(x), ctypes.byref(g), W0, delta,
                                    eta, None, 9, None, None, None, 0, None) == -1


def test_decode_workspace_sizes(lib):
    # one row tile per unit: no workspace
    assert lib.gradlev_decode_workspace_bytes(ctypes.byref(_desc(L=12, B=8, H=12, T=1))) == 0
    # 1024 -> 4096 for two sequences: 32 tiles of 128 rows x 1024 fp32 partial sums per
    # sequence, plus one counter per (sequence, strip of 128 columns), each 256-aligned
    d = _desc(B=2, T=1, d_in=1024, d_out=4096)
    assert lib.gradlev_decode_workspace_bytes(ctypes.byref(d)) == 2 * 32 * 1024 * 4 + 256
    assert lib.gradlev_decode_workspace_bytes(ctypes.byref(_desc(T=3))) == 0


def test_document_gates_arguments_rejected_before_launch(lib):
    """gradlev_document_gates validates everything before it launches: these calls
    return without touching a device."""
    P = ctypes.c_void_p
    ok_ptr = P(0x10000)
    d = _desc(L=1, B=2, T=8, H=3)
    call = lambda desc, ds, eta, et, at, eo, ao: lib.gradlev_document_gates(
        desc, ds, eta, et, at, eo, ao, None)
    assert call(None, ok_ptr, 0.1, None, None, ok_ptr, ok_ptr) == -1           # no descriptor
    assert call(ctypes.byref(_desc(reserved=1)), ok_ptr, 0.1, None, None, ok_ptr, ok_ptr) == -1
    assert call(ctypes.byref(_desc(T=-1)), ok_ptr, 0.1, None, None, ok_ptr, ok_ptr) == -1
    assert call(ctypes.byref(d), None, 0.1, None, None, ok_ptr, ok_ptr) == -1  # no starts
    assert call(ctypes.byref(d), ok_ptr, 0.1, None, None, None, ok_ptr) == -1  # no eta_out
    assert call(ctypes.byref(d), ok_ptr, 0.1, None, None, ok_ptr, None) == -1  # no alpha_out
    assert call(ctypes.byref(d), ok_ptr, float("nan"), None, None, ok_ptr, ok_ptr) == -1
    assert call(ctypes.byref(d), ok_ptr, float("inf"), None, None, ok_ptr, ok_ptr) == -1
    assert call(ctypes.byref(d), ok_ptr, 0.1, P(0x10002), None, ok_ptr, ok_ptr) == -1  # misaligned
    assert call(ctypes.byref(d), ok_ptr, 0.1, None, None, ok_ptr, P(0x10001)) == -1
    # nothing to do: OK with no pointers at all
    assert call(ctypes.byref(_desc(T=0)), None, float("nan"), None, None, None, None) == 0
    assert call(ctypes.byref(_desc(H=0)), None, 0.1, None, None, None, None) == 0


def test_fused_scan_rejects_bad_arguments(lib):
    """gradlev_fused_scan checks its arguments on the host before any CUDA call."""
    d = _desc()
    x, g, go, y, gi, pr = _t(), _t(), _t(), _t(), _t(), _t()
    null = _t(0)
    W = ctypes.c_void_p(0x2000)
    cons = ctypes.c_void_p(0x3000)

    def call(desc=ctypes.byref(d), eta=0.1, g_out=ctypes.byref(go), prop=None, c=None, w0=W):
        return lib.gradlev_fused_scan(desc, ctypes.byref(x), ctypes.byref(g), w0, eta, g_out,
                                      ctypes.byref(y), ctypes.byref(gi), prop, c, None, 0, None)

    assert call(desc=None) == -1
    assert call(w0=None) == -1
    assert call(eta=float("inf")) == -1
    assert call(g_out=ctypes.byref(null)) == -1
    assert call(g_out=None) == -1
    # a proposal without the output array, and the output array without a proposal
    assert call(prop=ctypes.byref(pr)) == -1
    assert call(c=cons) == -1
    # the consistency output must be 4-byte aligned
    assert call(prop=ctypes.byref(pr), c=ctypes.c_void_p(0x3002)) == -1
