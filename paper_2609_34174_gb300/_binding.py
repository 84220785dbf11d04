"""ctypes binding of include/gradlev.h.

Argument marshalling only: tensors are described by pointer and strides and
handed to the C ABI with the current torch CUDA stream; outputs and the
workspace are ordinary torch allocations.  All arithmetic happens in the CUDA
kernels of libgradlev.so.
"""
from __future__ import annotations

import ctypes
import os
import threading
from typing import Optional

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB_PATH = os.path.join(_HERE, "_build", "libgradlev.so")

ACT_NONE, ACT_GELU_TANH, ACT_GELU_ERF, ACT_TANH = 0, 1, 2, 3
_ACT_NAMES = {None: ACT_NONE, "none": ACT_NONE, "gelu_tanh": ACT_GELU_TANH, "gelu": ACT_GELU_TANH,
              "gelu_erf": ACT_GELU_ERF, "tanh": ACT_TANH}

GRADLEV_F32, GRADLEV_BF16 = 0, 1

_STATUS = {0: "ok", -1: "invalid argument", -2: "unsupported", -3: "CUDA error", -4: "timeout",
           -5: "workspace"}


class GradLevError(RuntimeError):
    """A libgradlev call returned a non-zero status."""

    def __init__(self, code: int, what: str):
        self.code = code
        super().__init__(f"{what}: status {code} ({_STATUS.get(code, 'unknown')})")


class _Desc(ctypes.Structure):
    _fields_ = [("L", ctypes.c_int32), ("B", ctypes.c_int32), ("T", ctypes.c_int32),
                ("H", ctypes.c_int32), ("d_in", ctypes.c_int32), ("d_out", ctypes.c_int32),
                ("dtype", ctypes.c_int32), ("reserved", ctypes.c_int32)]


class _Tensor(ctypes.Structure):
    _fields_ = [("data", ctypes.c_void_p), ("stride", ctypes.c_int64 * 4)]


_lib = None
_lib_lock = threading.Lock()


def library_path() -> str:
    return _LIB_PATH


def load_library():
    """Load libgradlev.so (building it first if nvcc is available)."""
    global _lib
    with _lib_lock:
        if _lib is not None:
            return _lib
        if not os.path.exists(_LIB_PATH):
            from . import build as _build
            _build.build()
        if not os.path.exists(_LIB_PATH):
            raise RuntimeError(f"libgradlev.so is missing at {_LIB_PATH}; run build() first")
        lib = ctypes.CDLL(_LIB_PATH)
        P = ctypes.c_void_p
        D = ctypes.POINTER(_Desc)
        Tp = ctypes.POINTER(_Tensor)
        lib.gradlev_forward_scan.argtypes = [D, Tp, Tp, P, ctypes.c_float, ctypes.c_int, Tp, Tp, P,
                                             ctypes.c_size_t, P]
        lib.gradlev_forward_scan.restype = ctypes.c_int
        lib.gradlev_costate_scan.argtypes = [D, Tp, Tp, P, ctypes.c_float, Tp, ctypes.c_int, Tp, Tp,
                                             P, ctypes.c_size_t, P]
        lib.gradlev_costate_scan.restype = ctypes.c_int
        lib.gradlev_fused_scan.argtypes = [D, Tp, Tp, P, ctypes.c_float, Tp, Tp, Tp, Tp, P, P,
                                           ctypes.c_size_t, P]
        lib.gradlev_fused_scan.restype = ctypes.c_int
        lib.gradlev_forward_scan_gated.argtypes = [D, Tp, Tp, P, P, P, ctypes.c_int, Tp, Tp, P,
                                                   ctypes.c_size_t, P]
        lib.gradlev_forward_scan_gated.restype = ctypes.c_int
        lib.gradlev_costate_scan_gated.argtypes = [D, Tp, Tp, P, P, P, Tp, ctypes.c_int, Tp, Tp, P,
                                                   ctypes.c_size_t, P]
        lib.gradlev_costate_scan_gated.restype = ctypes.c_int
        lib.gradlev_workspace_bytes_gated.argtypes = [D]
        lib.gradlev_workspace_bytes_gated.restype = ctypes.c_size_t
        lib.gradlev_document_gates.argtypes = [D, P, ctypes.c_float, P, P, P, P, P]
        lib.gradlev_document_gates.restype = ctypes.c_int
        lib.gradlev_decode_read.argtypes = [D, Tp, P, P, ctypes.c_int, Tp, Tp, P]
        lib.gradlev_decode_read.restype = ctypes.c_int
        lib.gradlev_decode_write.argtypes = [D, Tp, Tp, P, P, P, P, ctypes.c_int, Tp, Tp, P,
                                             ctypes.c_size_t, P]
        lib.gradlev_decode_write.restype = ctypes.c_int
        lib.gradlev_decode_workspace_bytes.argtypes = [D]
        lib.gradlev_decode_workspace_bytes.restype = ctypes.c_size_t
        lib.gradlev_suffix_scan.argtypes = [D, Tp, Tp, Tp, Tp, P, ctypes.c_size_t, P]
        lib.gradlev_suffix_scan.restype = ctypes.c_int
        lib.gradlev_suffix_workspace_bytes.argtypes = [D]
        lib.gradlev_suffix_workspace_bytes.restype = ctypes.c_size_t
        lib.gradlev_eta_grad.argtypes = [D, ctypes.c_int, Tp, Tp, Tp, Tp, P, P, ctypes.c_size_t, P]
        lib.gradlev_eta_grad.restype = ctypes.c_int
        lib.gradlev_eta_grad_workspace_bytes.argtypes = [D, ctypes.c_int]
        lib.gradlev_eta_grad_workspace_bytes.restype = ctypes.c_size_t
        lib.gradlev_gate_grads.argtypes = [D, ctypes.c_int, Tp, Tp, P, P, Tp, Tp, P, P, P,
                                           ctypes.c_size_t, P]
        lib.gradlev_gate_grads.restype = ctypes.c_int
        lib.gradlev_gate_grads_workspace_bytes.argtypes = [D, ctypes.c_int]
        lib.gradlev_gate_grads_workspace_bytes.restype = ctypes.c_size_t
        lib.gradlev_workspace_bytes.argtypes = [D]
        lib.gradlev_workspace_bytes.restype = ctypes.c_size_t
        lib.gradlev_workspace_status.argtypes = [P, P]
        lib.gradlev_workspace_status.restype = ctypes.c_int
        lib.gradlev_device_supported.argtypes = []
        lib.gradlev_device_supported.restype = ctypes.c_int
        lib.gradlev_status_string.argtypes = [ctypes.c_int]
        lib.gradlev_status_string.restype = ctypes.c_char_p
        lib.gradlev_abi_version.argtypes = []
        lib.gradlev_abi_version.restype = ctypes.c_int
        _lib = lib
        return lib


def device_supported() -> bool:
    return bool(load_library().gradlev_device_supported())


def _act_code(act) -> int:
    if isinstance(act, int):
        return act
    if act not in _ACT_NAMES:
        raise ValueError(f"unknown activation {act!r}")
    return _ACT_NAMES[act]


def _as5(t: torch.Tensor) -> torch.Tensor:
    """View a token tensor as [L, B, T, H, w] without copying."""
    if t.dim() == 5:
        return t
    if t.dim() == 4:   # [B, T, H, w]
        return t.unsqueeze(0)
    if t.dim() == 3:   # [B, T, w]
        return t.unsqueeze(0).unsqueeze(3)
    if t.dim() == 2:   # [T, w]
        return t.unsqueeze(0).unsqueeze(0).unsqueeze(3)
    raise ValueError(f"token tensors are 2- to 5-D, got {t.dim()}-D")


def _tensor(t5: Optional[torch.Tensor]) -> Optional[_Tensor]:
    if t5 is None:
        return None
    if t5.stride(4) != 1:
        raise ValueError("the feature dimension of a token tensor must be contiguous")
    st = _Tensor()
    st.data = t5.data_ptr()
    for i in range(4):
        s = t5.stride(i)
        if t5.shape[i] == 1:
            s = max(s, 1)
        st.stride[i] = s
    return st


_ws_cache = {}
_ws_lock = threading.Lock()


def _workspace(nbytes: int, device: torch.device) -> torch.Tensor:
    with _ws_lock:
        key = (device.index, torch.cuda.current_stream(device).cuda_stream)
        buf = _ws_cache.get(key)
        if buf is None or buf.numel() < nbytes:
            buf = torch.empty(max(nbytes, 256), dtype=torch.uint8, device=device)
            _ws_cache[key] = buf
        return buf


def _w0(W0: torch.Tensor, L: int, H: int, rows: int, cols: int) -> torch.Tensor:
    if W0.dtype != torch.float32:
        raise TypeError("W0 must be float32")
    if W0.dim() == 2:
        W0 = W0.reshape(1, 1, rows, cols)
    elif W0.dim() == 3:
        W0 = W0.unsqueeze(0)
    if tuple(W0.shape) != (L, H, rows, cols):
        raise ValueError(f"W0 must be [L,H,d_out,d_in] = {(L, H, rows, cols)}, got {tuple(W0.shape)}")
    return W0.contiguous()


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return GRADLEV_BF16
    if t.dtype == torch.float32:
        return GRADLEV_F32
    raise TypeError(f"token tensors must be bfloat16 or float32, got {t.dtype}")


def _check_same(ref: torch.Tensor, *others):
    for o in others:
        if o is None:
            continue
        if o.device != ref.device:
            raise ValueError("all tensors must be on the same device")
        if o.dtype != ref.dtype:
            raise TypeError("all token tensors must share one dtype")


def _desc(x5: torch.Tensor, d_out: int, dtype: int) -> _Desc:
    L, B, T, H, d_in = x5.shape
    return _Desc(L, B, T, H, d_in, d_out, dtype, 0)


def workspace_bytes(L, B, T, H, d_in, d_out, dtype=GRADLEV_BF16) -> int:
    d = _Desc(L, B, T, H, d_in, d_out, dtype, 0)
    return int(load_library().gradlev_workspace_bytes(ctypes.byref(d)))


def workspace_status(workspace: torch.Tensor) -> int:
    """Device-side status a previous call left in `workspace` (syncs the stream)."""
    lib = load_library()
    s = torch.cuda.current_stream(workspace.device).cuda_stream
    return int(lib.gradlev_workspace_status(ctypes.c_void_p(workspace.data_ptr()),
                                            ctypes.c_void_p(s)))


def _gates(eta, alpha, x5):
    """Per-token gate arrays for the gated entry points, or None for a plain scalar
    eta: fp32 [L,B,T,H] contiguous on the tensors' device."""
    if not isinstance(eta, torch.Tensor) and alpha is None:
        return None
    shape = tuple(x5.shape[:4])

    def norm(v):
        if isinstance(v, torch.Tensor):
            t = v.to(device=x5.device, dtype=torch.float32)
            return t.reshape(shape).contiguous()
        return torch.full(shape, float(v), dtype=torch.float32, device=x5.device)

    return norm(eta), (norm(alpha) if alpha is not None else None)


def _document_gates(doc_start, x5, eta, alpha):
    """Fold document starts into fp32 [L,B,T,H] (eta_t, alpha_t) on x5's device."""
    lib = load_library()
    L, B, T, H = (int(v) for v in x5.shape[:4])
    ds = doc_start if isinstance(doc_start, torch.Tensor) else torch.as_tensor(doc_start)
    ds = ds.to(device=x5.device)
    if ds.dim() == 1 and B == 1:
        ds = ds.unsqueeze(0)
    if tuple(ds.shape) != (B, T):
        raise ValueError(f"doc_start must be [B, T] = {(B, T)}, got {tuple(ds.shape)}")
    if ds.dtype != torch.uint8:
        ds = (ds != 0).to(torch.uint8)
    ds = ds.contiguous()
    shape = (L, B, T, H)

    def per_token(v):
        if not isinstance(v, torch.Tensor):
            return None
        return v.to(device=x5.device, dtype=torch.float32).reshape(shape).contiguous()

    et, at = per_token(eta), per_token(alpha)
    if alpha is not None and at is None:
        at = torch.full(shape, float(alpha), dtype=torch.float32, device=x5.device)
    eo = torch.empty(shape, dtype=torch.float32, device=x5.device)
    ao = torch.empty(shape, dtype=torch.float32, device=x5.device)
    desc = _Desc(L, B, T, H, 0, 0, 0, 0)
    stream = torch.cuda.current_stream(x5.device).cuda_stream
    ptr = lambda t: ctypes.c_void_p(t.data_ptr()) if t is not None else None
    with torch.cuda.device(x5.device):
        rc = lib.gradlev_document_gates(ctypes.byref(desc), ptr(ds),
                                        0.0 if et is not None else float(eta), ptr(et), ptr(at),
                                        ptr(eo), ptr(ao), ctypes.c_void_p(stream))
    _call(rc, "gradlev_document_gates")
    return eo, ao


def document_gates(doc_start, x, eta, alpha=None):
    """Per-token gates for sequences packed from several documents (Appendix C:
    a read sees only the writes of its own document; Appendix E).

    doc_start: bool / integer [B, T] (or [T] when B = 1), nonzero where a document
    begins, the same for every layer and head.  eta: scalar or per-token tensor;
    alpha: None, scalar or per-token tensor.  Returns fp32 (eta_t, alpha_t) with the
    token shape of x, with eta = alpha = 0 on the last token of every document that
    another follows.  forward_scan / costate_scan take doc_start= and do this
    themselves.
    """
    x5 = _as5(x)
    if not x5.is_cuda:
        raise ValueError("tensors must be on a CUDA device")
    eo, ao = _document_gates(doc_start, x5, eta, alpha)
    return eo.reshape(x.shape[:-1]), ao.reshape(x.shape[:-1])


def _call(rc: int, what: str):
    if rc != 0:
        raise GradLevError(rc, what)


def forward_scan(x, g_hat, W0, eta, act=None, y=None, act_out=None, want_act_out=False,
                 workspace=None, alpha=None, doc_start=None):
    """y_t = (W0 - eta sum_{s<t} ghat_s x_s^T) x_t for every token (Sec. 3 step 2, Eq. 3).

    x [L,B,T,H,d_in] (or [B,T,H,d_in], [B,T,d_in], [T,d_in]), g_hat with d_out features,
    W0 fp32 [L,H,d_out,d_in].  With want_act_out (or act_out given) also returns
    sigma(y) for the activation `act`.  Returns y, or (y, act_out).

    Gates (Eq. 2): `eta` may be a tensor of per-token step sizes with the token
    shape of x, and `alpha` an optional per-token retention (decay centred at W0;
    alpha = 0 resets to W0).  `doc_start` ([B, T], nonzero where a document begins)
    resets the fast weights at document starts (see document_gates).
    """
    lib = load_library()
    x5, g5 = _as5(x), _as5(g_hat)
    _check_same(x5, g5)
    if not x5.is_cuda:
        raise ValueError("tensors must be on a CUDA device")
    L, B, T, H, d_in = x5.shape
    d_out = g5.shape[4]
    if tuple(g5.shape[:4]) != (L, B, T, H):
        raise ValueError("x and g_hat token shapes differ")
    W = _w0(W0, L, H, d_out, d_in)
    if W.device != x5.device:
        raise ValueError("W0 must be on the tensors' device")
    code = _act_code(act)
    if y is None:
        y = torch.empty(tuple(x.shape[:-1]) + (d_out,), dtype=x5.dtype, device=x5.device)
    y5 = _as5(y)
    _check_same(x5, y5)
    if tuple(y5.shape) != (L, B, T, H, d_out):
        raise ValueError("y has the wrong shape")
    if want_act_out and act_out is None:
        act_out = torch.empty_like(y)
    a5 = _as5(act_out) if act_out is not None else None
    desc = _desc(x5, d_out, _dtype_code(x5))
    if doc_start is not None:
        eta, alpha = _document_gates(doc_start, x5, eta, alpha)
    gates = _gates(eta, alpha, x5)
    if gates is not None:
        nbytes = int(lib.gradlev_workspace_bytes_gated(ctypes.byref(desc)))
    else:
        nbytes = int(lib.gradlev_workspace_bytes(ctypes.byref(desc)))
    ws = workspace if workspace is not None else _workspace(nbytes, x5.device)
    tx, tg, ty = _tensor(x5), _tensor(g5), _tensor(y5)
    ta = _tensor(a5) if a5 is not None else None
    stream = torch.cuda.current_stream(x5.device).cuda_stream
    if gates is not None:
        et, al = gates
        with torch.cuda.device(x5.device):
            rc = lib.gradlev_forward_scan_gated(
                ctypes.byref(desc), ctypes.byref(tx), ctypes.byref(tg), ctypes.c_void_p(W.data_ptr()),
                ctypes.c_void_p(et.data_ptr()), ctypes.c_void_p(al.data_ptr()) if al is not None else None,
                code, ctypes.byref(ty), ctypes.byref(ta) if ta is not None else None,
                ctypes.c_void_p(ws.data_ptr()), ws.numel(), ctypes.c_void_p(stream))
        _call(rc, "gradlev_forward_scan_gated")
        if act_out is not None:
            return y, act_out
        return y
    with torch.cuda.device(x5.device):
        rc = lib.gradlev_forward_scan(ctypes.byref(desc), ctypes.byref(tx), ctypes.byref(tg),
                                      ctypes.c_void_p(W.data_ptr()), float(eta), code,
                                      ctypes.byref(ty), ctypes.byref(ta) if ta is not None else None,
                                      ctypes.c_void_p(ws.data_ptr()), ws.numel(),
                                      ctypes.c_void_p(stream))
    _call(rc, "gradlev_forward_scan")
    if act_out is not None:
        return y, act_out
    return y


def costate_scan(x, g_hat, W0, eta, g_out, act=None, z=None, g_in=None, workspace=None,
                 alpha=None, doc_start=None):
    """g_in_t = (W0 - eta sum_{s<t} ghat_s x_s^T)^T g_out_t (Sec. 3 step 3, Eq. 4).

    With z (the preactivation that fed this map's input through sigma = act) the
    result is sigma'(z_t) * (What_t^T g_out_t).  Returns g_in [.., d_in].
    Gates and doc_start as for forward_scan.
    """
    lib = load_library()
    x5, g5, go5 = _as5(x), _as5(g_hat), _as5(g_out)
    _check_same(x5, g5, go5)
    if not x5.is_cuda:
        raise ValueError("tensors must be on a CUDA device")
    L, B, T, H, d_in = x5.shape
    d_out = g5.shape[4]
    if tuple(g5.shape) != tuple(go5.shape) or tuple(g5.shape[:4]) != (L, B, T, H):
        raise ValueError("g_hat / g_out shapes differ from x")
    W = _w0(W0, L, H, d_out, d_in)
    code = _act_code(act)
    z5 = _as5(z) if z is not None else None
    if z5 is not None:
        _check_same(x5, z5)
        if tuple(z5.shape) != tuple(x5.shape):
            raise ValueError("z must have the shape of x")
    if g_in is None:
        g_in = torch.empty(x5.shape, dtype=x5.dtype, device=x5.device).view(x.shape)
    gi5 = _as5(g_in)
    _check_same(x5, gi5)
    desc = _desc(x5, d_out, _dtype_code(x5))
    if doc_start is not None:
        eta, alpha = _document_gates(doc_start, x5, eta, alpha)
    gates = _gates(eta, alpha, x5)
    if gates is not None:
        nbytes = int(lib.gradlev_workspace_bytes_gated(ctypes.byref(desc)))
    else:
        nbytes = int(lib.gradlev_workspace_bytes(ctypes.byref(desc)))
    ws = workspace if workspace is not None else _workspace(nbytes, x5.device)
    tx, tg, tgo, tgi = _tensor(x5), _tensor(g5), _tensor(go5), _tensor(gi5)
    tz = _tensor(z5) if z5 is not None else None
    stream = torch.cuda.current_stream(x5.device).cuda_stream
    if gates is not None:
        et, al = gates
        with torch.cuda.device(x5.device):
            rc = lib.gradlev_costate_scan_gated(
                ctypes.byref(desc), ctypes.byref(tx), ctypes.byref(tg), ctypes.c_void_p(W.data_ptr()),
                ctypes.c_void_p(et.data_ptr()), ctypes.c_void_p(al.data_ptr()) if al is not None else None,
                ctypes.byref(tgo), code, ctypes.byref(tz) if tz is not None else None,
                ctypes.byref(tgi), ctypes.c_void_p(ws.data_ptr()), ws.numel(), ctypes.c_void_p(stream))
        _call(rc, "gradlev_costate_scan_gated")
        return g_in
    with torch.cuda.device(x5.device):
        rc = lib.gradlev_costate_scan(ctypes.byref(desc), ctypes.byref(tx), ctypes.byref(tg),
                                      ctypes.c_void_p(W.data_ptr()), float(eta), ctypes.byref(tgo),
                                      code, ctypes.byref(tz) if tz is not None else None,
                                      ctypes.byref(tgi), ctypes.c_void_p(ws.data_ptr()), ws.numel(),
                                      ctypes.c_void_p(stream))
    _call(rc, "gradlev_costate_scan")
    return g_in


def fused_scan(x, g_hat, W0, eta, g_out, y=None, g_in=None, cons_proposal=None, cons=None,
               workspace=None):
    """Both reads of one map in one call (Sec. 3 steps 2 and 3, Eqs. 3-4):
    y_t = What_t x_t and g_in_t = What_t^T g_out_t over the same writes.

    With cons_proposal (shape of x) also the per-token consistency term
    cons_t = ||cons_proposal_t - g_in_t||^2 / d_in of Eq. 5, fp32 [L,B,T,H] (or the
    token shape of x).  Returns (y, g_in) or (y, g_in, cons).
    """
    lib = load_library()
    x5, g5, go5 = _as5(x), _as5(g_hat), _as5(g_out)
    _check_same(x5, g5, go5)
    if not x5.is_cuda:
        raise ValueError("tensors must be on a CUDA device")
    L, B, T, H, d_in = x5.shape
    d_out = g5.shape[4]
    if tuple(g5.shape) != tuple(go5.shape) or tuple(g5.shape[:4]) != (L, B, T, H):
        raise ValueError("g_hat / g_out shapes differ from x")
    W = _w0(W0, L, H, d_out, d_in)
    if W.device != x5.device:
        raise ValueError("W0 must be on the tensors' device")
    if y is None:
        y = torch.empty(tuple(x.shape[:-1]) + (d_out,), dtype=x5.dtype, device=x5.device)
    if g_in is None:
        g_in = torch.empty(x5.shape, dtype=x5.dtype, device=x5.device).view(x.shape)
    y5, gi5 = _as5(y), _as5(g_in)
    _check_same(x5, y5, gi5)
    if tuple(y5.shape) != (L, B, T, H, d_out) or tuple(gi5.shape) != tuple(x5.shape):
        raise ValueError("y / g_in have the wrong shape")
    p5 = None
    if cons_proposal is not None:
        p5 = _as5(cons_proposal)
        _check_same(x5, p5)
        if tuple(p5.shape) != tuple(x5.shape):
            raise ValueError("cons_proposal must have the shape of x")
        if cons is None:
            cons = torch.empty(tuple(x.shape[:-1]), dtype=torch.float32, device=x5.device)
        if cons.dtype != torch.float32 or not cons.is_contiguous() or cons.numel() != L * B * T * H:
            raise ValueError("cons must be a contiguous float32 tensor of L*B*T*H entries")
    desc = _desc(x5, d_out, _dtype_code(x5))
    nbytes = int(lib.gradlev_workspace_bytes(ctypes.byref(desc)))
    ws = workspace if workspace is not None else _workspace(nbytes, x5.device)
    tx, tg, tgo, ty, tgi = _tensor(x5), _tensor(g5), _tensor(go5), _tensor(y5), _tensor(gi5)
    tp = _tensor(p5) if p5 is not None else None
    stream = torch.cuda.current_stream(x5.device).cuda_stream
    with torch.cuda.device(x5.device):
        rc = lib.gradlev_fused_scan(ctypes.byref(desc), ctypes.byref(tx), ctypes.byref(tg),
                                    ctypes.c_void_p(W.data_ptr()), float(eta), ctypes.byref(tgo),
                                    ctypes.byref(ty), ctypes.byref(tgi),
                                    ctypes.byref(tp) if tp is not None else None,
                                    ctypes.c_void_p(cons.data_ptr()) if tp is not None else None,
                                    ctypes.c_void_p(ws.data_ptr()), ws.numel(),
                                    ctypes.c_void_p(stream))
    _call(rc, "gradlev_fused_scan")
    return (y, g_in, cons) if p5 is not None else (y, g_in)


def mlp_forward(x, g_hat_z, g_hat_y, W1, W2, eta1, eta2, act="gelu_tanh"):
    """Forward through the two-layer fast-weight MLP (Appendix A, eqs. scan1-proposed).

    Layer 1 writes z = (W1 + Delta1_t) x and, fused in its epilogue, h = sigma(z);
    layer 2 reads h.  Returns (z, h, y).
    """
    z, h = forward_scan(x, g_hat_z, W1, eta1, act=act, want_act_out=True)
    y = forward_scan(h, g_hat_y, W2, eta2)
    return z, h, y


def mlp_costate(x, h, z, g_hat_z, g_hat_y, W1, W2, eta1, eta2, g_out, act="gelu_tanh"):
    """Costates back through both layers (Appendix A eq. reconstructed-reverse, then
    the layer-1 transpose read).  Returns (g_z, g_x): g_z = sigma'(z) * (W2_t^T g_out)
    with sigma' fused in the layer-2 costate epilogue, g_x = W1_t^T g_z."""
    g_z = costate_scan(h, g_hat_y, W2, eta2, g_out, act=act, z=z)
    g_x = costate_scan(x, g_hat_z, W1, eta1, g_z)
    return g_z, g_x


# ------------------------------------------------------------------ deployment
def _tok1(t: torch.Tensor) -> torch.Tensor:
    """View a one-token tensor [L,B,H,w] (or [B,H,w], [B,w]) as [L,B,1,H,w]."""
    if t.dim() == 4:
        return t.unsqueeze(2)
    if t.dim() == 3:
        return t.unsqueeze(0).unsqueeze(2)
    if t.dim() == 2:
        return t.unsqueeze(0).unsqueeze(2).unsqueeze(3)
    raise ValueError(f"one-token tensors are 2- to 4-D, got {t.dim()}-D")


def _delta(delta: torch.Tensor, L, B, H, rows, cols) -> torch.Tensor:
    if delta.dtype != torch.float32 or not delta.is_contiguous():
        raise TypeError("delta must be a contiguous float32 tensor")
    if delta.numel() != L * B * H * rows * cols:
        raise ValueError(f"delta must be [L,B,H,d_out,d_in] = {(L, B, H, rows, cols)}")
    return delta


def _per_unit(v, L, B, H, device):
    if isinstance(v, torch.Tensor):
        return v.to(device=device, dtype=torch.float32).expand(L, B, H).contiguous()
    return torch.full((L, B, H), float(v), dtype=torch.float32, device=device)


def decode_read(x, W0, delta, act=None, want_act_out=False, y=None, act_out=None):
    """Deployment read for one token per unit: y = (W0 + delta) x (Sec. 3).

    x [L,B,H,d_in] (or [B,H,d_in], [B,d_in]); W0 fp32 [L,H,d_out,d_in]; delta fp32
    [L,B,H,d_out,d_in], the fast weights minus W0.  Returns y [.., d_out], or
    (y, sigma(y)) with want_act_out.
    """
    lib = load_library()
    x5 = _tok1(x)
    if not x5.is_cuda:
        raise ValueError("tensors must be on a CUDA device")
    L, B, _, H, d_in = x5.shape
    d_out = W0.shape[-2]
    W = _w0(W0, L, H, d_out, d_in)
    D = _delta(delta, L, B, H, d_out, d_in)
    code = _act_code(act)
    if y is None:
        y = torch.empty(tuple(x.shape[:-1]) + (d_out,), dtype=x5.dtype, device=x5.device)
    y5 = _tok1(y)
    _check_same(x5, y5)
    if want_act_out and act_out is None:
        act_out = torch.empty_like(y)
    a5 = _tok1(act_out) if act_out is not None else None
    desc = _desc(x5, d_out, _dtype_code(x5))
    tx, ty = _tensor(x5), _tensor(y5)
    ta = _tensor(a5) if a5 is not None else None
    stream = torch.cuda.current_stream(x5.device).cuda_stream
    with torch.cuda.device(x5.device):
        rc = lib.gradlev_decode_read(ctypes.byref(desc), ctypes.byref(tx), ctypes.c_void_p(W.data_ptr()),
                                     ctypes.c_void_p(D.data_ptr()), code, ctypes.byref(ty),
                                     ctypes.byref(ta) if ta is not None else None,
                                     ctypes.c_void_p(stream))
    _call(rc, "gradlev_decode_read")
    if act_out is not None:
        return y, act_out
    return y


def decode_workspace_bytes(L, B, H, d_in, d_out, dtype=GRADLEV_BF16) -> int:
    d = _Desc(L, B, 1, H, d_in, d_out, dtype, 0)
    return int(load_library().gradlev_decode_workspace_bytes(ctypes.byref(d)))


def decode_write(x, g, W0, delta, eta, alpha=None, want_g_in=True, act=None, z=None, g_in=None,
                 workspace=None):
    """Deployment write for one token per unit, after its target was scored (Sec. 3).

    With want_g_in, first g_in = (W0 + delta)^T g with the weights before the write
    (times sigma'(z) when z is given); then delta <- alpha delta - eta g x^T in place
    (Eq. 2).  x [L,B,H,d_in], g [L,B,H,d_out] (the true costate dl/dy), eta and alpha
    scalars or per-unit [L,B,H].  Returns g_in, or None.
    """
    lib = load_library()
    x5, g5 = _tok1(x), _tok1(g)
    _check_same(x5, g5)
    if not x5.is_cuda:
        raise ValueError("tensors must be on a CUDA device")
    L, B, _, H, d_in = x5.shape
    d_out = g5.shape[4]
    D = _delta(delta, L, B, H, d_out, d_in)
    W = _w0(W0, L, H, d_out, d_in) if want_g_in else None
    et = _per_unit(eta, L, B, H, x5.device)
    al = _per_unit(alpha, L, B, H, x5.device) if alpha is not None else None
    code = _act_code(act)
    z5 = _tok1(z) if z is not None else None
    if want_g_in and g_in is None:
        g_in = torch.empty(tuple(x.shape), dtype=x5.dtype, device=x5.device)
    gi5 = _tok1(g_in) if want_g_in else None
    desc = _desc(x5, d_out, _dtype_code(x5))
    ws = None
    if want_g_in:
        nbytes = int(lib.gradlev_decode_workspace_bytes(ctypes.byref(desc)))
        if nbytes:
            ws = workspace if workspace is not None else _workspace(nbytes, x5.device)
    tx, tg = _tensor(x5), _tensor(g5)
    tz = _tensor(z5) if z5 is not None else None
    tgi = _tensor(gi5) if gi5 is not None else None
    stream = torch.cuda.current_stream(x5.device).cuda_stream
    with torch.cuda.device(x5.device):
        rc = lib.gradlev_decode_write(
            ctypes.byref(desc), ctypes.byref(tx), ctypes.byref(tg),
            ctypes.c_void_p(W.data_ptr()) if W is not None else None, ctypes.c_void_p(D.data_ptr()),
            ctypes.c_void_p(et.data_ptr()), ctypes.c_void_p(al.data_ptr()) if al is not None else None,
            code, ctypes.byref(tz) if tz is not None else None,
            ctypes.byref(tgi) if tgi is not None else None,
            ctypes.c_void_p(ws.data_ptr()) if ws is not None else None,
            ws.numel() if ws is not None else 0, ctypes.c_void_p(stream))
    _call(rc, "gradlev_decode_write")
    return g_in


# ------------------------------------------------------------- outer gradients
def suffix_scan(q, k, v, r=None, workspace=None):
    """Anti-causal read r_s = sum_{t>s} (k_t . q_s) v_t (outer gradients through the
    reads).  q, k [L,B,T,H,dq] (or fewer leading dims), v [.., dv].  Returns r [.., dv]."""
    lib = load_library()
    q5, k5, v5 = _as5(q), _as5(k), _as5(v)
    _check_same(q5, k5, v5)
    if not q5.is_cuda:
        raise ValueError("tensors must be on a CUDA device")
    if tuple(k5.shape) != tuple(q5.shape) or tuple(v5.shape[:4]) != tuple(q5.shape[:4]):
        raise ValueError("q, k and v token shapes differ")
    dv = v5.shape[4]
    if r is None:
        r = torch.empty(tuple(v.shape), dtype=v5.dtype, device=v5.device)
    r5 = _as5(r)
    _check_same(q5, r5)
    desc = _desc(q5, dv, _dtype_code(q5))
    nbytes = int(lib.gradlev_suffix_workspace_bytes(ctypes.byref(desc)))
    ws = workspace if workspace is not None else (_workspace(nbytes, q5.device) if nbytes else None)
    tq, tk, tv, tr = _tensor(q5), _tensor(k5), _tensor(v5), _tensor(r5)
    stream = torch.cuda.current_stream(q5.device).cuda_stream
    with torch.cuda.device(q5.device):
        rc = lib.gradlev_suffix_scan(ctypes.byref(desc), ctypes.byref(tq), ctypes.byref(tk),
                                     ctypes.byref(tv), ctypes.byref(tr),
                                     ctypes.c_void_p(ws.data_ptr()) if ws is not None else None,
                                     ws.numel() if ws is not None else 0, ctypes.c_void_p(stream))
    _call(rc, "gradlev_suffix_scan")
    return r


def eta_grad(x, g_hat, upstream, read="forward", g_out=None, deta=None, workspace=None):
    """dL/deta_t of one map's read for per-token step sizes (writes detached).

    read="forward": upstream = dL/dy ([.., d_out]); read="costate": upstream = dL/dg_in
    ([.., d_in]) and g_out is required.  Returns fp32 [L,B,T,H] (the token shape of x).
    """
    lib = load_library()
    x5, g5, u5 = _as5(x), _as5(g_hat), _as5(upstream)
    go5 = _as5(g_out) if g_out is not None else None
    _check_same(x5, g5, u5, go5)
    if not x5.is_cuda:
        raise ValueError("tensors must be on a CUDA device")
    rd = {"forward": 0, "costate": 1}[read]
    if rd == 1 and go5 is None:
        raise ValueError("the costate read needs g_out")
    L, B, T, H, d_in = x5.shape
    d_out = g5.shape[4]
    desc = _desc(x5, d_out, _dtype_code(x5))
    if deta is None:
        deta = torch.empty((L, B, T, H), dtype=torch.float32, device=x5.device)
    if deta.dtype != torch.float32 or not deta.is_contiguous() or deta.numel() != L * B * T * H:
        raise ValueError("deta must be a contiguous float32 [L,B,T,H] tensor")
    nbytes = int(lib.gradlev_eta_grad_workspace_bytes(ctypes.byref(desc), rd))
    ws = workspace if workspace is not None else _workspace(nbytes, x5.device)
    tx, tg, tu = _tensor(x5), _tensor(g5), _tensor(u5)
    tgo = _tensor(go5) if go5 is not None else None
    stream = torch.cuda.current_stream(x5.device).cuda_stream
    with torch.cuda.device(x5.device):
        rc = lib.gradlev_eta_grad(ctypes.byref(desc), rd, ctypes.byref(tx), ctypes.byref(tg),
                                  ctypes.byref(tgo) if tgo is not None else None, ctypes.byref(tu),
                                  ctypes.c_void_p(deta.data_ptr()), ctypes.c_void_p(ws.data_ptr()),
                                  ws.numel(), ctypes.c_void_p(stream))
    _call(rc, "gradlev_eta_grad")
    return deta


def gate_grads(x, g_hat, eta, upstream, alpha=None, read="forward", g_out=None, dlog_alpha=None,
               deta=None, workspace=None):
    """Derivatives of one map's read with respect to its per-token gates (writes
    detached, gates learned: Sec. 3, practical architecture and training; Eq. 2).

    eta: per-token step sizes (tensor of the token shape of x, or a scalar); alpha:
    per-token retention or None (= 1).  read="forward": upstream = dL/dy ([.., d_out]);
    read="costate": upstream = dL/dg_in ([.., d_in]) and g_out is required.
    Returns (dlog_alpha, deta), fp32 [L,B,T,H]: alpha_t dL/dalpha_t (the derivative in
    log alpha_t) and dL/deta_t (written into dlog_alpha / deta when given: contiguous
    float32 of that shape).  64 x 64 bf16 maps.
    """
    lib = load_library()
    x5, g5, u5 = _as5(x), _as5(g_hat), _as5(upstream)
    go5 = _as5(g_out) if g_out is not None else None
    _check_same(x5, g5, u5, go5)
    if not x5.is_cuda:
        raise ValueError("tensors must be on a CUDA device")
    rd = {"forward": 0, "costate": 1}[read]
    if rd == 1 and go5 is None:
        raise ValueError("the costate read needs g_out")
    L, B, T, H, d_in = x5.shape
    d_out = g5.shape[4]
    shape = (L, B, T, H)

    def per_token(v):
        if isinstance(v, torch.Tensor):
            return v.to(device=x5.device, dtype=torch.float32).reshape(shape).contiguous()
        return torch.full(shape, float(v), dtype=torch.float32, device=x5.device)

    et = per_token(eta)
    at = per_token(alpha) if alpha is not None else None
    desc = _desc(x5, d_out, _dtype_code(x5))
    def out(t):
        if t is None:
            return torch.empty(shape, dtype=torch.float32, device=x5.device)
        if t.dtype != torch.float32 or not t.is_contiguous() or t.numel() != L * B * T * H:
            raise ValueError("gate_grads outputs must be contiguous float32 [L,B,T,H] tensors")
        return t

    dla = out(dlog_alpha)
    deta = out(deta)
    nbytes = int(lib.gradlev_gate_grads_workspace_bytes(ctypes.byref(desc), rd))
    ws = workspace if workspace is not None else _workspace(nbytes, x5.device)
    tx, tg, tu = _tensor(x5), _tensor(g5), _tensor(u5)
    tgo = _tensor(go5) if go5 is not None else None
    stream = torch.cuda.current_stream(x5.device).cuda_stream
    ptr = lambda t: ctypes.c_void_p(t.data_ptr()) if t is not None else None
    with torch.cuda.device(x5.device):
        rc = lib.gradlev_gate_grads(ctypes.byref(desc), rd, ctypes.byref(tx), ctypes.byref(tg),
                                    ptr(et), ptr(at), ctypes.byref(tgo) if tgo is not None else None,
                                    ctypes.byref(tu), ptr(dla), ptr(deta),
                                    ctypes.c_void_p(ws.data_ptr()), ws.numel(), ctypes.c_void_p(stream))
    _call(rc, "gradlev_gate_grads")
    return dla, deta
