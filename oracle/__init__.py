"""The parity oracle for the GradLev scans (test infrastructure).

A plain fp64 CPU implementation of the sequential online learner
(GradLev Sec. 3, Eqs. 2-4, and the online MLP of Appendix A), its suffix read and
the derivatives of an outer objective with respect to the per-token gates
(Sec. 3, practical architecture and training), written in C
(``gradlev_oracle.c``) and loaded through ctypes, plus the per-token consistency
term of the training objective (Eq. 5) written out in numpy.  Only ``tests/``,
``__graft_entry__.smoke()`` and the ``cpu_baseline`` / ``--impl reference``
legs of ``bench.py`` may import this package.  It shares no code with the CUDA
library and never calls it.

Every function here takes numpy fp64 arrays (the caller upcasts the exact
bf16/fp32 tensors fed to the GPU) and returns fp64 arrays.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import sys

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "gradlev_oracle.c")
_LIB_PATH = os.path.join(_HERE, "_build", "liboracle.so")
_lib = None

ACT_NONE, ACT_GELU_TANH, ACT_GELU_ERF, ACT_TANH = 0, 1, 2, 3


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (-O2, OpenMP) into oracle/_build/."""
    os.makedirs(os.path.dirname(_LIB_PATH), exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".{os.getpid()}.tmp"
    # -ffp-contract=off: no fused multiply-add, so every product and sum is a
    # separately rounded fp64 operation, as written.
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-ffp-contract=off",
           "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is not None:
        return _lib
    build()
    lib = ctypes.CDLL(_LIB_PATH)
    P = ctypes.c_void_p
    I = ctypes.c_int
    lib.oracle_linear_batch.argtypes = [I, I, I, I, P, P, P, P, P, P, P, P, I]
    lib.oracle_linear_batch.restype = I
    lib.oracle_mlp_batch.argtypes = [I, I, I, I, I, I, P, P, P, P, P, P, P, P, P,
                                     P, P, P, P, P, P, I]
    lib.oracle_mlp_batch.restype = I
    lib.oracle_act.argtypes = [I, ctypes.c_double]
    lib.oracle_act.restype = ctypes.c_double
    lib.oracle_act_deriv.argtypes = [I, ctypes.c_double]
    lib.oracle_act_deriv.restype = ctypes.c_double
    lib.oracle_suffix_batch.argtypes = [I, I, I, I, P, P, P, P, I]
    lib.oracle_suffix_batch.restype = I
    lib.oracle_gate_grads_batch.argtypes = [I, I, I, I, P, P, P, P, P, P, P, P, I]
    lib.oracle_gate_grads_batch.restype = I
    lib.oracle_max_threads.argtypes = []
    lib.oracle_max_threads.restype = I
    _lib = lib
    return lib


def _f64(a):
    return np.ascontiguousarray(a, dtype=np.float64)


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _steps(v, T):
    """A scalar or [T] per-token coefficient as a contiguous fp64 [T] array."""
    a = np.asarray(v, dtype=np.float64)
    if a.ndim == 0:
        a = np.full((T,), float(a))
    if a.shape != (T,):
        raise ValueError(f"per-token coefficient must be scalar or [{T}], got {a.shape}")
    return np.ascontiguousarray(a)


def max_threads() -> int:
    return int(_load().oracle_max_threads())


def linear_scan(x, ghat, W0, eta, alpha=None, gout=None, want_y=True, nthreads=0):
    """Sequential learner for U independent linear maps (Sec. 3, Eqs. 2-4).

    x [U,T,d], ghat [U,T,m], W0 [U,m,d] (or [m,d], shared), eta scalar or [T],
    alpha None (= 1) or scalar/[T], gout [U,T,m] or None.
    Returns (y [U,T,m] or None, gin [U,T,d] or None): y_t = W_t x_t and
    gin_t = W_t^T gout_t, each read before the token-t write.
    """
    lib = _load()
    x = _f64(x)
    ghat = _f64(ghat)
    U, T, d = x.shape
    m = ghat.shape[2]
    if ghat.shape != (U, T, m):
        raise ValueError("ghat shape mismatch")
    W0 = _f64(W0)
    if W0.shape == (m, d):
        W0 = np.ascontiguousarray(np.broadcast_to(W0, (U, m, d)))
    if W0.shape != (U, m, d):
        raise ValueError("W0 shape mismatch")
    eta_a = _steps(eta, T)
    alpha_a = None if alpha is None else _steps(alpha, T)
    gout_a = None if gout is None else _f64(gout)
    if gout_a is not None and gout_a.shape != (U, T, m):
        raise ValueError("gout shape mismatch")
    y = np.empty((U, T, m)) if want_y else None
    gin = np.empty((U, T, d)) if gout_a is not None else None
    rc = lib.oracle_linear_batch(U, T, d, m, _ptr(x), _ptr(ghat), _ptr(W0), _ptr(eta_a),
                                 _ptr(alpha_a), _ptr(gout_a), _ptr(y), _ptr(gin), int(nthreads))
    if rc != 0:
        raise MemoryError("oracle_linear_batch could not allocate scratch")
    return y, gin


def linear_scan_docs(x, ghat, W0, eta, doc_start, alpha=None, gout=None):
    """Document resets (Appendix C, scan reads; Appendix E, packed documents): every
    read sees only the writes of its own document (since the latest start), so each
    document is its own sequential learner starting from W0.

    doc_start [U,T] booleans, True where a document begins (token 0 always begins
    one); eta and alpha as in linear_scan (scalar or [T], shared by the units), each
    document taking its own slice.  Returns (y [U,T,m], gin [U,T,d] or None).
    """
    x = _f64(x)
    ghat = _f64(ghat)
    U, T, d = x.shape
    m = ghat.shape[2]
    W0 = _f64(W0)
    starts = np.asarray(doc_start, dtype=bool)
    if starts.shape != (U, T):
        raise ValueError(f"doc_start must be [{U},{T}]")
    eta_a = _steps(eta, T)
    alpha_a = _steps(alpha, T) if alpha is not None else None
    y = np.empty((U, T, m))
    gin = np.empty((U, T, d)) if gout is not None else None
    for u in range(U):
        cuts = [0] + [t for t in range(1, T) if starts[u, t]] + [T]
        for a, b in zip(cuts[:-1], cuts[1:]):
            w0 = W0 if W0.ndim == 2 else W0[u]
            yy, gg = linear_scan(x[u:u + 1, a:b], ghat[u:u + 1, a:b], w0, eta_a[a:b],
                                 alpha=None if alpha_a is None else alpha_a[a:b],
                                 gout=None if gout is None else _f64(gout)[u:u + 1, a:b])
            y[u, a:b] = yy[0]
            if gin is not None:
                gin[u, a:b] = gg[0]
    return y, gin


def mlp_scan(x, ghz, ghy, W10, W20, eta1, eta2, act=ACT_GELU_TANH, alpha=None, gout=None,
             nthreads=0):
    """Sequential online MLP (Appendix A) for U independent sequences.

    Widths: input d, hidden m, output k.  x [U,T,d], ghz [U,T,m], ghy [U,T,k],
    W10 [m,d], W20 [k,m], gout [U,T,k] or None.
    Returns a dict with z, h [U,T,m], y [U,T,k] and, when gout is given,
    gh (= W2_t^T gout), gz (= sigma'(z) * gh) [U,T,m] and gx (= W1_t^T gz) [U,T,d].
    A proposal of None writes the true costate instead (deployment): ghz None
    writes gz_t, ghy None writes gout_t.
    """
    lib = _load()
    x = _f64(x)
    U, T, d = x.shape
    W10 = _f64(W10)
    W20 = _f64(W20)
    m = W10.shape[0]
    k = W20.shape[0]
    ghz = None if ghz is None else _f64(ghz)
    ghy = None if ghy is None else _f64(ghy)
    if W10.shape != (m, d) or W20.shape != (k, m):
        raise ValueError("mlp shape mismatch")
    if (ghz is not None and ghz.shape != (U, T, m)) or (ghy is not None and ghy.shape != (U, T, k)):
        raise ValueError("mlp proposal shape mismatch")
    if (ghz is None or ghy is None) and gout is None:
        raise ValueError("deployment (a proposal of None) needs gout")
    e1 = _steps(eta1, T)
    e2 = _steps(eta2, T)
    al = None if alpha is None else _steps(alpha, T)
    go = None if gout is None else _f64(gout)
    if go is not None and go.shape != (U, T, k):
        raise ValueError("gout shape mismatch")
    out = {"z": np.empty((U, T, m)), "h": np.empty((U, T, m)), "y": np.empty((U, T, k))}
    if go is not None:
        out.update(gh=np.empty((U, T, m)), gz=np.empty((U, T, m)), gx=np.empty((U, T, d)))
    rc = lib.oracle_mlp_batch(U, T, d, m, k, int(act), _ptr(x), _ptr(ghz), _ptr(ghy), _ptr(W10),
                              _ptr(W20), _ptr(e1), _ptr(e2), _ptr(al), _ptr(go),
                              _ptr(out["z"]), _ptr(out["h"]), _ptr(out["y"]),
                              _ptr(out.get("gh")), _ptr(out.get("gz")), _ptr(out.get("gx")),
                              int(nthreads))
    if rc != 0:
        raise MemoryError("oracle_mlp_batch could not allocate scratch")
    return out


def mlp_deploy(x, W10, W20, eta1, eta2, gout, act=ACT_GELU_TANH, alpha=None, nthreads=0):
    """The deployed online MLP (Sec. 3; Appendix A): after each scored target both
    layers write their true costates, gout_t at layer 2 and gz_t at layer 1.
    Same shapes and outputs as mlp_scan."""
    return mlp_scan(x, None, None, W10, W20, eta1, eta2, act=act, alpha=alpha, gout=gout,
                    nthreads=nthreads)


def suffix_scan(q, k, v, nthreads=0):
    """Anti-causal read r_s = sum_{t>s} (k_t . q_s) v_t for U independent units
    (outer gradients through the reads).  q, k [U,T,dq], v [U,T,dv] -> r [U,T,dv]."""
    lib = _load()
    q, k, v = _f64(q), _f64(k), _f64(v)
    U, T, dq = q.shape
    dv = v.shape[2]
    if k.shape != (U, T, dq) or v.shape[:2] != (U, T):
        raise ValueError("suffix_scan shape mismatch")
    r = np.empty((U, T, dv))
    if lib.oracle_suffix_batch(U, T, dq, dv, _ptr(q), _ptr(k), _ptr(v), _ptr(r), int(nthreads)):
        raise MemoryError("oracle_suffix_batch could not allocate scratch")
    return r


def gate_grads(x, ghat, eta, alpha, a, b, nthreads=0):
    """Derivatives of an outer objective with respect to the per-token gates of the
    learner (Sec. 3, practical architecture and training: the gates are learned and
    their derivatives kept, the writes detached).  Each read of W_t adds
    a_t^T W_t b_t: the forward read with outer gradient u takes a = u, b = x; the
    costate read with outer gradient w takes a = gout, b = w.

    x [U,T,d], ghat [U,T,m], eta and alpha scalar, [T] or [U,T], a [U,T,m], b [U,T,d].
    Returns (alpha_j dL/dalpha_j, dL/deta_j), each [U,T]: the first is the derivative
    in log alpha_j, <W_j - W0, R_j> alpha_j with R_j = sum_{s>j} prod_{j<r<s} alpha_r
    a_s b_s^T; the second -ghat_j^T R_j x_j."""
    lib = _load()
    x, ghat, a, b = _f64(x), _f64(ghat), _f64(a), _f64(b)
    U, T, d = x.shape
    m = ghat.shape[2]
    if ghat.shape != (U, T, m) or a.shape != (U, T, m) or b.shape != (U, T, d):
        raise ValueError("gate_grads shape mismatch")

    def gates(v):
        v = np.asarray(v, dtype=np.float64)
        return np.ascontiguousarray(np.broadcast_to(v, (T,)) if v.ndim == 0 else np.broadcast_to(v, (U, T)))

    eta_a = np.ascontiguousarray(np.broadcast_to(gates(eta), (U, T)))
    alpha_a = np.ascontiguousarray(np.broadcast_to(gates(1.0 if alpha is None else alpha), (U, T)))
    ga = np.empty((U, T))
    ge = np.empty((U, T))
    if lib.oracle_gate_grads_batch(U, T, d, m, _ptr(x), _ptr(ghat), _ptr(eta_a), _ptr(alpha_a),
                                   _ptr(a), _ptr(b), _ptr(ga), _ptr(ge), int(nthreads)):
        raise MemoryError("oracle_gate_grads_batch could not allocate scratch")
    return ga, ge


def consistency(proposal, target):
    """Per-token consistency term of the training objective (Sec. 3, Eq. 5; Appendix A,
    eq. consistency): ||ghat_t - gtilde_t||^2 / w for every token, where ghat is a
    proposed costate, gtilde the costate reconstructed at the same place and w their
    width.  The objective averages these terms over tokens (and, for an MLP, adds
    one such term per adapted map).  proposal, target [U,T,w] -> [U,T] in fp64."""
    p = _f64(proposal)
    g = _f64(target)
    if p.shape != g.shape or p.ndim < 1:
        raise ValueError("consistency: proposal and target shapes differ")
    w = p.shape[-1]
    diff = p - g
    return (diff * diff).sum(axis=-1) / w


def act(code, z):
    """sigma(z) elementwise in fp64 (the oracle's activation)."""
    lib = _load()
    f = np.vectorize(lambda v: lib.oracle_act(int(code), float(v)), otypes=[np.float64])
    return f(np.asarray(z, dtype=np.float64))


def act_deriv(code, z):
    """sigma'(z) elementwise in fp64 (the oracle's derivative)."""
    lib = _load()
    f = np.vectorize(lambda v: lib.oracle_act_deriv(int(code), float(v)), otypes=[np.float64])
    return f(np.asarray(z, dtype=np.float64))


if __name__ == "__main__":  # pragma: no cover
    print(build(force="--force" in sys.argv))
