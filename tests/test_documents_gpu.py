"""GPU parity of document resets for packed sequences against the fp64 oracle's
per-document learners.

A read sees only the writes of its own document, those since the latest start
(Appendix C, scan reads; Appendix E, resets at document boundaries).  On the GPU
the starts are folded into the gates of Eq. 2 (alpha = eta = 0 on the token
before each start) and the gated scans run; the oracle instead runs one
sequential learner per document from W0, so the two share no reading of the
rule beyond the rule itself.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
import workloads as W
from parity_util import TOL, assert_parity, lbthw_units, rel_l2

gl = pytest.importorskip("paper_2609_34174_gb300")

pytestmark = pytest.mark.gpu


def _doc_start(B, T, seed, extra=()):
    """Random document lengths (1 to 89 tokens) plus the given starts, per batch row."""
    g = np.random.default_rng(seed)
    ds = np.zeros((B, T), dtype=bool)
    for b in range(B):
        t = 0
        while True:
            t += int(g.integers(1, 90))
            if t >= T:
                break
            ds[b, t] = True
        for c in extra:
            if c < T:
                ds[b, c] = True
    return ds


def _oracle_docs(inputs, ds, eta, alpha, wl):
    f64 = lambda t: t.double().cpu().numpy()
    x, g, go, W0 = f64(inputs["x"]), f64(inputs["g_hat"]), f64(inputs["g_out"]), f64(inputs["W0"])
    ys, gs = np.zeros(x.shape[:-1] + (g.shape[-1],)), np.zeros(x.shape)
    for l in range(wl.L):
        for b in range(wl.B):
            for h in range(wl.H):
                e = eta if not isinstance(eta, torch.Tensor) else f64(eta[l, b, :, h])
                a = None if alpha is None else f64(alpha[l, b, :, h])
                y, gin = oracle.linear_scan_docs(x[l, b, :, h][None], g[l, b, :, h][None], W0[l, h],
                                                 e, ds[b][None], alpha=a, gout=go[l, b, :, h][None])
                ys[l, b, :, h] = y[0]
                gs[l, b, :, h] = gin[0]
    return ys, gs


CASES = {
    # (workload, resize, per-token gates?)  64 x 64 bf16 runs the chunked retention
    # kernel; the others the token-serial kernels
    "chunked-64-scalar-eta": ("c5", dict(L=2, B=2, H=2, T=700), False),
    "chunked-64-eta_t-alpha_t": ("c5", dict(L=1, B=2, H=3, T=500), True),
    "serial-128x64-bf16": ("c2", dict(B=2, H=1, T=300, d_in=128, d_out=64), False),
    "serial-fp32": ("c1", dict(B=2, T=257), True),
}


@pytest.mark.parametrize("case", sorted(CASES))
def test_document_resets_match_per_document_learners(case):
    key, kw, per_token = CASES[case]
    wl = W.workload(key).resized(**kw)
    inputs = W.make_linear(wl)
    ds = _doc_start(wl.B, wl.T, 31 + wl.T, extra=(1, 63, 64, 65, 128, 129))
    eta, alpha = wl.eta, None
    if per_token:
        g = torch.Generator().manual_seed(32)
        shape = (wl.L, wl.B, wl.T, wl.H)
        eta = torch.rand(shape, generator=g) * (2 * wl.eta)
        alpha = 0.9 + 0.1 * torch.rand(shape, generator=g)
    dev = {k: (v.cuda() if isinstance(v, torch.Tensor) else v) for k, v in inputs.items()}
    e_dev = eta.cuda() if isinstance(eta, torch.Tensor) else eta
    a_dev = alpha.cuda() if alpha is not None else None
    dsd = torch.from_numpy(ds).cuda()
    y = gl.forward_scan(dev["x"], dev["g_hat"], dev["W0"], e_dev, alpha=a_dev, doc_start=dsd)
    gin = gl.costate_scan(dev["x"], dev["g_hat"], dev["W0"], e_dev, dev["g_out"], alpha=a_dev,
                          doc_start=dsd)
    torch.cuda.synchronize()
    yr, gr = _oracle_docs(inputs, ds, eta, alpha, wl)
    tol = TOL["f32"] if wl.dtype == "f32" else TOL["bf16"]
    key = "f32" if wl.dtype == "f32" else "bf16"
    for name, out, ref in (("forward", y, yr), ("costate", gin, gr)):
        assert_parity(f"{case} {name}", lbthw_units(out), lbthw_units(ref), key)
    # the first token of every document reads W0 alone
    f64 = lambda t: t.double().cpu().numpy()
    x, W0 = f64(inputs["x"]), f64(inputs["W0"])
    for b in range(wl.B):
        for t in np.flatnonzero(ds[b])[:8]:
            want = np.einsum("lhmd,lhd->lhm", W0, x[:, b, t])
            got = f64(y[:, b, t])
            assert rel_l2(got, want) <= tol


def _expected_gates(ds, L, H, eta, alpha):
    B, T = ds.shape
    e = np.broadcast_to(np.asarray(eta, dtype=np.float32), (L, B, T, H)).copy()
    a = (np.ones((L, B, T, H), dtype=np.float32) if alpha is None
         else np.broadcast_to(np.asarray(alpha, dtype=np.float32), (L, B, T, H)).copy())
    for b in range(B):
        for t in range(T - 1):
            if ds[b, t + 1]:
                e[:, b, t, :] = 0.0
                a[:, b, t, :] = 0.0
    return e, a


def test_document_gates_values():
    """The folded gate arrays, bit for bit: inputs kept except eta = alpha = 0 on the
    token before each start; a start flag on token 0 changes nothing."""
    L, B, T, H = 2, 3, 150, 4
    x = torch.zeros(L, B, T, H, 8, dtype=torch.bfloat16, device="cuda")
    ds = _doc_start(B, T, 5, extra=(0, 1, 149))
    ds_t = torch.from_numpy(ds.astype(np.uint8)).cuda()
    e, a = gl.document_gates(ds_t, x, 0.125)
    we, wa = _expected_gates(ds, L, H, 0.125, None)
    assert np.array_equal(e.cpu().numpy(), we) and np.array_equal(a.cpu().numpy(), wa)
    g = torch.Generator().manual_seed(6)
    et = torch.rand(L, B, T, H, generator=g)
    at = torch.rand(L, B, T, H, generator=g)
    e, a = gl.document_gates(ds_t, x, et.cuda(), at.cuda())
    we, wa = _expected_gates(ds, L, H, et.numpy(), at.numpy())
    assert np.array_equal(e.cpu().numpy(), we) and np.array_equal(a.cpu().numpy(), wa)


def test_document_gates_in_place_through_the_c_abi():
    """eta_out may be eta_t and alpha_out alpha_t."""
    from paper_2609_34174_gb300 import _binding as _B
    lib = _B.load_library()
    L, B, T, H = 1, 2, 97, 3
    ds = _doc_start(B, T, 8)
    g = torch.Generator().manual_seed(9)
    et = torch.rand(L, B, T, H, generator=g)
    at = torch.rand(L, B, T, H, generator=g)
    we, wa = _expected_gates(ds, L, H, et.numpy(), at.numpy())
    et_d, at_d = et.cuda(), at.cuda()
    ds_d = torch.from_numpy(ds.astype(np.uint8)).cuda()
    desc = _B._Desc(L, B, T, H, 0, 0, 0, 0)
    p = lambda t: ctypes.c_void_p(t.data_ptr())
    rc = lib.gradlev_document_gates(ctypes.byref(desc), p(ds_d), 0.0, p(et_d), p(at_d), p(et_d),
                                    p(at_d), ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert rc == 0
    torch.cuda.synchronize()
    assert np.array_equal(et_d.cpu().numpy(), we) and np.array_equal(at_d.cpu().numpy(), wa)


def test_document_resets_empty_sequence():
    x = torch.zeros(1, 2, 0, 2, 64, dtype=torch.bfloat16, device="cuda")
    W0 = torch.zeros(1, 2, 64, 64, device="cuda")
    ds = torch.zeros(2, 0, dtype=torch.bool, device="cuda")
    y = gl.forward_scan(x, x, W0, 0.01, doc_start=ds)
    torch.cuda.synchronize()
    assert y.shape == (1, 2, 0, 2, 64)
