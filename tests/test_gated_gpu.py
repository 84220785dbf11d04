"""GPU parity of the gated scans (Sec. 3 "Observation", Eq. 2 with per-token step
sizes eta_t and retention alpha_t, decay centred at W0) against the fp64 oracle,
which runs the same recurrence token by token.

Per-token eta_t alone takes the chunked kernels on eta-scaled proposals;
with alpha_t, bf16 64 x 64 maps run the tensor-core retention kernel (chunks of
128 tokens; few long units cut into segments whose states are carried) and
every other shape the token-serial kernels.  alpha_t = 0 marks resets (the fast
weights return to W0, as at a document boundary).
"""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from parity_util import TOL, assert_parity, lbthw_units, rel_l2

gl = pytest.importorskip("paper_2609_34174_gb300")

pytestmark = pytest.mark.gpu


def _gates(wl, seed, with_alpha, resets=True):
    g = torch.Generator().manual_seed(seed)
    shape = (wl.L, wl.B, wl.T, wl.H)
    eta = torch.rand(shape, generator=g, dtype=torch.float64) * (2 * wl.eta)
    alpha = None
    if with_alpha:
        alpha = 0.9 + 0.1 * torch.rand(shape, generator=g, dtype=torch.float64)
        if resets:
            alpha[..., wl.T // 3, :] = 0.0      # a document boundary
            alpha[..., (2 * wl.T) // 3, :] = 0.0
    return eta.float(), (alpha.float() if alpha is not None else None)


def _oracle(inputs, eta, alpha, wl):
    """fp64 oracle per unit with that unit's gate sequences."""
    f64 = lambda t: t.double().cpu().numpy()
    x, g, go, W0 = f64(inputs["x"]), f64(inputs["g_hat"]), f64(inputs["g_out"]), f64(inputs["W0"])
    e, a = f64(eta), (f64(alpha) if alpha is not None else None)
    ys, gs = np.zeros(x.shape[:-1] + (g.shape[-1],)), np.zeros(x.shape)
    for l in range(wl.L):
        for b in range(wl.B):
            for h in range(wl.H):
                y, gin = oracle.linear_scan(x[l, b, :, h][None], g[l, b, :, h][None], W0[l, h],
                                            e[l, b, :, h], alpha=None if a is None else a[l, b, :, h],
                                            gout=go[l, b, :, h][None])
                ys[l, b, :, h] = y[0]
                gs[l, b, :, h] = gin[0]
    return ys, gs


def _check(name, out, ref, tol):
    """Whole-output, per-unit and per-row bounds; out and ref [L,B,T,H,w]."""
    key = "f32" if tol == TOL["f32"] else "bf16"
    assert_parity(name, lbthw_units(out), lbthw_units(ref), key)


CASES = {
    # (workload, resize, alpha?)
    "eta_t-chunked-64": ("c5", dict(L=1, B=2, H=2, T=700), False),
    "eta_t-segmented-64": ("c4", dict(B=1, H=2, T=3000), False),
    "eta_t-chunked-128": ("c2", dict(B=1, H=2, T=900), False),
    "eta_t-wide-256x512": ("c2", dict(B=1, H=1, T=600, d_in=256, d_out=512, w_std=1 / 16), False),
    "alpha-serial-64": ("c5", dict(L=1, B=2, H=2, T=700), True),
    "alpha-serial-128x64": ("c2", dict(B=1, H=2, T=500, d_in=128, d_out=64), True),
    "alpha-serial-fp32": ("c1", dict(T=300), True),
    # forward read 48 wide (register kernel, one quarter of each row's inputs empty,
    # a 40-row output tile); costate read 40 wide (shared-memory kernel)
    "alpha-serial-48x40": ("c2", dict(B=1, H=2, T=333, d_in=48, d_out=40, w_std=1 / 7), True),
}


@pytest.mark.parametrize("case", sorted(CASES))
def test_gated_scans(case):
    key, kw, with_alpha = CASES[case]
    wl = W.workload(key).resized(**kw)
    inputs = W.make_linear(wl)
    eta, alpha = _gates(wl, 4242 + wl.T, with_alpha)
    dev = {k: (v.cuda() if isinstance(v, torch.Tensor) else v) for k, v in inputs.items()}
    y = gl.forward_scan(dev["x"], dev["g_hat"], dev["W0"], eta.cuda(),
                        alpha=alpha.cuda() if alpha is not None else None)
    gin = gl.costate_scan(dev["x"], dev["g_hat"], dev["W0"], eta.cuda(), dev["g_out"],
                          alpha=alpha.cuda() if alpha is not None else None)
    torch.cuda.synchronize()
    yr, gr = _oracle(inputs, eta, alpha, wl)
    tol = TOL["f32"] if wl.dtype == "f32" else TOL["bf16"]
    _check(f"{case} forward", y, yr, tol)
    _check(f"{case} costate", gin, gr, tol)


def test_reset_restarts_from_slow_weights():
    """Right after a reset (alpha = 0 at token r) the fast weights are
    W0 - eta_r ghat_r x_r^T, so the read at r+1 sees only that one write: the
    outputs after the reset do not depend on any token before r."""
    wl = W.workload("c5").resized(L=1, B=1, H=1, T=400)
    inputs = W.make_linear(wl)
    eta, alpha = _gates(wl, 7, True, resets=False)
    alpha[..., 200, :] = 0.0
    dev = {k: (v.cuda() if isinstance(v, torch.Tensor) else v) for k, v in inputs.items()}
    y1 = gl.forward_scan(dev["x"], dev["g_hat"], dev["W0"], eta.cuda(), alpha=alpha.cuda())
    x2 = dev["x"].clone()
    g2 = dev["g_hat"].clone()
    x2[:, :, :200] = torch.randn_like(x2[:, :, :200].float()).to(x2.dtype)
    g2[:, :, :200] = torch.randn_like(g2[:, :, :200].float()).to(g2.dtype)
    y2 = gl.forward_scan(x2, g2, dev["W0"], eta.cuda(), alpha=alpha.cuda())
    torch.cuda.synchronize()
    assert torch.equal(y1[:, :, 201:], y2[:, :, 201:])
    assert not torch.equal(y1[:, :, 150:200], y2[:, :, 150:200])


def test_constant_gates_match_plain_scan():
    """eta_t = eta everywhere and alpha = 1 is the plain scan (Eq. 3)."""
    wl = W.workload("c5").resized(L=1, B=1, H=2, T=500)
    inputs = W.make_linear(wl)
    dev = {k: (v.cuda() if isinstance(v, torch.Tensor) else v) for k, v in inputs.items()}
    shape = (wl.L, wl.B, wl.T, wl.H)
    y_plain = gl.forward_scan(dev["x"], dev["g_hat"], dev["W0"], wl.eta)
    y_serial = gl.forward_scan(dev["x"], dev["g_hat"], dev["W0"], wl.eta,
                               alpha=torch.ones(shape, device="cuda"))
    torch.cuda.synchronize()
    err = rel_l2(y_serial.double().cpu().numpy(), y_plain.double().cpu().numpy())
    assert err <= TOL["bf16"], f"serial vs chunked rel-L2 {err:.3e}"


# The retention path for bf16 64 x 64 maps runs in chunks of 128 tokens, built
# from 8-token pieces.  These cases put the chunk and piece boundaries, resets and
# odd gates where a chunked form of Eq. 2 could go wrong: T below, at and just past
# one and two chunks; resets on the last and first token of a piece and of a chunk
# and two in a row; a negative alpha; many units.
CHUNK_T = [1, 37, 64, 65, 127, 128, 129, 191, 255, 256, 257, 1000]


def _chunk_gates(shape, T, seed, resets=(7, 8, 63, 64, 127, 128, 130, 131, 500)):
    g = torch.Generator().manual_seed(seed)
    eta = torch.rand(shape, generator=g, dtype=torch.float64) * 0.04
    alpha = 0.85 + 0.15 * torch.rand(shape, generator=g, dtype=torch.float64)
    for t in resets:
        if t < T:
            alpha[:, :, t, :] = 0.0
    if T > 20:
        alpha[:, :, 20, :] = -0.5
    return eta.float(), alpha.float()


@pytest.mark.parametrize("T", CHUNK_T)
def test_retention_chunk_boundaries(T):
    wl = W.workload("c5").resized(L=2, B=1, H=3, T=T)
    inputs = W.make_linear(wl)
    eta, alpha = _chunk_gates((wl.L, wl.B, wl.T, wl.H), T, 900 + T)
    dev = {k: (v.cuda() if isinstance(v, torch.Tensor) else v) for k, v in inputs.items()}
    y = gl.forward_scan(dev["x"], dev["g_hat"], dev["W0"], eta.cuda(), alpha=alpha.cuda())
    gin = gl.costate_scan(dev["x"], dev["g_hat"], dev["W0"], eta.cuda(), dev["g_out"],
                          alpha=alpha.cuda())
    torch.cuda.synchronize()
    yr, gr = _oracle(inputs, eta, alpha, wl)
    _check(f"T={T} forward", y, yr, TOL["bf16"])
    _check(f"T={T} costate", gin, gr, TOL["bf16"])


def test_retention_fused_activation_epilogues():
    """sigma(y) from the forward read and sigma'(z) (.) g_in from the costate read
    (the MLP's fused epilogues) on the retention path."""
    wl = W.workload("c5").resized(L=1, B=2, H=2, T=300)
    inputs = W.make_linear(wl)
    eta, alpha = _chunk_gates((wl.L, wl.B, wl.T, wl.H), wl.T, 77)
    dev = {k: (v.cuda() if isinstance(v, torch.Tensor) else v) for k, v in inputs.items()}
    gz = torch.Generator().manual_seed(78)
    z = torch.randn(dev["x"].shape, generator=gz).to(torch.bfloat16)
    y, hy = gl.forward_scan(dev["x"], dev["g_hat"], dev["W0"], eta.cuda(), act="gelu_tanh",
                            want_act_out=True, alpha=alpha.cuda())
    gin = gl.costate_scan(dev["x"], dev["g_hat"], dev["W0"], eta.cuda(), dev["g_out"],
                          act="gelu_tanh", z=z.cuda(), alpha=alpha.cuda())
    torch.cuda.synchronize()
    yr, gr = _oracle(inputs, eta, alpha, wl)
    _check("y", y, yr, TOL["bf16"])
    _check("sigma(y)", hy, oracle.act(oracle.ACT_GELU_TANH, y.double().cpu().numpy()), TOL["bf16"])
    want = oracle.act_deriv(oracle.ACT_GELU_TANH, z.double().numpy()) * gr
    _check("sigma'(z) g_in", gin, want, TOL["bf16"])


@pytest.mark.parametrize("offset", [0, 4], ids=["aligned-rows", "8-byte-rows"])
def test_retention_strided_views(offset):
    """Token rows taken from wider buffers: 16-byte aligned rows (the chunked
    kernel) and rows that start 8 bytes off (the token-serial kernel)."""
    wl = W.workload("c5").resized(L=1, B=2, H=2, T=200)
    inputs = W.make_linear(wl)
    eta, alpha = _chunk_gates((wl.L, wl.B, wl.T, wl.H), wl.T, 55)
    wide = {}
    for k in ("x", "g_hat", "g_out"):
        t = inputs[k]
        buf = torch.zeros(t.shape[:-1] + (96,), dtype=t.dtype)
        buf[..., offset:offset + 64] = t
        wide[k] = buf.cuda()[..., offset:offset + 64]
    W0 = inputs["W0"].cuda()
    y = gl.forward_scan(wide["x"], wide["g_hat"], W0, eta.cuda(), alpha=alpha.cuda())
    gin = gl.costate_scan(wide["x"], wide["g_hat"], W0, eta.cuda(), wide["g_out"],
                          alpha=alpha.cuda())
    torch.cuda.synchronize()
    yr, gr = _oracle(inputs, eta, alpha, wl)
    _check("forward", y, yr, TOL["bf16"])
    _check("costate", gin, gr, TOL["bf16"])


@pytest.mark.parametrize("T", [1500, 5000])
def test_retention_segments(T):
    """Few long units: the sequence is cut into segments (512 tokens here, the last
    one ragged) whose start states come from an aggregate pass and the affine carry
    (a, U) then (a', U') = (a' a, a' U + U').  Resets sit on, before and after
    segment boundaries, and a negative alpha inside a segment."""
    wl = W.workload("c4").resized(B=1, H=2, T=T)
    inputs = W.make_linear(wl)
    eta, alpha = _chunk_gates((wl.L, wl.B, wl.T, wl.H), T, 300 + T,
                              resets=(511, 512, 1023, 1025, 2047, 4095, 4096))
    if T > 3000:
        alpha[:, :, 3000, :] = -0.7
    dev = {k: (v.cuda() if isinstance(v, torch.Tensor) else v) for k, v in inputs.items()}
    y = gl.forward_scan(dev["x"], dev["g_hat"], dev["W0"], eta.cuda(), alpha=alpha.cuda())
    gin = gl.costate_scan(dev["x"], dev["g_hat"], dev["W0"], eta.cuda(), dev["g_out"],
                          alpha=alpha.cuda())
    torch.cuda.synchronize()
    yr, gr = _oracle(inputs, eta, alpha, wl)
    _check(f"T={T} segmented forward", y, yr, TOL["bf16"])
    _check(f"T={T} segmented costate", gin, gr, TOL["bf16"])


def test_retention_full_size_c4_every_unit():
    """The long-context workload at full size with retention (the bench's gated
    configuration): every unit and token row against the oracle."""
    import bench
    wl = W.workload("c4")
    inputs = W.make_linear(wl)
    gates = bench.make_gates(wl, "alpha", "cpu")
    eta, alpha = gates["eta_t"], gates["alpha_t"]
    dev = {k: (v.cuda() if isinstance(v, torch.Tensor) else v) for k, v in inputs.items()}
    y = gl.forward_scan(dev["x"], dev["g_hat"], dev["W0"], eta.cuda(), alpha=alpha.cuda())
    gin = gl.costate_scan(dev["x"], dev["g_hat"], dev["W0"], eta.cuda(), dev["g_out"],
                          alpha=alpha.cuda())
    torch.cuda.synchronize()
    yr, gr = _oracle(inputs, eta, alpha, wl)
    _check("c4 retention forward", y, yr, TOL["bf16"])
    _check("c4 retention costate", gin, gr, TOL["bf16"])


def test_retention_many_items_per_cta_odd_chunks():
    """More units than SMs, each of three chunks (257 tokens, the last ragged): every
    CTA runs several items whose chunk counts are odd, so the two chunk buffers
    (score, then P' and the state update) and the two output accumulators, with their
    barrier phases, alternate from one item to the next."""
    wl = W.workload("c5").resized(L=1, B=4, H=100, T=257)
    inputs = W.make_linear(wl)
    eta, alpha = _chunk_gates((wl.L, wl.B, wl.T, wl.H), wl.T, 4001)
    dev = {k: (v.cuda() if isinstance(v, torch.Tensor) else v) for k, v in inputs.items()}
    y = gl.forward_scan(dev["x"], dev["g_hat"], dev["W0"], eta.cuda(), alpha=alpha.cuda())
    gin = gl.costate_scan(dev["x"], dev["g_hat"], dev["W0"], eta.cuda(), dev["g_out"],
                          alpha=alpha.cuda())
    torch.cuda.synchronize()
    yr, gr = _oracle(inputs, eta, alpha, wl)
    _check("400 units x 3 chunks forward", y, yr, TOL["bf16"])
    _check("400 units x 3 chunks costate", gin, gr, TOL["bf16"])


def test_retention_segmented_many_items():
    """Segmented units with more items than SMs: 100 units of 1300 tokens cut into
    512 + 512 + 276 (four, four and three chunks), 300 items, so the aggregate pass
    and the scan each run several items of mixed chunk counts per CTA."""
    wl = W.workload("c4").resized(B=4, H=25, T=1300)
    inputs = W.make_linear(wl)
    eta, alpha = _chunk_gates((wl.L, wl.B, wl.T, wl.H), wl.T, 4002,
                              resets=(511, 512, 1023, 1024, 1299))
    dev = {k: (v.cuda() if isinstance(v, torch.Tensor) else v) for k, v in inputs.items()}
    y = gl.forward_scan(dev["x"], dev["g_hat"], dev["W0"], eta.cuda(), alpha=alpha.cuda())
    gin = gl.costate_scan(dev["x"], dev["g_hat"], dev["W0"], eta.cuda(), dev["g_out"],
                          alpha=alpha.cuda())
    torch.cuda.synchronize()
    yr, gr = _oracle(inputs, eta, alpha, wl)
    _check("segmented 100 x 1300 forward", y, yr, TOL["bf16"])
    _check("segmented 100 x 1300 costate", gin, gr, TOL["bf16"])
