"""GPU parity of the deployment calls (decode_read / decode_write) against the
fp64 oracle.

Deployment updates each map from its true costate after the token is scored
(Sec. 3; Appendix A).  For one map whose costates g_t are supplied, that learner
is the oracle's sequential learner with the written costates set to g_t and the
costate read queried by the same g_t; for the two-layer MLP it is the oracle's
deployment mode (layer 1 writes its reconstructed gz_t).  Every case runs the
CUDA calls token by token on the same seeded inputs and compares every read.
"""
import zlib

import numpy as np
import pytest
import torch

import oracle
from parity_util import TOL, assert_parity, rel_l2

gl = pytest.importorskip("paper_2609_34174_gb300")

pytestmark = pytest.mark.gpu


def _gen(seed):
    g = torch.Generator()
    g.manual_seed(seed)
    return g


def _problem(L, B, H, T, din, dout, dtype, seed):
    r = _gen(seed)
    x = torch.randn(L, B, T, H, din, generator=r) / np.sqrt(din)
    g = torch.randn(L, B, T, H, dout, generator=r)
    W0 = torch.randn(L, H, dout, din, generator=r) / np.sqrt(din)
    return x.to(dtype), g.to(dtype), W0


def _f64(t):
    return t.to(torch.float64).numpy()


def _run_linear(x, g, W0, eta_t, alpha_t, eta_unit=None):
    """Token-by-token deployment on the GPU; returns (y, g_in) as [L,B,T,H,w] cpu tensors."""
    L, B, T, H, din = x.shape
    dout = g.shape[-1]
    xd, gd, Wd = x.cuda(), g.cuda(), W0.cuda()
    delta = torch.zeros(L, B, H, dout, din, dtype=torch.float32, device="cuda")
    ys, gis = [], []
    for t in range(T):
        ys.append(gl.decode_read(xd[:, :, t], Wd, delta))
        eta = eta_unit if eta_unit is not None else float(eta_t[t])
        alpha = None if alpha_t is None else float(alpha_t[t])
        gis.append(gl.decode_write(xd[:, :, t], gd[:, :, t], Wd, delta, eta, alpha=alpha))
    torch.cuda.synchronize()
    return torch.stack(ys, 2).cpu(), torch.stack(gis, 2).cpu()


CASES = {
    # (L, B, H, T, d_in, d_out, dtype, gated)
    "64x64-bf16-gated-reset": (2, 2, 3, 40, 64, 64, torch.bfloat16, True),
    "96x72-f32": (1, 1, 2, 30, 96, 72, torch.float32, False),
    "1024x300-bf16-row-tiles": (1, 2, 1, 10, 1024, 300, torch.bfloat16, False),
    "4096x40-f32-many-strips": (1, 1, 1, 6, 4096, 40, torch.float32, True),
    "8x5-bf16-tiny": (1, 3, 1, 25, 8, 5, torch.bfloat16, False),
    "160x33-f32-partial-strip": (1, 1, 1, 20, 160, 33, torch.float32, True),
    "256x1000-bf16-tiles-and-strips": (2, 1, 2, 6, 256, 1000, torch.bfloat16, False),
    "4x3-f32-one-piece": (1, 2, 1, 12, 4, 3, torch.float32, False),
}


@pytest.mark.parametrize("case", sorted(CASES))
def test_decode_linear_matches_oracle(case):
    L, B, H, T, din, dout, dtype, gated = CASES[case]
    x, g, W0 = _problem(L, B, H, T, din, dout, dtype, seed=zlib.crc32(case.encode()) % 10000)
    rng = np.random.default_rng(7)
    eta_t = rng.uniform(0.05, 0.15, T) if gated else np.full(T, 0.1)
    alpha_t = None
    if gated:
        alpha_t = rng.uniform(0.85, 1.0, T)
        alpha_t[T // 2] = 0.0  # a reset
    y, gin = _run_linear(x, g, W0, eta_t, alpha_t)
    units = [(l, b, h) for l in range(L) for b in range(B) for h in range(H)]
    xu = np.stack([_f64(x[l, b, :, h]) for (l, b, h) in units])
    gu = np.stack([_f64(g[l, b, :, h]) for (l, b, h) in units])
    wu = np.stack([_f64(W0[l, h]) for (l, b, h) in units])
    yr, gr = oracle.linear_scan(xu, gu, wu, eta_t, alpha=alpha_t, gout=gu)
    yg = np.stack([_f64(y[l, b, :, h]) for (l, b, h) in units])
    gg = np.stack([_f64(gin[l, b, :, h]) for (l, b, h) in units])
    key = "bf16" if dtype == torch.bfloat16 else "f32"
    tol = TOL[key]
    assert_parity(f"{case} y", yg, yr, key)
    assert_parity(f"{case} g_in", gg, gr, key)
    # the fast weights matter: the slow-only reads differ by far more than the tolerance
    y0, _ = oracle.linear_scan(xu, gu, wu, 0.0)
    assert rel_l2(y0, yr) > 5 * tol


def test_decode_per_unit_step_sizes():
    """eta given per unit ([L,B,H]): each unit follows its own learner."""
    L, B, H, T, din, dout = 1, 2, 2, 16, 64, 128
    x, g, W0 = _problem(L, B, H, T, din, dout, torch.float32, seed=11)
    eta_u = torch.tensor([0.02, 0.05, 0.1, 0.2]).reshape(L, B, H)
    y, gin = _run_linear(x, g, W0, None, None, eta_unit=eta_u.cuda())
    for i, (l, b, h) in enumerate([(0, b, h) for b in range(B) for h in range(H)]):
        yr, gr = oracle.linear_scan(_f64(x[l, b, :, h])[None], _f64(g[l, b, :, h])[None],
                                    _f64(W0[l, h]), float(eta_u[l, b, h]),
                                    gout=_f64(g[l, b, :, h])[None])
        assert_parity(f"unit {i} y", _f64(y[l, b, :, h])[None], yr, "f32")
        assert_parity(f"unit {i} g_in", _f64(gin[l, b, :, h])[None], gr, "f32")


def test_decode_write_is_reproducible():
    """The column sums of g_in over several row tiles are added in a fixed order."""
    L, B, H, din, dout = 1, 2, 1, 1024, 700
    x, g, W0 = _problem(L, B, H, 1, din, dout, torch.bfloat16, seed=5)
    xd, gd, Wd = x[:, :, 0].cuda(), g[:, :, 0].cuda(), W0.cuda()
    base = torch.randn(L, B, H, dout, din, generator=_gen(6)).cuda() * 0.01
    outs = []
    for _ in range(2):
        delta = base.clone()
        gi = gl.decode_write(xd, gd, Wd, delta, 0.1)
        outs.append((gi.clone(), delta))
    torch.cuda.synchronize()
    assert torch.equal(outs[0][0], outs[1][0])
    assert torch.equal(outs[0][1], outs[1][1])


def _mlp_deploy_gpu(x, gout, W1, W2, eta1, eta2, act):
    """The deployed two-layer MLP of Appendix A, token by token."""
    B, T, d = x.shape
    m, k = W1.shape[0], W2.shape[0]
    xd, god = x.cuda(), gout.cuda()
    W1d, W2d = W1.cuda(), W2.cuda()
    D1 = torch.zeros(1, B, 1, m, d, device="cuda")
    D2 = torch.zeros(1, B, 1, k, m, device="cuda")
    rec = {key: [] for key in ("z", "h", "y", "gz")}
    for t in range(T):
        xt = xd[:, t].reshape(1, B, 1, d)
        z, h = gl.decode_read(xt, W1d, D1, act=act, want_act_out=True)
        y = gl.decode_read(h, W2d, D2)
        gy = god[:, t].reshape(1, B, 1, k)          # the scored token's costate dl/dy
        gz = gl.decode_write(h, gy, W2d, D2, eta2, act=act, z=z)   # sigma'(z) fused
        gl.decode_write(xt, gz, W1d, D1, eta1, want_g_in=False)
        for key, v in (("z", z), ("h", h), ("y", y), ("gz", gz)):
            rec[key].append(v.reshape(B, -1))
    torch.cuda.synchronize()
    return {key: torch.stack(v, 1).to(torch.float64).cpu().numpy() for key, v in rec.items()}


@pytest.mark.parametrize("shape", [(2, 24, 128, 512, 128), (2, 4, 1024, 4096, 1024)],
                         ids=["128-512-128", "paper-1024-4096-1024"])
def test_decode_mlp_deployment(shape):
    """Appendix A deployed: layer 2 writes the scored costate, layer 1 writes its
    reconstructed gz (with sigma' fused in the layer-2 write)."""
    B, T, d, m, k = shape
    r = _gen(31 + d)
    x = (torch.randn(B, T, d, generator=r)).to(torch.bfloat16)
    gout = (torch.randn(B, T, k, generator=r) * 0.5).to(torch.bfloat16)
    W1 = torch.randn(m, d, generator=r) / np.sqrt(d)
    W2 = torch.randn(k, m, generator=r) / np.sqrt(m)
    eta1, eta2 = 0.5 / d, 0.5 / m
    out = _mlp_deploy_gpu(x, gout, W1, W2, eta1, eta2, "gelu_tanh")
    ref = oracle.mlp_deploy(_f64(x), _f64(W1), _f64(W2), eta1, eta2, gout=_f64(gout),
                            act=oracle.ACT_GELU_TANH)
    for key in ("z", "h", "y", "gz"):
        assert_parity(key, out[key], ref[key], "bf16")
