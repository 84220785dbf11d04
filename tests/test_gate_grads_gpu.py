"""GPU parity of the derivatives with respect to the per-token gates (eta_t and the
retention alpha_t of Eq. 2; Sec. 3, practical architecture and training: gates
learned, writes detached) against the fp64 oracle, which walks the learner forwards
and its decayed suffix state backwards token by token.  The oracle is pinned to
central differences of the sequential learner (tests/test_oracle_pins.py).

Outputs: alpha_t dL/dalpha_t (the derivative in log alpha_t) and dL/deta_t, fp32
[L, B, T, H], compared per unit and per token with the bf16 bounds of the scans.
"""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from parity_util import assert_parity, lbthw_units

gl = pytest.importorskip("paper_2609_34174_gb300")

pytestmark = pytest.mark.gpu


def _rand(shape, seed, scale=1.0):
    g = torch.Generator().manual_seed(seed)
    return (torch.randn(*shape, generator=g) * scale).to(torch.bfloat16)


def _gates(shape, seed, resets=True, with_alpha=True):
    g = torch.Generator().manual_seed(seed)
    eta = (torch.rand(shape, generator=g, dtype=torch.float64) * 0.04).float()
    if not with_alpha:
        return eta, None
    alpha = 0.85 + 0.15 * torch.rand(shape, generator=g, dtype=torch.float64)
    T = shape[2]
    if resets:
        for t in (7, 127, 128, 300, 511, 512, 1025):
            if t < T:
                alpha[:, :, t, :] = 0.0
        if T > 40:
            alpha[:, :, 40, :] = -0.5
    return eta, alpha.float()


def _oracle(x, gh, go, u, eta, alpha, read):
    """Per unit: (alpha dL/dalpha, dL/deta) [U, T] with that unit's gate sequences."""
    xu, gu, uu = lbthw_units(x), lbthw_units(gh), lbthw_units(u)
    eu = lbthw_units(eta)
    au = lbthw_units(alpha) if alpha is not None else np.ones_like(eu)
    if read == "forward":
        a, b = uu, xu
    else:
        a, b = lbthw_units(go), uu
    return oracle.gate_grads(xu, gu, eu, au, a, b)


def _run(L, B, T, H, read, seed, resets=True, with_alpha=True):
    x = _rand((L, B, T, H, 64), seed, 1 / 8)
    gh = _rand((L, B, T, H, 64), seed + 1, 0.5)
    go = _rand((L, B, T, H, 64), seed + 2, 0.5)
    u = _rand((L, B, T, H, 64), seed + 3)
    eta, alpha = _gates((L, B, T, H), seed + 4, resets, with_alpha)
    dla, de = gl.gate_grads(x.cuda(), gh.cuda(), eta.cuda(), u.cuda(),
                            alpha=alpha.cuda() if alpha is not None else None, read=read,
                            g_out=go.cuda() if read == "costate" else None)
    torch.cuda.synchronize()
    ra, re = _oracle(x, gh, go, u, eta, alpha, read)
    return lbthw_units(dla.cpu()), lbthw_units(de.cpu()), ra, re


CASES = {
    # (L, B, T, H): one token, below / at / past one chunk of 128, several units, a
    # long sequence whose chunk states are carried over 24 chunks (resets on and next
    # to chunk boundaries, a negative alpha)
    "T1": (1, 1, 1, 2),
    "T100": (1, 2, 100, 2),
    "T128": (1, 1, 128, 3),
    "T129": (2, 1, 129, 2),
    "T700": (1, 2, 700, 2),
    "T3000": (1, 1, 3000, 2),
}


@pytest.mark.parametrize("read", ["forward", "costate"])
@pytest.mark.parametrize("case", sorted(CASES))
def test_gate_grads_match_oracle(case, read):
    L, B, T, H = CASES[case]
    dla, de, ra, re = _run(L, B, T, H, read, 100 + T)
    assert_parity(f"{case} {read} dlog_alpha", dla, ra, "bf16")
    assert_parity(f"{case} {read} deta", de, re, "bf16")
    assert np.all(dla[:, 0] == 0.0)  # no write precedes the first token


@pytest.mark.parametrize("read", ["forward", "costate"])
def test_gate_grads_unit_retention(read):
    """alpha = None (retention 1): dL/deta equals the step-size gradient of the
    undecayed suffix read (eta_grad), and the log-alpha derivative is that of alpha = 1."""
    L, B, T, H = 1, 2, 600, 2
    dla, de, ra, re = _run(L, B, T, H, read, 71, with_alpha=False)
    assert_parity(f"unit retention {read} dlog_alpha", dla, ra, "bf16")
    assert_parity(f"unit retention {read} deta", de, re, "bf16")


def test_gate_grads_strided_views():
    """Token tensors that are feature slices of a wider buffer."""
    L, B, T, H = 1, 2, 400, 2
    big = _rand((L, B, T, H, 192), 81, 1 / 8).cuda()
    x, gh, u = big[..., :64], big[..., 64:128], big[..., 128:]
    eta, alpha = _gates((L, B, T, H), 82)
    dla, de = gl.gate_grads(x, gh, eta.cuda(), u, alpha=alpha.cuda())
    torch.cuda.synchronize()
    ra, re = _oracle(x.cpu(), gh.cpu(), None, u.cpu(), eta, alpha, "forward")
    assert_parity("strided dlog_alpha", lbthw_units(dla.cpu()), ra, "bf16")
    assert_parity("strided deta", lbthw_units(de.cpu()), re, "bf16")


def _bench_upstream(wl, seed):
    return _rand((wl.L, wl.B, wl.T, wl.H, wl.d_out), seed)


def test_gate_grads_full_size_c4_every_unit():
    """The long-context workload at full size with the bench's retention gates: every
    unit and token against the oracle."""
    import bench
    wl = W.workload("c4")
    inp = W.make_linear(wl)
    g = bench.make_gates(wl, "alpha", "cpu")
    u = _bench_upstream(wl, 91)
    dla, de = gl.gate_grads(inp["x"].cuda(), inp["g_hat"].cuda(), g["eta_t"].cuda(), u.cuda(),
                            alpha=g["alpha_t"].cuda())
    torch.cuda.synchronize()
    ra, re = _oracle(inp["x"], inp["g_hat"], None, u, g["eta_t"], g["alpha_t"], "forward")
    assert_parity("c4 dlog_alpha", lbthw_units(dla.cpu()), ra, "bf16")
    assert_parity("c4 deta", lbthw_units(de.cpu()), re, "bf16")


def test_gate_grads_full_size_c5_every_unit():
    """The layer-sweep workload at full size (1152 units of 8192 tokens), costate read,
    in the configuration the bench times: every unit and token against the oracle,
    one layer at a time."""
    import bench
    wl = W.workload("c5")
    inp = W.make_linear(wl)
    g = bench.make_gates(wl, "alpha", "cpu")
    u = _rand((wl.L, wl.B, wl.T, wl.H, wl.d_in), 92)
    dla, de = gl.gate_grads(inp["x"].cuda(), inp["g_hat"].cuda(), g["eta_t"].cuda(), u.cuda(),
                            alpha=g["alpha_t"].cuda(), read="costate", g_out=inp["g_out"].cuda())
    torch.cuda.synchronize()
    dla, de = dla.cpu(), de.cpu()
    from parity_util import Parity
    pa, pe = Parity("c5 dlog_alpha", "bf16"), Parity("c5 deta", "bf16")
    for l in range(wl.L):
        sl = lambda t: t[l:l + 1]
        ra, re = _oracle(sl(inp["x"]), sl(inp["g_hat"]), sl(inp["g_out"]), sl(u), sl(g["eta_t"]),
                         sl(g["alpha_t"]), "costate")
        pa.add(lbthw_units(sl(dla)), ra)
        pe.add(lbthw_units(sl(de)), re)
    pa.check()
    pe.check()


def test_gate_grads_rejects_other_shapes():
    x = torch.zeros((1, 1, 10, 1, 32), dtype=torch.bfloat16, device="cuda")
    eta = torch.zeros((1, 1, 10, 1), device="cuda")
    with pytest.raises(gl.GradLevError):
        gl.gate_grads(x, x, eta, x)
