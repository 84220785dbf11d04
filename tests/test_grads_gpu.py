"""GPU parity of the anti-causal suffix read and the step-size gradients built on
it (outer gradients through the reads, writes detached) against the fp64 oracle.
The oracle's suffix read is pinned to finite differences of the sequential
learner in every eta_t (tests/test_oracle_pins.py)."""
import numpy as np
import pytest
import torch

import oracle
from parity_util import TOL, rel_l2

gl = pytest.importorskip("paper_2609_34174_gb300")

pytestmark = pytest.mark.gpu


def _rand(shape, seed, dtype, scale=1.0):
    g = torch.Generator()
    g.manual_seed(seed)
    return (torch.randn(*shape, generator=g) * scale).to(dtype)


def _units(t):
    """[L,B,T,H,w] -> fp64 [L*B*H, T, w] in (l, b, h) order."""
    L, B, T, H, w = t.shape
    return t.permute(0, 1, 3, 2, 4).reshape(L * B * H, T, w).to(torch.float64).numpy()


SUFFIX = {
    # (L, B, T, H, dq, dv, dtype)
    "64x64-bf16": (1, 2, 300, 2, 64, 64, torch.bfloat16),
    "96x40-f32-ragged": (1, 1, 257, 1, 96, 40, torch.float32),
    "17x33-f32-odd": (2, 1, 65, 3, 17, 33, torch.float32),
    "128x64-bf16": (1, 1, 200, 2, 128, 64, torch.bfloat16),
    "8x8-f32-one-token": (1, 1, 1, 1, 8, 8, torch.float32),
}


@pytest.mark.parametrize("case", sorted(SUFFIX))
def test_suffix_scan_matches_oracle(case):
    L, B, T, H, dq, dv, dt = SUFFIX[case]
    q = _rand((L, B, T, H, dq), 1, dt, 1 / np.sqrt(dq))
    k = _rand((L, B, T, H, dq), 2, dt, 1 / np.sqrt(dq))
    v = _rand((L, B, T, H, dv), 3, dt)
    r = gl.suffix_scan(q.cuda(), k.cuda(), v.cuda())
    torch.cuda.synchronize()
    ref = oracle.suffix_scan(_units(q), _units(k), _units(v))
    out = _units(r.cpu())
    tol = TOL["bf16"] if dt == torch.bfloat16 else TOL["f32"]
    if T == 1:
        assert np.abs(out).max() == 0.0
    else:
        assert rel_l2(out, ref) <= tol, f"rel-L2 {rel_l2(out, ref):.3e}"
        assert np.abs(out[:, -1]).max() == 0.0  # nothing comes after the last token


@pytest.mark.parametrize("dt", [torch.float32, torch.bfloat16], ids=["f32", "bf16"])
@pytest.mark.parametrize("read", ["forward", "costate"])
def test_eta_grad_matches_oracle(read, dt):
    L, B, T, H, d, m = 1, 2, 333, 2, 64, 48
    x = _rand((L, B, T, H, d), 11, dt, 1 / np.sqrt(d))
    gh = _rand((L, B, T, H, m), 12, dt, 0.1)
    go = _rand((L, B, T, H, m), 13, dt, 0.1)
    up = _rand((L, B, T, H, m if read == "forward" else d), 14, dt)
    deta = gl.eta_grad(x.cuda(), gh.cuda(), up.cuda(), read=read,
                       g_out=go.cuda() if read == "costate" else None)
    torch.cuda.synchronize()
    xu, gu, gou, uu = _units(x), _units(gh), _units(go), _units(up)
    if read == "forward":
        ref = -np.sum(gu * oracle.suffix_scan(xu, xu, uu), axis=2)
    else:
        ref = -np.sum(xu * oracle.suffix_scan(gu, gou, uu), axis=2)
    out = deta.permute(0, 1, 3, 2).reshape(L * B * H, T).double().cpu().numpy()
    tol = TOL["bf16"] if dt == torch.bfloat16 else TOL["f32"]
    assert rel_l2(out, ref) <= tol, f"rel-L2 {rel_l2(out, ref):.3e}"
