"""GPU parity of the anti-causal suffix read and the step-size gradients built on
it (outer gradients through the reads, writes detached) against the fp64 oracle.
The oracle's suffix read is pinned to finite differences of the sequential
learner in every eta_t (tests/test_oracle_pins.py)."""
import numpy as np
import pytest
import torch

import oracle
from parity_util import TOL, assert_parity

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
    # tensor-core reverse kernel (bf16, 64-wide q and k)
    "64x128-bf16-tc": (1, 1, 1024, 2, 64, 128, torch.bfloat16),
    "64x64-bf16-tc-segmented-ragged-start": (1, 1, 3000, 2, 64, 64, torch.bfloat16),
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
    key = "bf16" if dt == torch.bfloat16 else "f32"
    if T == 1:
        assert np.abs(out).max() == 0.0
    else:
        assert_parity(case, out, ref, key)
        assert np.abs(out[:, -1]).max() == 0.0  # nothing comes after the last token


def test_suffix_scan_shared_q_and_k():
    """q and k one tensor (the forward read's case): one tile per chunk."""
    L, B, T, H = 1, 2, 700, 1
    x = _rand((L, B, T, H, 64), 5, torch.bfloat16, 1 / 8)
    v = _rand((L, B, T, H, 64), 6, torch.bfloat16)
    xd = x.cuda()
    r = gl.suffix_scan(xd, xd, v.cuda())
    torch.cuda.synchronize()
    ref = oracle.suffix_scan(_units(x), _units(x), _units(v))
    assert_parity("shared q and k", _units(r.cpu()), ref, "bf16")


@pytest.mark.parametrize("m", [48, 64], ids=["cuda-core", "tensor-core"])
@pytest.mark.parametrize("dt", [torch.float32, torch.bfloat16], ids=["f32", "bf16"])
@pytest.mark.parametrize("read", ["forward", "costate"])
def test_eta_grad_matches_oracle(read, dt, m):
    L, B, T, H, d = 1, 2, 333, 2, 64
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
    assert_parity(f"eta grad {read}", out, ref, "bf16" if dt == torch.bfloat16 else "f32")


def test_eta_grad_long_context_every_unit():
    """The long-context workload at full size (B2 H16 T32768, 64 x 64): the
    segmented tensor-core reverse kernel; every unit checked against the oracle,
    per unit and per token."""
    import workloads as W
    wl = W.workload("c4")
    inp = W.make_linear(wl, device="cuda")
    u = _rand((wl.L, wl.B, wl.T, wl.H, wl.d_out), 21, torch.bfloat16).cuda()
    deta = gl.eta_grad(inp["x"], inp["g_hat"], u)
    torch.cuda.synchronize()
    xu, gu, uu = _units(inp["x"].cpu()), _units(inp["g_hat"].cpu()), _units(u.cpu())
    ref = -np.sum(gu * oracle.suffix_scan(xu, xu, uu), axis=2)
    out = deta.permute(0, 1, 3, 2).reshape(wl.units, wl.T).double().cpu().numpy()
    assert_parity("c4 eta grad", out, ref, "bf16")


def test_suffix_scan_and_eta_grad_strided_views():
    """Token tensors that are feature slices of wider buffers (non-default token
    strides) on the tensor-core reverse kernel."""
    L, B, T, H = 1, 2, 640, 2
    big = _rand((L, B, T, H, 192), 31, torch.bfloat16, 1 / 8).cuda()
    q, k, v = big[..., :64], big[..., 64:128], big[..., 128:]
    r = gl.suffix_scan(q, k, v)
    torch.cuda.synchronize()
    ref = oracle.suffix_scan(_units(q.cpu()), _units(k.cpu()), _units(v.cpu()))
    assert_parity("strided suffix", _units(r.cpu()), ref, "bf16")
    # eta gradient of the forward read with x, ghat and u all strided views
    x, gh, u = big[..., :64], big[..., 64:128] * 1, big[..., 128:]
    deta = gl.eta_grad(x, big[..., 64:128], u)
    torch.cuda.synchronize()
    xu, gu, uu = _units(x.cpu()), _units(gh.cpu()), _units(u.cpu())
    want = -np.sum(gu * oracle.suffix_scan(xu, xu, uu), axis=2)
    got = deta.permute(0, 1, 3, 2).reshape(L * B * H, T).double().cpu().numpy()
    assert_parity("strided eta grad", got, want, "bf16")


def test_empty_sequences():
    """T = 0: nothing to read, no error."""
    x = torch.zeros((1, 2, 0, 2, 64), dtype=torch.bfloat16, device="cuda")
    g = torch.zeros((1, 2, 0, 2, 64), dtype=torch.bfloat16, device="cuda")
    r = gl.suffix_scan(x, x, g)
    deta = gl.eta_grad(x, g, g)
    deta_c = gl.eta_grad(x, g, x, read="costate", g_out=g)
    torch.cuda.synchronize()
    assert r.shape == g.shape and deta.shape == (1, 2, 0, 2) and deta_c.shape == (1, 2, 0, 2)
