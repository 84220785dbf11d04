"""GPU parity of the fused pass (gradlev_fused_scan): the forward and the costate
read of one map in a single call (Sec. 3, steps 2 and 3, Eqs. 3-4), with the
per-token consistency term of the training objective (Eq. 5).

Both outputs are compared with the fp64 sequential learner (one walk reads y_t and
g_in_t from the same W_t) on every unit and every token row; the consistency term
is compared with the oracle's definition applied to the oracle's g_in.
"""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from parity_util import (ROW_TOL, TOL, all_units, assert_parity, check_all_units_by_layer,
                         gpu_units, oracle_linear, to_device)

gl = pytest.importorskip("paper_2609_34174_gb300")

pytestmark = pytest.mark.gpu


def _proposal(like: torch.Tensor, seed: int) -> torch.Tensor:
    g = torch.Generator(device="cpu").manual_seed(seed)
    p = torch.randn(like.shape, generator=g, dtype=torch.float32) * float(like.float().std())
    return p.to(like.dtype)


def _check_cons(name, cons, p_units, gin_ref, key):
    """cons_t = ||p_t - gin_t||^2 / w.  The kernel forms it from its own g_in, whose
    rows are within the per-row bound eps of the oracle's.  With d = p - gin and the
    kernel's g_in = gin + delta, ||delta|| <= eps ||gin||:
        |cons' - cons| <= (2 ||d|| eps ||gin|| + eps^2 ||gin||^2) / w."""
    ref = oracle.consistency(p_units, gin_ref)                       # [U, T]
    w = gin_ref.shape[-1]
    eps = ROW_TOL[key]
    dn = np.linalg.norm(p_units - gin_ref, axis=-1)
    gn = np.linalg.norm(gin_ref, axis=-1)
    bound = (2 * dn * eps * gn + (eps * gn) ** 2) / w + 1e-30
    err = np.abs(cons - ref)
    worst = float((err / bound).max()) if err.size else 0.0
    assert np.isfinite(cons).all(), f"{name}: non-finite consistency"
    assert worst <= 1.0, f"{name}: consistency error {worst:.3f} of its bound"


def _run(wl, inputs, seed=5, cons=True):
    dev = to_device(inputs)
    p = _proposal(dev["x"], seed) if cons else None
    out = gl.fused_scan(dev["x"], dev["g_hat"], dev["W0"], wl.eta, dev["g_out"],
                        cons_proposal=p.to("cuda") if p is not None else None)
    torch.cuda.synchronize()
    units = all_units(wl)
    yr, gr = oracle_linear(inputs, units, wl.eta)
    key = "f32" if wl.dtype == "f32" else "bf16"
    assert_parity("fused forward", gpu_units(out[0], units), yr, key)
    assert_parity("fused costate", gpu_units(out[1], units), gr, key)
    if cons:
        cu = np.stack([out[2][l, b, :, h].double().cpu().numpy() for (l, b, h) in units])
        pu = W.units_fp64(p, units)
        _check_cons("fused consistency", cu, pu, gr, key)
    return out, dev


CASES = {
    # one chunk, then several chunks with a ragged tail, several units and layers
    "one_chunk": ("c5", dict(L=1, B=1, H=2, T=128)),
    "ragged": ("c5", dict(L=2, B=1, H=3, T=777)),
    # few units over a long sequence: segments with the look-back carry
    "segmented": ("c4", dict(B=1, H=2, T=3000)),
    "segmented_many": ("c4", dict(B=1, H=3, T=8192 + 5)),
}


@pytest.mark.parametrize("case", sorted(CASES))
def test_fused_tensor_core_path(case):
    key, kw = CASES[case]
    _run(W.workload(key).resized(**kw), W.make_linear(W.workload(key).resized(**kw)))


@pytest.mark.parametrize("T", [1, 2, 127, 129, 255])
def test_fused_short_sequences(T):
    wl = W.workload("c5").resized(L=1, B=1, H=2, T=T)
    _run(wl, W.make_linear(wl))


def test_fused_forward_equals_forward_scan_bit_for_bit():
    """The fused pass's forward read runs the forward scan's arithmetic: the same
    state, the same masked score, the same products."""
    wl = W.workload("c4").resized(B=1, H=2, T=3000)
    inputs = W.make_linear(wl)
    out, dev = _run(wl, inputs, cons=False)
    y = gl.forward_scan(dev["x"], dev["g_hat"], dev["W0"], wl.eta)
    torch.cuda.synchronize()
    assert torch.equal(out[0], y)


@pytest.mark.parametrize("shape", [dict(d_in=64, d_out=128), dict(d_in=128, d_out=128),
                                   dict(d_in=48, d_out=80)], ids=str)
def test_fused_other_shapes_run_both_scans(shape):
    """Shapes the single-pass kernel does not cover: the two scans back to back,
    and the consistency term from its row-reduction kernel."""
    wl = W.workload("c5").resized(L=1, B=1, H=2, T=600, **shape)
    _run(wl, W.make_linear(wl))


def test_fused_fp32():
    wl = W.workload("c1").resized(B=2, H=2, T=300)
    _run(wl, W.make_linear(wl))


def test_fused_zero_length_and_degenerate_eta():
    wl = W.workload("c5").resized(L=1, B=1, H=2, T=0)
    inputs = W.make_linear(wl)
    dev = to_device(inputs)
    y, gin = gl.fused_scan(dev["x"], dev["g_hat"], dev["W0"], wl.eta, dev["g_out"])
    assert y.numel() == 0 and gin.numel() == 0
    wl = W.workload("c4").resized(B=1, H=2, T=1500)
    inputs = W.make_linear(wl)
    dev = to_device(inputs)
    y, gin = gl.fused_scan(dev["x"], dev["g_hat"], dev["W0"], 0.0, dev["g_out"])
    torch.cuda.synchronize()
    units = all_units(wl)
    yr, gr = oracle_linear(inputs, units, 0.0)
    assert_parity("eta=0 forward", gpu_units(y, units), yr)
    assert_parity("eta=0 costate", gpu_units(gin, units), gr)


@pytest.mark.parametrize("key", ["c4", "c5"])
def test_fused_full_size_every_unit(key):
    """The workload at its full size, as the bench times it, every unit checked."""
    wl = W.workload(key)
    inputs = W.make_linear(wl, device="cuda")
    y, gin = gl.fused_scan(inputs["x"], inputs["g_hat"], inputs["W0"], wl.eta, inputs["g_out"])
    torch.cuda.synchronize()
    check_all_units_by_layer(f"{key} fused", wl, inputs, wl.eta, y=y, gin=gin)


def test_fused_consistency_vanishes_at_exact_costates():
    """Theorem 1 on the device: proposals equal to the costates the read reconstructs
    give a consistency term at the rounding level of those costates."""
    wl = W.workload("c5").resized(L=1, B=1, H=2, T=500)
    inputs = W.make_linear(wl)
    dev = to_device(inputs)
    y, gin = gl.fused_scan(dev["x"], dev["g_hat"], dev["W0"], wl.eta, dev["g_out"])
    y2, gin2, cons = gl.fused_scan(dev["x"], dev["g_hat"], dev["W0"], wl.eta, dev["g_out"],
                                   cons_proposal=gin)
    torch.cuda.synchronize()
    assert torch.equal(gin, gin2)
    # only the bf16 rounding of g_in separates the proposal from the fp32 reconstruction
    scale = (gin.float() ** 2).sum(-1) / gin.shape[-1]
    assert float((cons / (scale + 1e-30)).max()) < 2 ** -14
