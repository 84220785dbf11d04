"""GPU parity: the CUDA scans against the fp64 sequential-learner oracle.

Every test generates seeded inputs, runs the CUDA library through the C ABI
(via the ctypes binding) and compares element by element with the oracle run
on the same tensors upcast to fp64.  Tolerances: relative L2 <= 1e-5 for fp32
inputs and <= 2e-2 for bf16 inputs (fp32 accumulation).
"""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from parity_util import (TOL, all_units, assert_parity, check_all_units_by_layer, gpu_units,
                         oracle_linear, to_device)

gl = pytest.importorskip("paper_2609_34174_gb300")

pytestmark = pytest.mark.gpu


def _run_linear(wl, inputs, units=None, check_units=None):
    dev = to_device(inputs)
    y = gl.forward_scan(dev["x"], dev["g_hat"], dev["W0"], wl.eta)
    gin = gl.costate_scan(dev["x"], dev["g_hat"], dev["W0"], wl.eta, dev["g_out"])
    torch.cuda.synchronize()
    units = units or all_units(wl)
    yr, gr = oracle_linear(inputs, units, wl.eta)
    return gpu_units(y, units), gpu_units(gin, units), yr, gr


def _assert_close(name, out, ref, tol):
    """Whole-output, per-unit and per-row bounds (parity_util.Parity); out and
    ref [U, T, w]."""
    key = "f32" if tol == TOL["f32"] else "bf16"
    return assert_parity(name, out, ref, key)["rel_l2"]


# ---------------------------------------------------------------- fp32 path
def test_c1_fp32_full_size():
    wl = W.workload("c1")
    inputs = W.make_linear(wl)
    y, g, yr, gr = _run_linear(wl, inputs)
    _assert_close("c1 forward", y, yr, TOL["f32"])
    _assert_close("c1 costate", g, gr, TOL["f32"])


def test_fp32_ragged_many_units():
    wl = W.workload("c1").resized(B=2, H=3, T=301, d_in=48, d_out=80)
    inputs = W.make_linear(wl)
    y, g, yr, gr = _run_linear(wl, inputs)
    _assert_close("fp32 ragged forward", y, yr, TOL["f32"])
    _assert_close("fp32 ragged costate", g, gr, TOL["f32"])


# ---------------------------------------------------------- tensor-core path
REDUCED = {
    # head widths 128, one segment, ragged tail
    "c2_small": ("c2", dict(B=2, H=2, T=1000)),
    # head widths 128, several segments with look-back carry
    "c2_segmented": ("c2", dict(B=1, H=2, T=2048 + 77)),
    # 64-wide heads, several segments with look-back, unit-norm x and Student-t writes
    "c4_segmented": ("c4", dict(B=1, H=2, T=3000)),
    # 64-wide heads, independent layers, ragged tail
    "c5_small": ("c5", dict(L=2, B=1, H=3, T=777)),
}


@pytest.mark.parametrize("case", sorted(REDUCED))
def test_bf16_reduced(case):
    key, kw = REDUCED[case]
    wl = W.workload(key).resized(**kw)
    inputs = W.make_linear(wl)
    y, g, yr, gr = _run_linear(wl, inputs)
    _assert_close(f"{case} forward", y, yr, TOL["bf16"])
    _assert_close(f"{case} costate", g, gr, TOL["bf16"])


@pytest.mark.parametrize("T", [1, 2, 127, 128, 129, 255, 513])
def test_short_and_ragged_sequences(T):
    wl = W.workload("c5").resized(L=1, B=1, H=2, T=T)
    inputs = W.make_linear(wl)
    y, g, yr, gr = _run_linear(wl, inputs)
    _assert_close(f"T={T} forward", y, yr, TOL["bf16"])
    _assert_close(f"T={T} costate", g, gr, TOL["bf16"])


def test_first_token_reads_slow_weights():
    """t = 0 reads W0 only (exclusive scan): equal to a bf16-rounded W0 x_0."""
    wl = W.workload("c5").resized(L=1, B=1, H=2, T=300)
    inputs = W.make_linear(wl)
    y, g, yr, gr = _run_linear(wl, inputs)
    np.testing.assert_allclose(y[:, 0], yr[:, 0], rtol=2e-2, atol=2e-2 * np.abs(yr[:, 0]).max())


@pytest.mark.parametrize("which", ["eta0", "ghat0"])
def test_degenerate_plain_gemm(which):
    wl = W.workload("c4").resized(B=1, H=2, T=1500)
    inputs = W.make_linear(wl)
    eta = wl.eta
    if which == "eta0":
        eta = 0.0
    else:
        inputs["g_hat"] = torch.zeros_like(inputs["g_hat"])
    dev = to_device(inputs)
    y = gl.forward_scan(dev["x"], dev["g_hat"], dev["W0"], eta)
    gin = gl.costate_scan(dev["x"], dev["g_hat"], dev["W0"], eta, dev["g_out"])
    torch.cuda.synchronize()
    units = all_units(wl)
    yr, gr = oracle_linear(inputs, units, eta)
    _assert_close("degenerate forward", gpu_units(y, units), yr, TOL["bf16"])
    _assert_close("degenerate costate", gpu_units(gin, units), gr, TOL["bf16"])


@pytest.mark.parametrize("eta", [1e-40, 1e-30, -3e-25, 3e20, 0.01], ids=str)
def test_step_sizes_outside_the_scaled_state_window(eta):
    """The chunk kernel holds its state in units of -eta; step sizes whose
    reciprocal (or W0 / eta) would leave fp32 run on the CUDA-core kernel.  Every
    finite eta, a subnormal one included, matches the oracle."""
    wl = W.workload("c5").resized(L=1, B=1, H=2, T=300)
    inputs = W.make_linear(wl)
    dev = to_device(inputs)
    y = gl.forward_scan(dev["x"], dev["g_hat"], dev["W0"], eta)
    gin = gl.costate_scan(dev["x"], dev["g_hat"], dev["W0"], eta, dev["g_out"])
    torch.cuda.synchronize()
    units = all_units(wl)
    yr, gr = oracle_linear(inputs, units, eta)
    _assert_close(f"eta={eta} forward", gpu_units(y, units), yr, TOL["bf16"])
    _assert_close(f"eta={eta} costate", gpu_units(gin, units), gr, TOL["bf16"])


def test_strided_inputs_and_outputs():
    """Token tensors that are slices of wider buffers (non-default strides)."""
    wl = W.workload("c5").resized(L=1, B=2, H=2, T=400)
    inputs = W.make_linear(wl)
    dev = to_device(inputs)
    L, B, T, H, d = dev["x"].shape
    big = torch.zeros((L, B, T, H, 2 * d), dtype=torch.bfloat16, device="cuda")
    big[..., 32:32 + d] = dev["x"]
    x_view = big[..., 32:32 + d]
    assert x_view.stride(3) == 2 * d
    ybig = torch.zeros((L, B, T, H, 3 * d), dtype=torch.bfloat16, device="cuda")
    y_view = ybig[..., 64:64 + d]
    gl.forward_scan(x_view, dev["g_hat"], dev["W0"], wl.eta, y=y_view)
    gbig = torch.zeros_like(ybig)
    g_view = gbig[..., 128:128 + d]
    gl.costate_scan(x_view, dev["g_hat"], dev["W0"], wl.eta, dev["g_out"], g_in=g_view)
    torch.cuda.synchronize()
    units = all_units(wl)
    yr, gr = oracle_linear(inputs, units, wl.eta)
    _assert_close("strided forward", gpu_units(y_view, units), yr, TOL["bf16"])
    _assert_close("strided costate", gpu_units(g_view, units), gr, TOL["bf16"])
    # nothing outside the views was written
    assert ybig[..., :64].abs().max().item() == 0 and ybig[..., 128:].abs().max().item() == 0
    assert gbig[..., :128].abs().max().item() == 0


def test_deterministic_and_status_ok():
    wl = W.workload("c4").resized(B=1, H=2, T=4000)
    dev = to_device(W.make_linear(wl))
    ws = torch.empty(gl.workspace_bytes(wl.L, wl.B, wl.T, wl.H, wl.d_in, wl.d_out),
                     dtype=torch.uint8, device="cuda")
    y1 = gl.forward_scan(dev["x"], dev["g_hat"], dev["W0"], wl.eta, workspace=ws)
    assert gl.workspace_status(ws) == 0
    y2 = gl.forward_scan(dev["x"], dev["g_hat"], dev["W0"], wl.eta, workspace=ws)
    g1 = gl.costate_scan(dev["x"], dev["g_hat"], dev["W0"], wl.eta, dev["g_out"], workspace=ws)
    g2 = gl.costate_scan(dev["x"], dev["g_hat"], dev["W0"], wl.eta, dev["g_out"], workspace=ws)
    assert gl.workspace_status(ws) == 0
    assert torch.equal(y1, y2) and torch.equal(g1, g2)


def test_theorem1_recovery_on_gpu():
    """Supplying the serial learner's true costates reproduces its outputs (Theorem 1),
    within the bf16 tolerance: the serial learner here is the oracle itself driven by
    a squared loss, its costates g_t = y_t - c_t fed back as proposals."""
    wl = W.workload("c5").resized(L=1, B=1, H=2, T=600)
    inputs = W.make_linear(wl)
    units = all_units(wl)
    T, d, m = wl.T, wl.d_in, wl.d_out
    x = W.units_fp64(inputs["x"], units)
    w0 = W.w0_fp64(inputs["W0"], units)
    c = np.random.default_rng(5).standard_normal((len(units), T, m)) * 0.5
    # serial learner with l_t = 1/2 ||y_t - c_t||^2
    g = np.zeros((len(units), T, m))
    ys = np.zeros((len(units), T, m))
    for u in range(len(units)):
        Wm = w0[u].copy()
        for t in range(T):
            ys[u, t] = Wm @ x[u, t]
            g[u, t] = ys[u, t] - c[u, t]
            Wm -= wl.eta * np.outer(g[u, t], x[u, t])
    gh = torch.zeros_like(inputs["g_hat"])
    for i, (l, b, h) in enumerate(units):
        gh[l, b, :, h, :] = torch.from_numpy(g[i]).to(torch.bfloat16)
    dev = to_device(dict(inputs, g_hat=gh))
    y = gl.forward_scan(dev["x"], dev["g_hat"], dev["W0"], wl.eta)
    torch.cuda.synchronize()
    # the bf16-rounded costates differ from g by ~2^-9 relative, well inside tolerance
    _assert_close("theorem-1 recovery", gpu_units(y, units), ys, TOL["bf16"])


# ------------------------------------------------------------- activations
@pytest.mark.parametrize("act", ["gelu_tanh", "gelu_erf", "tanh"])
def test_fused_activation_small_mlp(act):
    """Appendix A MLP with widths the tensor-core path tiles (64 -> 128 -> 64):
    sigma fused in the layer-1 forward epilogue, sigma' in the layer-2 costate
    epilogue, checked against the fp64 MLP oracle."""
    code = {"gelu_tanh": oracle.ACT_GELU_TANH, "gelu_erf": oracle.ACT_GELU_ERF,
            "tanh": oracle.ACT_TANH}[act]
    wl = W.workload("c3").resized(B=2, T=700, d=64, m=128, k=64)
    inp = W.make_mlp(wl)
    dev = to_device(inp)
    z, h, y = gl.mlp_forward(dev["x"], dev["g_hat_z"], dev["g_hat_y"], dev["W1"], dev["W2"],
                             wl.eta1, wl.eta2, act=act)
    gz, gx = gl.mlp_costate(dev["x"], h, z, dev["g_hat_z"], dev["g_hat_y"], dev["W1"], dev["W2"],
                            wl.eta1, wl.eta2, dev["g_out"], act=act)
    torch.cuda.synchronize()
    f64 = lambda t: t.to(torch.float64).cpu().numpy()
    ref = oracle.mlp_scan(f64(inp["x"]), f64(inp["g_hat_z"]), f64(inp["g_hat_y"]), f64(inp["W1"]),
                          f64(inp["W2"]), wl.eta1, wl.eta2, act=code, gout=f64(inp["g_out"]))
    _assert_close("mlp z", f64(z), ref["z"], TOL["bf16"])
    _assert_close("mlp h", f64(h), ref["h"], TOL["bf16"])
    _assert_close("mlp y", f64(y), ref["y"], TOL["bf16"])
    _assert_close("mlp g_z", f64(gz), ref["gz"], TOL["bf16"])
    _assert_close("mlp g_x", f64(gx), ref["gx"], TOL["bf16"])


# ------------------------------------------------ full sizes, every unit
@pytest.mark.parametrize("key", ["c2", "c4", "c5"])
def test_full_size_every_unit(key):
    """The workload at its full size, in the launch configuration the bench times,
    with every unit checked against the oracle: whole output, each unit and each
    token row (the oracle walks the units one layer at a time)."""
    wl = W.workload(key)
    inputs = W.make_linear(wl, device="cuda")
    y = gl.forward_scan(inputs["x"], inputs["g_hat"], inputs["W0"], wl.eta)
    gin = gl.costate_scan(inputs["x"], inputs["g_hat"], inputs["W0"], wl.eta, inputs["g_out"])
    torch.cuda.synchronize()
    res = check_all_units_by_layer(key, wl, inputs, wl.eta, y=y, gin=gin)
    print(f"{key} every unit: {res}")
    assert res["forward"]["units"] == wl.units and res["costate"]["units"] == wl.units


# ------------------------------------------------ pipeline phase bookkeeping
SWEEP_T = sorted(set(list(range(1, 3 * 128 + 1, 11)) + [63, 64, 65, 127, 128, 129, 191, 192, 193,
                                                        255, 256, 257, 383, 384]))


@pytest.mark.parametrize("dq", [64, 128])
def test_length_sweep_one_to_three_chunks(dq):
    """Every sequence length in a dense sweep over 1..3 chunks (128 tokens each),
    many units per launch, so each CTA walks its stage ring, TMEM buffers and
    barrier phases through many item boundaries with partial chunks.  Each length
    is checked against the oracle."""
    for T in SWEEP_T:
        wl = W.workload("c2" if dq == 128 else "c5").resized(L=1, B=3, H=5, T=T, d_in=dq, d_out=64,
                                                            seed=300 + T)
        inputs = W.make_linear(wl)
        y, g, yr, gr = _run_linear(wl, inputs)
        _assert_close(f"T={T} forward", y, yr, TOL["bf16"])
        _assert_close(f"T={T} costate", g, gr, TOL["bf16"])


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32], ids=["bf16", "f32"])
def test_empty_sequences_every_entry_point(dtype):
    """T = 0 (the header allows it): every token entry point returns without error."""
    L, B, H, d, m = 1, 2, 2, 64, 64
    z = lambda w: torch.zeros((L, B, 0, H, w), dtype=dtype, device="cuda")
    x, g = z(d), z(m)
    W0 = torch.zeros((L, H, m, d), device="cuda")
    eta_t = torch.zeros((L, B, 0, H), device="cuda")
    y = gl.forward_scan(x, g, W0, 0.1)
    gi = gl.costate_scan(x, g, W0, 0.1, g)
    yg = gl.forward_scan(x, g, W0, eta_t, alpha=eta_t)
    gg = gl.costate_scan(x, g, W0, eta_t, g)
    r = gl.suffix_scan(x, x, g)
    de = gl.eta_grad(x, g, g)
    torch.cuda.synchronize()
    assert y.shape == g.shape and gi.shape == x.shape and yg.shape == g.shape
    assert gg.shape == x.shape and r.shape == g.shape and de.shape == (L, B, 0, H)
