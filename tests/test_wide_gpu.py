"""GPU parity of the wide-layer path (state, score and output passes over
segments; dq a multiple of 128 and at least 256) against the fp64 oracle.

Covers the two-layer MLP of Appendix A at its full widths (512 -> 2048 -> 512)
with sigma fused in the layer-1 forward epilogue and sigma' in the layer-2
costate epilogue, plus plain linear scans whose forward and costate land on
different paths (wide one way, 64-wide chunk kernel or CUDA-core kernel the
other), ragged and single-segment lengths, and several units with their own W0.
"""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from parity_util import TOL, assert_parity, to_device, all_units, gpu_units, oracle_linear

gl = pytest.importorskip("paper_2609_34174_gb300")

pytestmark = pytest.mark.gpu


def _close(name, out, ref):
    """Whole-output, per-unit (per-sequence) and per-row bf16 bounds; [U, T, w]."""
    assert_parity(name, out, ref, "bf16")


LINEAR = {
    # (L, B, T, H, d_in, d_out)
    "512x2048-ragged": (1, 1, 1100, 1, 512, 2048),
    "2048x512-short": (1, 1, 700, 1, 2048, 512),
    "256x64-multi-unit": (2, 2, 1300, 2, 256, 64),
    "192x256-narrow-tiles": (1, 2, 900, 1, 192, 256),
    "256x384-single-segment": (1, 1, 384, 1, 256, 384),
    "256x256-one-token": (1, 2, 1, 1, 256, 256),
}


@pytest.mark.parametrize("case", sorted(LINEAR))
def test_wide_linear(case):
    L, B, T, H, din, dout = LINEAR[case]
    wl = W.workload("c2").resized(L=L, B=B, T=T, H=H, d_in=din, d_out=dout, seed=1000 + T,
                                  w_std=1 / np.sqrt(din))
    inputs = W.make_linear(wl)
    dev = to_device(inputs)
    y = gl.forward_scan(dev["x"], dev["g_hat"], dev["W0"], wl.eta)
    gin = gl.costate_scan(dev["x"], dev["g_hat"], dev["W0"], wl.eta, dev["g_out"])
    torch.cuda.synchronize()
    units = all_units(wl)
    yr, gr = oracle_linear(inputs, units, wl.eta)
    _close(f"{case} forward", gpu_units(y, units), yr)
    _close(f"{case} costate", gpu_units(gin, units), gr)


def _mlp_check(wl, inp, units, act="gelu_tanh"):
    code = {"gelu_tanh": oracle.ACT_GELU_TANH, "gelu_erf": oracle.ACT_GELU_ERF,
            "tanh": oracle.ACT_TANH}[act]
    dev = {k: (v.cuda() if isinstance(v, torch.Tensor) else v) for k, v in inp.items()}
    z, h, y = gl.mlp_forward(dev["x"], dev["g_hat_z"], dev["g_hat_y"], dev["W1"], dev["W2"],
                             wl.eta1, wl.eta2, act=act)
    gz, gx = gl.mlp_costate(dev["x"], h, z, dev["g_hat_z"], dev["g_hat_y"], dev["W1"], dev["W2"],
                            wl.eta1, wl.eta2, dev["g_out"], act=act)
    torch.cuda.synchronize()
    sel = lambda t: t[units].to(torch.float64).cpu().numpy()
    ref = oracle.mlp_scan(sel(inp["x"]), sel(inp["g_hat_z"]), sel(inp["g_hat_y"]),
                          inp["W1"].double().cpu().numpy(), inp["W2"].double().cpu().numpy(),
                          wl.eta1, wl.eta2, act=code, gout=sel(inp["g_out"]),
                          nthreads=len(units))
    for name, out in (("z", z), ("h", h), ("y", y), ("gz", gz), ("gx", gx)):
        _close(f"mlp {name}", sel(out), ref[name])


def test_mlp_full_widths_reduced_length():
    """512 -> 2048 -> 512, GELU-tanh, two sequences of 1100 tokens (three
    segments, the last one ragged)."""
    wl = W.workload("c3").resized(B=2, T=1100)
    _mlp_check(wl, W.make_mlp(wl), [0, 1])


@pytest.mark.parametrize("act", ["gelu_erf", "tanh"])
def test_mlp_other_activations(act):
    wl = W.workload("c3").resized(B=1, T=520, d=256, m=512, k=256, act=act)
    _mlp_check(wl, W.make_mlp(wl), [0], act=act)


def test_mlp_full_size_every_sequence():
    """The MLP workload at its full size (4 x 4096 tokens, 512 -> 2048 -> 512) in
    the launch configuration the bench times; all four sequences are checked
    against the oracle in full, per sequence and per token row."""
    wl = W.workload("c3")
    inp = W.make_mlp(wl, device="cuda")
    _mlp_check(wl, inp, [0, 1, 2, 3])


def test_paper_shaped_final_mlp():
    """The adapted final MLP at the paper's own shape: 1024 -> 4096 -> 1024 with
    GELU, T = 1024 (the training context), two sequences, checked in full."""
    wl = W.workload("c3").resized(B=2, T=1024, d=1024, m=4096, k=1024)
    _mlp_check(wl, W.make_mlp(wl), [0, 1])
