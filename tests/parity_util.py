"""Helpers shared by the GPU parity tests: run the CUDA scans and the fp64
oracle on the same seeded tensors and compare them."""
from __future__ import annotations

import numpy as np
import torch

import oracle
import workloads as W

# Tolerances on relative L2 error against the fp64 oracle.  fp32 inputs use
# fp32 FMA throughout; bf16 inputs run bf16 products with fp32 accumulation and
# bf16 outputs.
TOL = {"f32": 1e-5, "bf16": 2e-2}


def rel_l2(out: np.ndarray, ref: np.ndarray) -> float:
    out = np.asarray(out, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    den = np.linalg.norm(ref)
    num = np.linalg.norm(out - ref)
    return float(num / den) if den > 0 else float(num)


def all_units(wl):
    return [(l, b, h) for l in range(wl.L) for b in range(wl.B) for h in range(wl.H)]


def oracle_linear(inputs, units, eta, costate=True):
    """Oracle outputs for the given (l, b, h) units: (y [U,T,m], gin [U,T,d] or None)."""
    x = W.units_fp64(inputs["x"], units)
    g = W.units_fp64(inputs["g_hat"], units)
    w0 = W.w0_fp64(inputs["W0"], units)
    go = W.units_fp64(inputs["g_out"], units) if costate else None
    return oracle.linear_scan(x, g, w0, eta, gout=go)


def gpu_units(t: torch.Tensor, units) -> np.ndarray:
    return np.stack([t[l, b, :, h, :].to(torch.float64).cpu().numpy() for (l, b, h) in units])


def to_device(inputs, device="cuda"):
    return {k: (v.to(device) if isinstance(v, torch.Tensor) else v) for k, v in inputs.items()}
