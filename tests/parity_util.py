"""Helpers shared by the GPU parity tests: run the CUDA scans and the fp64
oracle on the same seeded tensors and compare them.

Every comparison takes outputs laid out unit-major, [U, T, w] (or [U, T] for one
number per token), and asserts three things against the oracle:

1. the relative L2 error over the whole output is within TOL;
2. the relative L2 error of every unit (one (layer, batch, head) sequence) is
   within TOL, so a unit that nobody samples cannot hide in the norm of the rest;
3. every token row is within ROW_TOL, measured against the larger of that row's
   own norm and the unit's RMS row norm (ROW_FLOOR x RMS).  A row that the kernel
   got wrong (stale, zero, another token's) is off by about its own norm, an
   error near 1, while the rounding of bf16 operands and outputs leaves about
   2^-8 of the row.  The floor keeps rows that happen to be near zero from
   turning rounding into a large relative error.
"""
from __future__ import annotations

import numpy as np
import torch

import oracle
import workloads as W

# Tolerances on relative L2 error against the fp64 oracle.  fp32 inputs use
# fp32 FMA throughout; bf16 inputs run bf16 products with fp32 accumulation and
# bf16 outputs.
TOL = {"f32": 1e-5, "bf16": 2e-2}
# Per token row: the same bounds.  One bf16 rounding of the state (or of the
# masked score) and one of the output leave about 4e-3 of a row's norm.
ROW_TOL = {"f32": 1e-5, "bf16": 2e-2}
# Rows are measured against max(||ref_t||, ROW_FLOOR * RMS row norm of the unit).
ROW_FLOOR = 1.0


def rel_l2(out: np.ndarray, ref: np.ndarray) -> float:
    out = np.asarray(out, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    den = np.linalg.norm(ref)
    num = np.linalg.norm(out - ref)
    return float(num / den) if den > 0 else float(num)


class Parity:
    """Accumulates one output's comparison over batches of units, then asserts.

    add(out, ref) takes [U, T, w] or [U, T] arrays (any dtype; compared in fp64).
    check() asserts the whole-output, per-unit and per-row bounds and returns the
    worst figures, for messages and logs.
    """

    def __init__(self, name: str, key: str = "bf16", tol: float | None = None,
                 row_tol: float | None = None):
        self.name = name
        self.tol = TOL[key] if tol is None else tol
        self.row_tol = ROW_TOL[key] if row_tol is None else row_tol
        self.num2 = 0.0
        self.den2 = 0.0
        self.units = 0
        self.worst_unit = (0.0, -1)
        self.worst_row = (0.0, -1, -1)

    def add(self, out, ref) -> "Parity":
        out = np.asarray(out, dtype=np.float64)
        ref = np.asarray(ref, dtype=np.float64)
        assert out.shape == ref.shape, f"{self.name}: shape {out.shape} vs {ref.shape}"
        if out.ndim == 2:
            out, ref = out[..., None], ref[..., None]
        assert out.ndim == 3, f"{self.name}: expected [U, T, w], got {out.shape}"
        assert np.isfinite(out).all(), f"{self.name}: non-finite output"
        diff = out - ref
        e_row = np.sqrt(np.sum(diff * diff, axis=2))            # [U, T]
        r_row = np.sqrt(np.sum(ref * ref, axis=2))
        u_num = np.sqrt(np.sum(e_row ** 2, axis=1))              # [U]
        u_den = np.sqrt(np.sum(r_row ** 2, axis=1))
        self.num2 += float(np.sum(u_num ** 2))
        self.den2 += float(np.sum(u_den ** 2))
        T = out.shape[1]
        if T > 0:
            u_err = np.where(u_den > 0, u_num / np.where(u_den > 0, u_den, 1.0), u_num)
            i = int(np.argmax(u_err))
            if u_err[i] >= self.worst_unit[0]:
                self.worst_unit = (float(u_err[i]), self.units + i)
            rms = u_den / np.sqrt(T)
            scale = np.maximum(r_row, ROW_FLOOR * rms[:, None])
            row = np.where(scale > 0, e_row / np.where(scale > 0, scale, 1.0), e_row)
            u, t = np.unravel_index(int(np.argmax(row)), row.shape)
            if row[u, t] >= self.worst_row[0]:
                self.worst_row = (float(row[u, t]), self.units + int(u), int(t))
        self.units += out.shape[0]
        return self

    def whole(self) -> float:
        num, den = np.sqrt(self.num2), np.sqrt(self.den2)
        return float(num / den) if den > 0 else float(num)

    def check(self) -> dict:
        err = self.whole()
        ue, ui = self.worst_unit
        re, ru, rt = self.worst_row
        msg = (f"{self.name}: rel-L2 {err:.3e}, worst unit {ui} {ue:.3e}, "
               f"worst row (unit {ru}, token {rt}) {re:.3e} over {self.units} units")
        assert err <= self.tol, f"{msg}; whole-output bound {self.tol:.1e}"
        assert ue <= self.tol, f"{msg}; per-unit bound {self.tol:.1e}"
        assert re <= self.row_tol, f"{msg}; per-row bound {self.row_tol:.1e}"
        return {"rel_l2": err, "worst_unit": ue, "worst_row": re, "units": self.units}


def assert_parity(name, out, ref, key: str = "bf16", tol=None, row_tol=None) -> dict:
    """One-shot Parity: out and ref [U, T, w] or [U, T]."""
    return Parity(name, key, tol, row_tol).add(out, ref).check()


def lbthw_units(a) -> np.ndarray:
    """[L,B,T,H,w] (torch or numpy) -> fp64 [L*B*H, T, w] in (l, b, h) order;
    [L,B,T,H] -> [L*B*H, T]."""
    if isinstance(a, torch.Tensor):
        a = a.detach()
        if a.dim() == 5:
            L, B, T, H, w = a.shape
            return a.permute(0, 1, 3, 2, 4).reshape(L * B * H, T, w).to(torch.float64).cpu().numpy()
        L, B, T, H = a.shape
        return a.permute(0, 1, 3, 2).reshape(L * B * H, T).to(torch.float64).cpu().numpy()
    a = np.asarray(a, dtype=np.float64)
    if a.ndim == 5:
        L, B, T, H, w = a.shape
        return np.ascontiguousarray(a.transpose(0, 1, 3, 2, 4).reshape(L * B * H, T, w))
    L, B, T, H = a.shape
    return np.ascontiguousarray(a.transpose(0, 1, 3, 2).reshape(L * B * H, T))


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


def check_all_units_by_layer(name, wl, inputs, eta, y=None, gin=None) -> dict:
    """Every unit of a linear workload (inputs possibly on the device), one layer
    at a time so that host memory stays bounded: the forward output y and/or the
    costate output gin, each [L,B,T,H,w], against the oracle."""
    key = "f32" if wl.dtype == "f32" else "bf16"
    py = Parity(f"{name} forward", key) if y is not None else None
    pg = Parity(f"{name} costate", key) if gin is not None else None
    for l in range(wl.L):
        sl = lambda t: t[l:l + 1]
        x = lbthw_units(sl(inputs["x"]))
        g = lbthw_units(sl(inputs["g_hat"]))
        w0 = np.repeat(inputs["W0"][l].to(torch.float64).cpu().numpy()[None], wl.B, axis=0)
        w0 = np.ascontiguousarray(w0.reshape(wl.B * wl.H, wl.d_out, wl.d_in))
        go = lbthw_units(sl(inputs["g_out"])) if gin is not None else None
        yr, gr = oracle.linear_scan(x, g, w0, eta, gout=go, want_y=y is not None)
        if py is not None:
            py.add(lbthw_units(sl(y)), yr)
        if pg is not None:
            pg.add(lbthw_units(sl(gin)), gr)
    out = {}
    if py is not None:
        out["forward"] = py.check()
    if pg is not None:
        out["costate"] = pg.check()
    return out


def to_device(inputs, device="cuda"):
    return {k: (v.to(device) if isinstance(v, torch.Tensor) else v) for k, v in inputs.items()}
