"""Seeded synthetic inputs for the GradLev scan workloads.

This module only draws random tensors with the shapes and distributions of
the five scan workloads (and reduced-size variants for tests).  It holds none
of the method's arithmetic, imports neither the oracle nor the CUDA library,
and is the one piece both sides share: the same tensors are fed to the CUDA
path and, upcast to fp64, to the oracle.

Layouts (all row-major, last dimension contiguous):
  linear workloads: x [L,B,T,H,d_in], g_hat/g_out [L,B,T,H,d_out],
                    W0 [L,H,d_out,d_in] fp32 (one slow matrix per layer and head)
  MLP workload:     x [B,T,d], g_hat_z [B,T,m], g_hat_y/g_out [B,T,k],
                    W1 [m,d], W2 [k,m] fp32

Every tensor gets its own generator seeded from (workload seed, tensor index),
so a tensor's values do not depend on the sizes of the others.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional

import torch

__all__ = ["LinearWorkload", "MLPWorkload", "WORKLOADS", "make_linear", "make_mlp", "workload"]

BASE_SEED = 20260917


@dataclasses.dataclass(frozen=True)
class LinearWorkload:
    name: str
    L: int
    B: int
    T: int
    H: int
    d_in: int
    d_out: int
    dtype: str            # "f32" or "bf16": dtype of x, g_hat, g_out and outputs
    eta: float
    x_dist: str           # "normal" (std x_std), "layernorm" (rows of H*d_in), "unitnorm" (per head)
    x_std: float
    g_dist: str           # "normal" or "student_t4" (scaled to std g_std)
    g_std: float
    w_std: float          # W0 ~ N(0, w_std^2)
    seed: int

    @property
    def units(self) -> int:
        return self.L * self.B * self.H

    @property
    def tokens(self) -> int:
        """Tokens per call counted over all heads and layers: L*B*T."""
        return self.L * self.B * self.T

    def resized(self, **kw) -> "LinearWorkload":
        return dataclasses.replace(self, **kw)


@dataclasses.dataclass(frozen=True)
class MLPWorkload:
    name: str
    B: int
    T: int
    d: int                # input width
    m: int                # hidden width
    k: int                # output width
    dtype: str
    eta1: float
    eta2: float
    act: str              # "gelu_tanh"
    g_std: float
    seed: int

    @property
    def tokens(self) -> int:
        return self.B * self.T

    def resized(self, **kw) -> "MLPWorkload":
        return dataclasses.replace(self, **kw)


# The five workloads: sizes, dtypes, step sizes and input distributions.
WORKLOADS = {
    "c1": LinearWorkload("linear-B1-T256-64x64-fp32", L=1, B=1, T=256, H=1, d_in=64, d_out=64,
                         dtype="f32", eta=0.1, x_dist="normal", x_std=1 / 8, g_dist="normal",
                         g_std=1.0, w_std=1 / 8, seed=BASE_SEED + 0),
    "c2": LinearWorkload("multihead-B4-H8-T2048-128x128-bf16", L=1, B=4, T=2048, H=8, d_in=128,
                         d_out=128, dtype="bf16", eta=0.05, x_dist="layernorm", x_std=1.0,
                         g_dist="normal", g_std=0.02, w_std=1 / math.sqrt(128),
                         seed=BASE_SEED + 1),
    "c3": MLPWorkload("mlp-B4-T4096-512x2048x512-gelu-bf16", B=4, T=4096, d=512, m=2048, k=512,
                      dtype="bf16", eta1=0.01, eta2=0.01, act="gelu_tanh", g_std=0.02,
                      seed=BASE_SEED + 2),
    # The paper's adapted final MLP at its training context (not one of the five
    # scan workloads; used by tests and bench --workload paper_mlp).
    "paper_mlp": MLPWorkload("final-mlp-B2-T1024-1024x4096x1024-gelu-bf16", B=2, T=1024, d=1024,
                             m=4096, k=1024, dtype="bf16", eta1=0.01, eta2=0.01, act="gelu_tanh",
                             g_std=0.02, seed=BASE_SEED + 7),
    "c4": LinearWorkload("longctx-B2-H16-T32768-64x64-bf16", L=1, B=2, T=32768, H=16, d_in=64,
                         d_out=64, dtype="bf16", eta=0.02, x_dist="unitnorm", x_std=1.0,
                         g_dist="student_t4", g_std=0.02, w_std=1 / 8, seed=BASE_SEED + 3),
    "c5": LinearWorkload("layersweep-L12-B8-H12-T8192-64x64-bf16", L=12, B=8, T=8192, H=12,
                         d_in=64, d_out=64, dtype="bf16", eta=0.01, x_dist="layernorm",
                         x_std=1.0, g_dist="normal", g_std=0.02, w_std=1 / 8,
                         seed=BASE_SEED + 4),
}


def workload(key: str):
    return WORKLOADS[key]


def _gen(device, seed: int, idx: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed * 1000 + idx)
    return g


def _torch_dtype(name: str) -> torch.dtype:
    return {"f32": torch.float32, "bf16": torch.bfloat16}[name]


def _randn(shape, gen, device):
    return torch.randn(shape, generator=gen, device=device, dtype=torch.float32)


def _layernorm_rows(v: torch.Tensor, width: int) -> torch.Tensor:
    """No-affine layer norm (eps 1e-5, biased variance) over rows of `width`."""
    shp = v.shape
    r = v.reshape(-1, width)
    mu = r.mean(dim=1, keepdim=True)
    var = r.var(dim=1, unbiased=False, keepdim=True)
    return ((r - mu) / torch.sqrt(var + 1e-5)).reshape(shp)


def _draw_g(shape, dist, std, gen, device):
    if dist == "normal":
        return _randn(shape, gen, device) * std
    if dist == "student_t4":
        # t_4 = Z / sqrt(chi2_4 / 4), chi2_4 a sum of four squared normals;
        # Var(t_4) = 2, so scale by std / sqrt(2).
        z = _randn(shape, gen, device)
        chi = torch.zeros(shape, device=device, dtype=torch.float32)
        for _ in range(4):
            chi += _randn(shape, gen, device) ** 2
        return z / torch.sqrt(chi / 4.0) * (std / math.sqrt(2.0))
    raise ValueError(dist)


def make_linear(wl: LinearWorkload, device="cpu", with_gout: bool = True):
    """Inputs of a linear-map workload on `device`.

    Returns dict(x, g_hat, g_out, W0, eta) with the layouts of the module doc.
    """
    dev = torch.device(device)
    L, B, T, H, d, m = wl.L, wl.B, wl.T, wl.H, wl.d_in, wl.d_out
    dt = _torch_dtype(wl.dtype)
    W0 = _randn((L, H, m, d), _gen(dev, wl.seed, 0), dev) * wl.w_std
    x = _randn((L, B, T, H, d), _gen(dev, wl.seed, 1), dev)
    if wl.x_dist == "normal":
        x = x * wl.x_std
    elif wl.x_dist == "layernorm":
        x = _layernorm_rows(x, H * d)
    elif wl.x_dist == "unitnorm":
        x = x / torch.linalg.vector_norm(x, dim=-1, keepdim=True)
    else:
        raise ValueError(wl.x_dist)
    x = x.to(dt)
    g_hat = _draw_g((L, B, T, H, m), wl.g_dist, wl.g_std, _gen(dev, wl.seed, 2), dev).to(dt)
    g_out = None
    if with_gout:
        g_out = _draw_g((L, B, T, H, m), wl.g_dist, wl.g_std, _gen(dev, wl.seed, 3), dev).to(dt)
    return {"x": x, "g_hat": g_hat, "g_out": g_out, "W0": W0, "eta": wl.eta}


def make_mlp(wl: MLPWorkload, device="cpu"):
    """Inputs of the two-layer MLP workload on `device`.

    Returns dict(x, g_hat_z, g_hat_y, g_out, W1, W2, eta1, eta2).  W1 and W2 are
    Xavier-normal: std sqrt(2 / (fan_in + fan_out)).
    """
    dev = torch.device(device)
    B, T, d, m, k = wl.B, wl.T, wl.d, wl.m, wl.k
    dt = _torch_dtype(wl.dtype)
    W1 = _randn((m, d), _gen(dev, wl.seed, 0), dev) * math.sqrt(2.0 / (m + d))
    W2 = _randn((k, m), _gen(dev, wl.seed, 1), dev) * math.sqrt(2.0 / (k + m))
    x = _layernorm_rows(_randn((B, T, d), _gen(dev, wl.seed, 2), dev), d).to(dt)
    ghz = (_randn((B, T, m), _gen(dev, wl.seed, 3), dev) * wl.g_std).to(dt)
    ghy = (_randn((B, T, k), _gen(dev, wl.seed, 4), dev) * wl.g_std).to(dt)
    gout = (_randn((B, T, k), _gen(dev, wl.seed, 5), dev) * wl.g_std).to(dt)
    return {"x": x, "g_hat_z": ghz, "g_hat_y": ghy, "g_out": gout, "W1": W1, "W2": W2,
            "eta1": wl.eta1, "eta2": wl.eta2}


def unit_view(t: torch.Tensor, l: int, b: int, h: int) -> torch.Tensor:
    """The [T, width] slice of one (layer, batch, head) unit of an [L,B,T,H,w] tensor."""
    return t[l, b, :, h, :]


def units_fp64(t: torch.Tensor, units) -> "numpy.ndarray":
    """Stack the given (l, b, h) units of an [L,B,T,H,w] tensor as fp64 [U, T, w]."""
    import numpy as np
    return np.stack([t[l, b, :, h, :].to(torch.float64).cpu().numpy() for (l, b, h) in units])


def w0_fp64(W0: torch.Tensor, units) -> "numpy.ndarray":
    """W0 [L,H,m,d] for the given (l, b, h) units as fp64 [U, m, d]."""
    import numpy as np
    return np.stack([W0[l, h].to(torch.float64).cpu().numpy() for (l, b, h) in units])
