"""The seeded input generators: shapes, dtypes, distributions, determinism."""
import math

import pytest
import torch

import workloads as W


def test_linear_shapes_and_dtypes():
    wl = W.workload("c5").resized(L=2, B=1, T=64, H=3)
    t = W.make_linear(wl)
    assert t["x"].shape == (2, 1, 64, 3, 64) and t["x"].dtype == torch.bfloat16
    assert t["g_hat"].shape == (2, 1, 64, 3, 64) and t["g_out"].shape == t["g_hat"].shape
    assert t["W0"].shape == (2, 3, 64, 64) and t["W0"].dtype == torch.float32
    c1 = W.make_linear(W.workload("c1"))
    assert c1["x"].dtype == torch.float32


def test_deterministic():
    wl = W.workload("c4").resized(T=100)
    a, b = W.make_linear(wl), W.make_linear(wl)
    for k in ("x", "g_hat", "g_out", "W0"):
        assert torch.equal(a[k], b[k])


def test_layernorm_rows():
    wl = W.workload("c2").resized(B=2, T=32)
    x = W.make_linear(wl)["x"].float().reshape(-1, wl.H * wl.d_in)
    assert x.mean(dim=1).abs().max() < 0.02
    assert (x.var(dim=1, unbiased=False) - 1).abs().max() < 0.02


def test_unitnorm_and_student_t():
    wl = W.workload("c4").resized(B=1, H=4, T=4096)
    t = W.make_linear(wl)
    n = torch.linalg.vector_norm(t["x"].float(), dim=-1)
    assert (n - 1).abs().max() < 1e-2
    g = t["g_hat"].float()
    assert abs(g.std().item() - 0.02) < 0.002
    # heavy tails: kurtosis of t_4 is infinite; sample excess kurtosis is well above 0
    k = ((g - g.mean()) ** 4).mean() / g.var() ** 2 - 3
    assert k > 1.0


def test_mlp_shapes():
    wl = W.workload("c3").resized(B=1, T=16)
    t = W.make_mlp(wl)
    assert t["x"].shape == (1, 16, 512) and t["g_hat_z"].shape == (1, 16, 2048)
    assert t["g_hat_y"].shape == (1, 16, 512) and t["g_out"].shape == (1, 16, 512)
    assert t["W1"].shape == (2048, 512) and t["W2"].shape == (512, 2048)
    assert abs(t["W1"].std().item() - math.sqrt(2 / 2560)) < 1e-3


def test_bench_gate_recipe():
    """The gated bench modes' synthetic gates: eta_t in [0, 2 eta], alpha_t in
    [0.9, 1], document starts with every document 512 to 1535 tokens long (the last
    one cut by T), the same on every call."""
    import bench
    wl = W.workload("c5").resized(L=2, B=3, H=2, T=5000)
    g = bench.make_gates(wl, "alpha", "cpu")
    assert g["eta_t"].shape == (2, 3, 5000, 2) and g["alpha_t"].shape == (2, 3, 5000, 2)
    assert float(g["eta_t"].min()) >= 0 and float(g["eta_t"].max()) <= 2 * wl.eta
    assert float(g["alpha_t"].min()) >= 0.9 and float(g["alpha_t"].max()) <= 1.0
    d = bench.make_gates(wl, "docs", "cpu")["doc_start"]
    assert d.shape == (3, 5000) and d.dtype == torch.uint8
    for b in range(3):
        starts = [0] + torch.nonzero(d[b]).flatten().tolist()
        assert d[b, 0] == 0 and len(starts) >= 4
        lengths = [b2 - a for a, b2 in zip(starts[:-1], starts[1:])]
        assert all(512 <= n <= 1535 for n in lengths)
    assert torch.equal(d, bench.make_gates(wl, "docs", "cpu")["doc_start"])
    assert bench.make_gates(wl, None, "cpu") == {}
