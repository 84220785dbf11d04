"""Determinism: every result the library writes is reproducible bit for bit
(no float atomics on outputs, fixed reduction orders), including the segmented
look-back, the wide-layer passes and the reverse (suffix) read."""
import pytest
import torch

import workloads as W

gl = pytest.importorskip("paper_2609_34174_gb300")

pytestmark = pytest.mark.gpu


def _twice(fn):
    a = fn().clone()
    b = fn().clone()
    torch.cuda.synchronize()
    return a, b


@pytest.mark.parametrize("wl_key,resize", [
    ("c5", dict(L=1, B=2)),                    # one segment per unit
    ("c4", dict(B=1, H=4, T=6000)),            # segmented: decoupled look-back
    ("c2", dict(B=1, T=3000)),                 # 128-wide heads, segmented
    ("c2", dict(B=1, T=900, H=2, d_in=512, d_out=256, w_std=1 / 22.6)),  # wide-layer passes
])
def test_scans_are_bitwise_reproducible(wl_key, resize):
    wl = W.workload(wl_key).resized(**resize)
    d = {k: (v.cuda() if isinstance(v, torch.Tensor) else v) for k, v in W.make_linear(wl).items()}
    y = _twice(lambda: gl.forward_scan(d["x"], d["g_hat"], d["W0"], wl.eta))
    g = _twice(lambda: gl.costate_scan(d["x"], d["g_hat"], d["W0"], wl.eta, d["g_out"]))
    assert torch.equal(*y)
    assert torch.equal(*g)


def test_suffix_read_and_eta_grad_are_bitwise_reproducible():
    wl = W.workload("c4").resized(B=1, H=2, T=5000)
    d = {k: (v.cuda() if isinstance(v, torch.Tensor) else v) for k, v in W.make_linear(wl).items()}
    r = _twice(lambda: gl.suffix_scan(d["x"], d["x"], d["g_hat"]))
    e = _twice(lambda: gl.eta_grad(d["x"], d["g_hat"], d["g_out"]))
    assert torch.equal(*r)
    assert torch.equal(*e)
