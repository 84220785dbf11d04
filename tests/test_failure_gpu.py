"""Failure detection without a GPU fault.

Every device-side wait in the scan kernels is bounded; when one expires the
kernel records an error bit in the workspace status word and returns, so the
context stays usable and the host reports GRADLEV_ERR_TIMEOUT.  The fault is
injected from the host: a test-only setting makes one segment never publish
its look-back flag (a flag nothing sets) and shortens the bound, so its
successor's wait runs out.
"""
import numpy as np
import pytest
import torch

import workloads as W
from parity_util import TOL, all_units, gpu_units, oracle_linear, rel_l2, to_device

gl = pytest.importorskip("paper_2609_34174_gb300")

pytestmark = pytest.mark.gpu

GRADLEV_ERR_TIMEOUT = -4


def test_lookback_timeout_is_reported_and_context_survives(monkeypatch):
    wl = W.workload("c4").resized(B=1, H=2, T=3000)  # several segments with look-back
    inputs = W.make_linear(wl)
    dev = to_device(inputs)
    ws = torch.empty(gl.workspace_bytes(wl.L, wl.B, wl.T, wl.H, wl.d_in, wl.d_out),
                     dtype=torch.uint8, device="cuda")

    # segment 0 of the first (unit, tile) pair never publishes; its successor waits 50 ms
    monkeypatch.setenv("GRADLEV_TEST_SKIP_PUBLISH", "0")
    monkeypatch.setenv("GRADLEV_TEST_LOOKBACK_LIMIT_MS", "50")
    gl.forward_scan(dev["x"], dev["g_hat"], dev["W0"], wl.eta, workspace=ws)
    assert gl.workspace_status(ws) == GRADLEV_ERR_TIMEOUT

    # the context is intact: the next call is correct and reports OK
    monkeypatch.delenv("GRADLEV_TEST_SKIP_PUBLISH")
    monkeypatch.delenv("GRADLEV_TEST_LOOKBACK_LIMIT_MS")
    y = gl.forward_scan(dev["x"], dev["g_hat"], dev["W0"], wl.eta, workspace=ws)
    assert gl.workspace_status(ws) == 0
    units = all_units(wl)
    yr, _ = oracle_linear(inputs, units, wl.eta, costate=False)
    err = rel_l2(gpu_units(y, units), yr)
    assert err <= TOL["bf16"], f"after recovery: rel-L2 {err:.3e}"
