"""The bench's reference arm (the fp64 oracle timed on the host cores) prints one
valid JSON line for each kind of step: the scans, the step-size gradients of the
reads, and deployment of the paper-shaped MLP."""
import contextlib
import io
import json
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _line(argv):
    buf = io.StringIO()
    with contextlib.redirect_stdout(buf):
        assert bench.main(argv) == 0
    lines = [ln for ln in buf.getvalue().splitlines() if ln.strip().startswith("{")]
    assert len(lines) == 1
    return json.loads(lines[0])


@pytest.mark.parametrize("extra,metric", [
    ([], bench.METRIC),
    (["--grads"], bench.GRADS_METRIC),
], ids=["scans", "grads"])
def test_reference_line_small_workload(extra, metric):
    d = _line(["--impl", "reference", "--workload", "c1", "--steps", "1", "--warmup", "3"] + extra)
    assert d["impl"] == "reference" and d["metric"] == metric
    assert d["value"] > 0 and d["unit"] == "tokens/s" and d["higher_is_better"] is True
    assert d["e2e"]["value"] == d["value"]
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["d2h_bytes_per_step"] == 0
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] >= 1


@pytest.mark.parametrize("extra,words", [
    (["--gates", "alpha"], "eta_t and alpha_t"),
    (["--gates", "docs", "--resize", "T=3000"], "one learner per document"),
], ids=["retention", "documents"])
def test_reference_line_gated(extra, words):
    """The gated modes time the oracle on the gated workload itself: each unit with
    its own gate sequences, or one learner per document."""
    d = _line(["--impl", "reference", "--workload", "c1", "--steps", "1", "--warmup", "3"] + extra)
    assert d["impl"] == "reference" and d["metric"] == bench.METRIC and d["value"] > 0
    assert words in d["cpu_baseline"]["sample"]
    assert d["config"]["gates"]


def test_reference_line_deployment():
    d = _line(["--impl", "reference", "--workload", "decode_mlp", "--steps", "1", "--warmup", "3"])
    assert d["impl"] == "reference" and d["metric"] == bench.DECODE_METRIC
    assert d["value"] > 0 and "deployed MLP" in d["cpu_baseline"]["sample"]
