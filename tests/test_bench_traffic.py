"""The bench's roofline.traffic comes from a committed ncu record, and only while the
kernel sources it was taken on are unchanged (no GPU needed)."""
import json

import bench


def _record(tmp_path, digest):
    rec = {"what": "test", "kernel_source_sha1": digest,
           "entries": {"c5:fwd": {"kernel": "k", "bytes_per_launch": 123456789}}}
    p = tmp_path / "traffic.json"
    p.write_text(json.dumps(rec))
    return str(p)


def test_traffic_is_read_while_the_sources_match(tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "TRAFFIC_RECORD", _record(tmp_path, bench.kernel_source_digest()))
    assert bench.recorded_traffic("c5", "fwd") == 123456789
    assert bench.recorded_traffic("c5", "costate") is None  # no entry for it
    assert bench.recorded_traffic("c2", "fwd") is None


def test_traffic_is_dropped_once_the_sources_change(tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "TRAFFIC_RECORD", _record(tmp_path, bench.kernel_source_digest()))
    monkeypatch.setattr(bench, "kernel_source_digest", lambda: "0" * 40)
    assert bench.recorded_traffic("c5", "fwd") is None


def test_traffic_missing_record(tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "TRAFFIC_RECORD", str(tmp_path / "absent.json"))
    assert bench.recorded_traffic("c5", "fwd") is None


def test_committed_record_has_both_scans_of_the_default_workload():
    with open(bench.TRAFFIC_RECORD) as f:
        rec = json.load(f)
    for key in ("c5:fwd", "c5:costate", "c4:fwd", "c4:costate"):
        assert rec["entries"][key]["bytes_per_launch"] > 0
    assert len(rec["kernel_source_sha1"]) == 40
