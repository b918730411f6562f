"""bench.py reports the decode kernel's DRAM traffic from a committed ncu
record only while the kernel's sources still hash to the record's sha."""
import json
import os

import bench

SOURCES = ["paper_2403_09636_gb300/csrc/dmc_decode.cu", "paper_2403_09636_gb300/csrc/dmc_internal.cuh",
           "paper_2403_09636_gb300/csrc/dmc_split.cuh"]


def _tree(tmp_path, sha):
    os.makedirs(tmp_path / "profiles", exist_ok=True)
    for f in SOURCES:
        dst = tmp_path / f
        os.makedirs(dst.parent, exist_ok=True)
        dst.write_bytes(open(os.path.join(bench.ROOT, f), "rb").read())
    rec = {"source_sha": sha, "sources": SOURCES, "captured_dram_bytes": 303.0,
           "captured_algorithmic_bytes": 300.0}
    (tmp_path / "profiles" / "dmc_decode_wl.traffic.json").write_text(json.dumps(rec))


def test_committed_traffic_scales_a_current_record(tmp_path, monkeypatch):
    sha = bench.decode_source_sha(SOURCES)
    _tree(tmp_path, sha)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert abs(bench.committed_traffic("wl", SOURCES, 1000.0) - 1010.0) < 1e-9


def test_committed_traffic_ignores_a_stale_or_missing_record(tmp_path, monkeypatch):
    _tree(tmp_path, "0" * 16)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.committed_traffic("wl", SOURCES, 1000.0) is None
    assert bench.committed_traffic("other", SOURCES, 1000.0) is None
