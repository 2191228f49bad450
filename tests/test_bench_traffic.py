"""bench.py's roofline `traffic`: the ncu DRAM bytes recorded in profiles/traffic.txt are
reported only for the source they were measured on (CPU; no GPU needed)."""
import hashlib
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402

ATTN = "paper_2608_26574_gb300/csrc/dard_attention.cu"
SCORE = "paper_2608_26574_gb300/csrc/dard_score.cu"


def _records():
    out = {}
    for line in open(os.path.join(ROOT, "profiles", "traffic.txt")):
        parts = line.split()
        if len(parts) >= 3 and not line.startswith("#"):
            out[parts[0]] = (parts[1], float(parts[2]))
    return out


def _digest(rel):
    return hashlib.sha256(open(os.path.join(ROOT, rel), "rb").read()).hexdigest()[:16]


SOURCES = {"attn_tc1": ATTN, "attn_tc2": ATTN,
           "attn_pair": "paper_2608_26574_gb300/csrc/dard_attention_pair.cu",
           "score_pass1": SCORE, "score_pass2": SCORE, "score_fused": SCORE}


def test_recorded_traffic_matches_the_current_sources():
    """Every record carries the hash of the source it was captured on, and that is the
    committed source: a kernel whose source changed has its record removed until it is
    measured again, so no stale number stays in the file."""
    for kernel, (digest, _) in _records().items():
        assert kernel in SOURCES, kernel
        assert digest == _digest(SOURCES[kernel]), (kernel, "profiles/traffic.txt is stale")


def test_traffic_for_reports_only_for_the_measured_source(tmp_path, monkeypatch):
    """bench.traffic_for returns a record's bytes (scaled by the units of a launch) only
    while the kernel's source hash matches the record."""
    (tmp_path / "profiles").mkdir()
    (tmp_path / "paper_2608_26574_gb300" / "csrc").mkdir(parents=True)
    for rel in (ATTN, SCORE):
        (tmp_path / rel).write_bytes(open(os.path.join(ROOT, rel), "rb").read())
    (tmp_path / "profiles" / "traffic.txt").write_text(
        f"# comment line\nattn_tc2 {_digest(ATTN)} 1000\nscore_pass1 0123456789abcdef 5\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.traffic_for("attn_tc2", ATTN, 1.0) == 1000.0
    assert bench.traffic_for("attn_tc2", ATTN, 2.0) == 2000.0
    assert bench.traffic_for("attn_tc2", SCORE, 1.0) is None      # another file's hash
    assert bench.traffic_for("score_pass1", SCORE, 1.0) is None   # a stale record
    assert bench.traffic_for("no_such_kernel", ATTN, 1.0) is None
