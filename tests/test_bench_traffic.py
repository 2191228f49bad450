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


def test_recorded_traffic_matches_the_current_sources():
    """Every kernel's record carries the hash of the source it was captured on, and that
    is the committed source: the profiles are not stale."""
    rec = _records()
    for kernel, src in (("attn_tc2", ATTN), ("attn_tc1", ATTN), ("score_pass1", SCORE),
                        ("score_pass2", SCORE)):
        assert kernel in rec, kernel
        assert rec[kernel][0] == _digest(src), (kernel, "profiles/traffic.txt is stale")


def test_traffic_for_reports_only_for_the_measured_source():
    rec = _records()
    assert bench.traffic_for("attn_tc2", ATTN, 1.0) == rec["attn_tc2"][1]
    assert bench.traffic_for("attn_tc2", ATTN, 2.0) == 2 * rec["attn_tc2"][1]
    assert bench.traffic_for("attn_tc2", SCORE, 1.0) is None  # another file's hash
    assert bench.traffic_for("no_such_kernel", ATTN, 1.0) is None
