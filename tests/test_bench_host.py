"""Host-side logic of bench.py (no GPU): the DRAM traffic of the spatial
kernel is reported only while profiles/ holds a capture of the current
source; any change to the kernel source turns it into null."""
import hashlib
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
SRC = os.path.join(ROOT, "paper_2608_17995_gb300", "csrc", "spatial_tc.cu")
SUMMARY = "spatial_tc_flux1024.md"


def test_traffic_read_while_the_capture_is_current():
    import bench
    text = open(os.path.join(ROOT, "profiles", SUMMARY)).read()
    sha = hashlib.sha1(open(SRC, "rb").read()).hexdigest()[:12]
    if "kernel_source_sha1: " + sha not in text:
        pytest.skip("the committed capture is of another version of the kernel")
    t = bench.profiled_traffic(SRC, SUMMARY)
    assert t is not None and t > 15.0e6


def test_traffic_null_when_source_changed(tmp_path):
    import bench
    changed = tmp_path / "spatial_tc.cu"
    changed.write_bytes(open(SRC, "rb").read() + b"\n// changed\n")
    assert bench.profiled_traffic(str(changed), SUMMARY) is None
    assert bench.profiled_traffic(SRC, "no_such_summary.md") is None
