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


def test_reference_arm_prints_one_contract_line():
    """bench.py --impl reference (the oracle timed on the host cores) prints
    one JSON line with the base contract's keys, the reference-arm markers and
    a zero-copy e2e object, and exits 0 without a GPU."""
    import json
    import subprocess
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--steps", "1", "--warmup", "3"],
                       cwd=ROOT, stdout=subprocess.PIPE, stderr=subprocess.PIPE, text=True,
                       timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.strip().startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference"
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
                "higher_is_better", "config", "cpu_baseline", "e2e"):
        assert key in d, key
    assert d["steps"] == 1 and d["warmup"] == 3 and d["n_gpus"] == 1
    assert d["higher_is_better"] is True and d["value"] > 0
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["value"] == d["value"]
    assert d["cpu_baseline"]["cores"] >= 1
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}
    assert d["config"]["workload"].startswith("FLUX-1024")
