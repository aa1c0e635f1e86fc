"""bench.py on the CPU: the reference arm's JSON line (the oracle timed on
the host cores) carries the contract's keys, and the recorded DRAM traffic
is taken only for the workload and kernel source it was captured on."""

import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def test_reference_arm_line():
    out = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--steps", "1", "--warmup", "3"],
                         cwd=ROOT, capture_output=True, text=True, timeout=600, check=True).stdout
    lines = [l for l in out.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    r = json.loads(lines[0])
    assert r["impl"] == "reference" and r["n_gpus"] == 1 and r["steps"] == 1 and r["warmup"] == 3
    assert r["unit"] == "verified tokens/s" and r["higher_is_better"] is True and r["value"] > 0
    assert r["metric"].startswith("verified tokens/s")
    assert r["config"]["workload"].startswith("qwen3-32b verify")
    cb = r["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == r["value"] and cb["sample"]
    assert r["e2e"] == {"value": r["value"], "unit": r["unit"], "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}


def test_recorded_traffic_follows_workload_and_source():
    with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
        rec = json.load(f)
    r2 = rec["verify_attention@workload2"]
    assert bench.recorded_traffic("verify_attention", 2, r2["source_hash"]) == r2["dram_bytes_per_launch"]
    assert r2["dram_bytes_per_launch"] == r2["read"] + r2["write"]
    assert bench.recorded_traffic("verify_attention", 2, "0" * 16) is None  # another source
    assert bench.recorded_traffic("verify_attention", 4, r2["source_hash"]) is None  # never captured there
    # every record names the source file its hash covers, and a capture under profiles/
    for key, r in rec.items():
        assert os.path.exists(os.path.join(ROOT, r["source"])), key
        assert os.path.exists(os.path.join(ROOT, r["capture"])), key
