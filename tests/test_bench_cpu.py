"""bench.py's CPU legs: the oracle baseline's bounded sample and the reference arm's JSON line."""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SMALL = "pythia160m-mlkv6-b1-L128"


def test_oracle_sample_counts_repeated_steps():
    sys.path.insert(0, ROOT)
    import bench
    from mlkv_synth import workloads
    w = workloads.by_name(SMALL)
    wall, cpu, seqs = bench.oracle_sample(w, 1, 2, reps=3)
    assert wall > 0 and cpu >= 0
    assert seqs == 3


def test_cpu_baseline_grows_to_its_budget():
    # One sequence of 128 positions is far below the budget: whole steps are repeated.
    sys.path.insert(0, ROOT)
    import bench
    from mlkv_synth import workloads
    w = workloads.by_name(SMALL)
    cb = bench.cpu_baseline(w, budget_cpu_s=0.3)
    assert cb["kind"] == "oracle" and cb["unit"] == bench.UNIT
    assert cb["cores"] >= 1 and cb["value"] > 0
    assert "decode steps" in cb["sample"]


def test_reference_arm_line():
    out = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--config", SMALL,
                          "--steps", "2", "--warmup", "1"], cwd=ROOT, capture_output=True,
                         text=True, timeout=300)
    assert out.returncode == 0, out.stderr[-2000:]
    line = json.loads(out.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference"
    assert line["value"] > 0 and line["steps"] == 2
    assert line["warmup"] == 3   # at least three warm-up steps, whatever is asked
    assert line["e2e"] == {"value": line["value"], "unit": line["unit"],
                           "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
    assert line["cpu_baseline"]["kind"] == "oracle"
    assert line["cpu_baseline"]["value"] == pytest.approx(line["value"])
    assert line["config"]["workload"] == SMALL


def test_recorded_traffic_needs_current_kernel_and_launch_kind():
    """The roofline's `traffic` is taken from a recorded ncu capture only when the capture was of
    the kernel sources as they are and of the same launch kind (one multi-layer launch per step,
    or one launch per layer); otherwise it is null."""
    sys.path.insert(0, ROOT)
    import bench
    from mlkv_synth import workloads
    with open(os.path.join(ROOT, "profiles", "decode_traffic.json")) as f:
        rec = json.load(f)
    forms = ("multi-layer", "fused", "per-layer")
    for entry in rec["entries"]:
        assert entry["launch"] in forms
        assert entry["dram_bytes_per_launch"] > 0
        # the summary the figure comes from states it and the sources it was taken on
        with open(os.path.join(ROOT, entry["source"])) as f:
            summary = f.read()
        assert f"{entry['dram_bytes_per_launch']:,}" in summary, entry["source"]
        assert entry["kernel_source_sha256_16"] in summary, entry["source"]
        w = workloads.by_name(entry["workload"])
        current = entry["kernel_source_sha256_16"] == bench._kernel_source_hash(entry["kernel"])
        got = bench._recorded_traffic(w, entry["kernel"], entry["launch"])
        assert got == (entry["dram_bytes_per_launch"] if current else None)
        for other in forms:
            if other != entry["launch"] and not any(
                    e["workload"] == entry["workload"] and e["launch"] == other
                    for e in rec["entries"]):
                assert bench._recorded_traffic(w, entry["kernel"], other) is None
        assert bench._recorded_traffic(w, "no_such_kernel", entry["launch"]) is None
