"""The benchmark's JSON line: the keys and value types the benchmark contract
asks for, on the smallest workload.

- the reference arm (the fp64 oracle on the host cores) runs without a GPU;
- the default arm (marked gpu) times the library, with the end-to-end,
  roofline, CPU-baseline, clock and launch-count objects.
"""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SMALL = "k2_n256_d128_v4096"
BASE_KEYS = {"metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
             "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config"}


def _run(*args, timeout=600) -> dict:
    proc = subprocess.run([sys.executable, "bench.py", *args], cwd=ROOT, capture_output=True,
                          text=True, timeout=timeout)
    assert proc.returncode == 0, proc.stderr[-4000:]
    out = proc.stdout
    lines = [ln for ln in out.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, out          # exactly one JSON line on stdout
    return json.loads(lines[0])


def _check_base(j: dict, steps: int, warmup: int):
    assert BASE_KEYS <= j.keys(), BASE_KEYS - j.keys()
    assert j["value"] > 0 and j["ms_per_step"] > 0
    assert j["n_gpus"] == 1 and j["steps"] == steps and j["warmup"] == warmup
    assert j["higher_is_better"] is True and j["unit"] == "tokens/s"
    assert j["scaling"] in ("weak", "strong")
    assert j["config"]["workload"] == SMALL
    assert j["vs_baseline"] is None


def test_cpu_baseline_sample_stays_within_the_workload():
    sys.path.insert(0, ROOT)
    import bench
    wl = bench.workload_from_name(SMALL)
    cb = bench.cpu_baseline(wl, 0.5)
    rows = int(cb["sample"].split()[1])          # "first <rows> tokens of each ..."
    assert cb["value"] > 0 and 1 <= rows <= wl.N


def test_reference_arm_line():
    j = _run("--impl", "reference", "--steps", "1", "--warmup", "3", "--workload", SMALL)
    _check_base(j, 1, 3)
    assert j["impl"] == "reference" and j["dtype"] == "f64"
    cb = j["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == j["value"]
    assert cb["sample"]
    assert j["e2e"] == {"value": j["value"], "unit": j["unit"], "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}


@pytest.mark.gpu
def test_default_arm_line():
    j = _run("--steps", "3", "--warmup", "3", "--workload", SMALL, "--cpu-seconds", "1")
    _check_base(j, 3, 3)
    assert j["dtype"] == "bf16" and j["data"] == "synthetic"
    assert "not a reportable configuration" in j["config"]["l2"]   # 1 MB of inputs
    r = j["roofline"]
    assert r["bound"] == "tensor" and r["unit"] == "TFLOP/s"
    assert r["achieved"] > 0 and r["peak"] > 0
    assert abs(r["frac"] - r["achieved"] / r["peak"]) < 1e-9
    assert "traffic" in r
    cb = j["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] > 0 and cb["cores"] >= 1 and cb["sample"]
    e = j["e2e"]
    assert e["value"] > 0 and e["unit"] == j["unit"]
    # hidden states (bf16) and targets (int32) in, losses back, per step
    assert e["h2d_bytes_per_step"] >= 2 * 256 * 128 * 2 + 2 * 256 * 4
    assert e["d2h_bytes_per_step"] > 0
    c = j["clocks"]
    assert {"sm_mhz", "sm_max_mhz", "reasons"} <= c.keys()
    # the library's own kernels, counted around the timed calls
    assert j["gpu_launches"] >= 3 * 8
    assert j["device_flags"] == 0
