"""The one JSON line bench.py prints, as the benchmark contract fixes it: the
GPU arm (tiny workload, on the GPU) and the reference arm (the oracle on the
host cores, tiny workload).  Run as child processes, the way the driver
launches them."""

import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _run(args, timeout=900):
    out = subprocess.run([sys.executable, "bench.py", *args], cwd=ROOT, capture_output=True,
                         text=True, timeout=timeout)
    assert out.returncode == 0, out.stderr[-3000:]
    lines = [ln for ln in out.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, out.stdout[-3000:]
    return json.loads(lines[0])


def _common(d):
    for key in ("metric", "unit", "dtype", "data", "scaling"):
        assert isinstance(d[key], str) and d[key]
    assert d["value"] > 0 and d["ms_per_step"] > 0
    assert d["n_gpus"] == 1 and d["higher_is_better"] is True
    assert d["steps"] >= 1 and d["warmup"] >= 3
    assert "vs_baseline" in d
    assert d["config"]["workload"].startswith("tiny")


@pytest.mark.gpu
def test_gpu_arm_line():
    d = _run(["--workload", "tiny", "--steps", "2", "--warmup", "3", "--no-cpu-baseline",
              "--e2e-steps", "1"])
    _common(d)
    rf = d["roofline"]
    assert rf["bound"] == "hbm" and rf["unit"] == "GB/s"
    assert rf["achieved"] > 0 and rf["peak"] > 0
    assert abs(rf["frac"] - rf["achieved"] / rf["peak"]) < 1e-9
    assert "traffic" in rf
    e2e = d["e2e"]
    assert e2e["value"] > 0 and e2e["unit"] == d["unit"]
    assert e2e["h2d_bytes_per_step"] > 0 and e2e["d2h_bytes_per_step"] > 0
    clocks = d["clocks"]
    if clocks is None:
        # no nvidia-smi sample fell inside a timed region this short
        assert d["ms_per_step"] * d["steps"] < 1000.0
    else:
        assert clocks["sm_mhz"] > 0 and clocks["sm_max_mhz"] > 0
        assert isinstance(clocks["reasons"], list)
    assert d["gpu_launches"] > 0
    assert d["batched_requests"]["requests_per_call"] == 4


def test_reference_arm_line():
    d = _run(["--impl", "reference", "--workload", "tiny", "--steps", "1", "--warmup", "3",
              "--ref-step-seconds", "0.2"])
    _common(d)
    assert d["impl"] == "reference"
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"]
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}
