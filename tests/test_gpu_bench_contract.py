"""The benchmark's output contract: `python bench.py` prints one JSON line with
the keys, types and consistency the measurement rules ask for (run here with
few steps and a short CPU-baseline sample)."""

import json
import os
import subprocess
import sys

import pytest
import torch

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def run_bench(*args):
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *args],
                       capture_output=True, text=True, timeout=900, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-3000:]
    lines = [l for l in r.stdout.splitlines() if l.strip().startswith("{")]
    assert len(lines) == 1, r.stdout[-2000:]
    return json.loads(lines[0])


@pytest.fixture(scope="module")
def line():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    return run_bench("--steps", "5", "--warmup", "3", "--cpu-budget", "2")


def test_top_level_keys(line):
    for k, t in (("metric", str), ("value", float), ("unit", str), ("n_gpus", int),
                 ("steps", int), ("warmup", int), ("ms_per_step", float),
                 ("higher_is_better", bool), ("scaling", str), ("dtype", str), ("data", str),
                 ("config", dict), ("gpu_launches", int)):
        assert isinstance(line[k], t), k
    assert line["n_gpus"] == 1 and line["steps"] == 5 and line["warmup"] == 3
    assert line["scaling"] == "weak" and line["higher_is_better"] is True
    assert "vs_baseline" in line and line["vs_baseline"] is None
    assert "workload" in line["config"]
    # two of our kernels per timed step: the append and the attention
    assert line["gpu_launches"] == 2 * line["steps"]


def test_value_matches_step_time(line):
    flop = 1.5307149312e12 + 2.0 * 4680 * 1536 * 224
    assert abs(line["value"] - flop / (line["ms_per_step"] * 1e-3) / 1e12) <= 0.01 * line["value"]


def test_roofline_object(line):
    r = line["roofline"]
    for k in ("bound", "achieved", "peak", "unit", "frac", "traffic"):
        assert k in r, k
    assert r["bound"] == "tensor" and r["unit"] == "TFLOP/s"
    assert abs(r["frac"] - r["achieved"] / r["peak"]) < 1e-6
    assert 0.3 < r["frac"] < 1.6
    # a short timed region is compared with the burst peak (the sustained one
    # applies once the region runs for seconds under the power cap)
    assert "burst" in r["peak_source"] and abs(r["frac"] - r["frac_of_burst"]) < 1e-9


def test_append_roofline_object(line):
    a = line["roofline_append"]
    assert a["bound"] == "hbm" and a["unit"] == "GB/s"
    assert abs(a["frac"] - a["achieved"] / a["peak"]) < 1e-6
    b = a["back_to_back"]
    assert 0.0 < b["ms"] <= line["append_ms"] * 1.5
    assert abs(b["frac"] - b["achieved"] / a["peak"]) < 1e-6 and 0.05 < b["frac"] < 1.5


def test_cpu_baseline_object(line):
    c = line["cpu_baseline"]
    for k in ("value", "unit", "cores", "kind", "sample"):
        assert k in c, k
    assert c["kind"] == "oracle" and c["cores"] >= 1 and c["value"] > 0


def test_end_to_end_object(line):
    e = line["e2e"]
    for k in ("value", "unit", "h2d_bytes_per_step", "d2h_bytes_per_step"):
        assert k in e, k
    assert e["h2d_bytes_per_step"] > 0 and e["d2h_bytes_per_step"] > 0
    assert e["value"] != line["value"]  # measured separately, not repeated


def test_clock_record(line):
    c = line["clocks"]
    for k in ("sm_mhz", "sm_max_mhz", "reasons"):
        assert k in c, k
    assert isinstance(c["reasons"], list)
