"""bench.py's own arm on a small workload prints one JSON line with every key
of the benchmark contract (the metric, the timing, the roofline of the
dominant kernel, the clocks, the launch count, the end-to-end leg through
host buffers and the CPU baseline)."""

import json
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_bench_line_has_the_contract_keys():
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--workload", "grpo", "--steps", "3",
                        "--warmup", "3", "--e2e-steps", "2", "--ref-seconds", "1"],
                       capture_output=True, text=True, timeout=900, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-3000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.strip()]
    assert len(lines) == 1, r.stdout
    out = json.loads(lines[0])
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better", "scaling",
              "vs_baseline", "dtype", "data", "config", "roofline", "clocks", "gpu_launches", "e2e", "cpu_baseline"):
        assert k in out, k
    assert out["n_gpus"] == 1 and out["steps"] == 3 and out["warmup"] == 3 and out["higher_is_better"] is True
    assert out["value"] > 0 and out["gpu_launches"] == 9 * 3
    rf = out["roofline"]
    assert rf["bound"] == "hbm" and rf["unit"] == "GB/s" and rf["peak"] > 0
    assert rf["frac"] == pytest.approx(rf["achieved"] / rf["peak"])
    e2e = out["e2e"]
    assert e2e["value"] > 0 and e2e["h2d_bytes_per_step"] > 0 and e2e["d2h_bytes_per_step"] > 0
    assert e2e["download_matches_device"] is True
    cb = out["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] > 0
    assert set(out["clocks"]) >= {"sm_mhz", "sm_max_mhz", "reasons"}
    # the fused LM-head workload, timed in the same process after the logits step
    lm = out["kernels"]["lmhead_step (fused LM-head workload)"]
    assert (lm["M"], lm["N"], lm["K"], lm["flags"], lm["steps"]) == (32768, 151936, 4096, 0, 3)
    g = lm["gemm"]
    assert g["TFLOP/s"] > 0 and g["frac_burst"] == pytest.approx(g["TFLOP/s"] / g["peak_burst"])
    assert g["frac_sustained"] == pytest.approx(g["TFLOP/s"] / g["peak_sustained"])
    assert set(lm["clocks"]) >= {"sm_mhz", "sm_max_mhz", "reasons"}
