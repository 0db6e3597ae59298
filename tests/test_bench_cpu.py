"""bench.py's reference arm (the float64 oracle timed on the host) runs without
a GPU: on the small workload it prints one JSON line with the keys the driver
reads."""

import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_reference_arm_prints_one_json_line():
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload", "tiny",
                        "--steps", "2", "--warmup", "1", "--ref-seconds", "1"],
                       capture_output=True, text=True, timeout=600, env=env, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.strip()]
    assert len(lines) == 1, r.stdout
    out = json.loads(lines[0])
    assert out["impl"] == "reference" and out["unit"] == "tokens/s" and out["higher_is_better"] is True
    assert out["value"] > 0 and out["steps"] == 2 and out["warmup"] == 1
    assert out["config"]["workload"].startswith("tiny")
    # the same config, key for key, as the repository's own arm prints for this workload
    sys.path.insert(0, ROOT)
    import bench
    import workloads as W
    spec = W.SPECS["tiny"]
    assert out["config"] == bench._logits_config(spec, W.generate(spec, seed=W.seed_for(spec.name)), 1)
    cb = out["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == out["value"] and "sampled rows" in cb["sample"]
    assert cb["cores"] == len(os.sched_getaffinity(0)) or cb["cores"] == 32
    assert f"{cb['cores']} processes" in cb["sample"]
    assert out["e2e"] == {"value": out["value"], "unit": "tokens/s", "h2d_bytes_per_step": 0,
                          "d2h_bytes_per_step": 0}


def test_traffic_key_ignores_comments_only():
    """The DRAM-traffic table is keyed to a kernel's code: an edited comment
    keeps the key, an edited statement changes it."""
    import bench
    a = "int f(int x) {  // one\n    return x + 1; /* two */\n}\n"
    b = "// header\nint f(int x) {  // other words\n\n    return x + 1;\n}\n"
    c = "int f(int x) {\n    return x + 2;\n}\n"
    assert bench._code_only(a) == bench._code_only(b)
    assert bench._code_only(a) != bench._code_only(c)
