"""The bench's reference arm (the oracle timed on the host cores) keeps the
JSON contract of the GPU arm's line: the same metric, unit and workload
config, `impl: reference`, a cpu_baseline describing the run, and an e2e entry
with no host-device traffic."""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_reference_arm_line():
    out = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--steps", "1",
                          "--warmup", "3", "--oracle-layers", "1"],
                         cwd=ROOT, capture_output=True, text=True, timeout=900)
    assert out.returncode == 0, out.stderr[-2000:]
    d = json.loads(out.stdout.strip().splitlines()[-1])
    sys.path.insert(0, ROOT)
    import bench
    from paper_2609_17983_gb300 import synth
    assert d["impl"] == "reference"
    assert d["metric"] == bench.METRIC and d["unit"] == "positions/s"
    assert d["config"] == bench.workload_config(synth.preset(bench.WORKLOAD), 1)
    assert d["steps"] == 1 and d["warmup"] == 3 and d["n_gpus"] == 1
    assert d["higher_is_better"] is True and d["vs_baseline"] is None
    # a step is the 40 rows through the first layers_per_step of 32 layers, as it ran
    assert d["layers_per_step"] == 1 and d["layers_per_position"] == 32
    assert d["value"] > 0 and abs(d["value"] * d["ms_per_step"] / 1e3 - 40 / 32) < 1e-9
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == d["value"] and cb["cores"] >= 1
    assert "first 1 of 32 layers" in cb["sample"]
    assert d["e2e"] == {"value": d["value"], "unit": "positions/s", "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}
