"""The bench's reference arm (the float64 oracle timed on the host cores) prints the JSON line
the measurement contract asks for; it runs on the CPU, so it is checked here."""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _run(*args):
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--steps", "1", "--warmup", "3", *args],
                       capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    return json.loads(r.stdout.strip().splitlines()[-1])


def test_reference_line_keys():
    d = _run("--workload", "tiny_f32", "--cpu-tokens", "64")
    assert d["impl"] == "reference" and d["unit"] == "tokens/s" and d["higher_is_better"]
    assert d["value"] > 0 and d["ms_per_step"] > 0 and d["n_gpus"] == 1
    assert d["config"]["workload"] == "tiny_f32"
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"]
    e2e = d["e2e"]
    assert e2e["value"] == d["value"] and e2e["unit"] == d["unit"]
    assert e2e["h2d_bytes_per_step"] == 0 and e2e["d2h_bytes_per_step"] == 0


def test_reference_counts_shared_experts_and_layers():
    plain = _run("--workload", "tiny_f32", "--cpu-tokens", "64")
    shared = _run("--workload", "tiny_f32", "--cpu-tokens", "64", "--shared-experts", "2",
                  "--shared-dff", "64")
    assert shared["config"]["shared_experts"] == 2
    assert "2 shared experts of d_ff 64" in shared["cpu_baseline"]["sample"]
    assert plain["config"]["shared_experts"] == 0
