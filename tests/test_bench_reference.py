"""The benchmark's reference arm (the CPU oracle) keeps the line contract.

`bench.py --impl reference` times the oracle on the host cores and prints one
JSON line with the same metric, unit and config keys as the GPU arm, plus its
own cpu_baseline and e2e objects.  Run here on the small workload (256 x 512
-> 512), which takes about a second; no GPU is involved.
"""

import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_reference_line():
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                          "--workload", "single_m256_k512_n512", "--steps", "2", "--warmup", "3"],
                         check=True, capture_output=True, text=True, timeout=600, cwd=ROOT).stdout
    lines = [l for l in out.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference"
    assert d["metric"].startswith("W8A8 linear INT8 TOPS") and d["unit"] == "TOPS"
    assert d["value"] > 0 and d["higher_is_better"] is True
    assert d["steps"] == 2 and d["warmup"] == 3 and d["n_gpus"] == 1
    assert d["config"]["workload"] == "single_m256_k512_n512"
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"]
    assert d["e2e"]["value"] == d["value"] and d["e2e"]["h2d_bytes_per_step"] == 0


def test_warmup_floor():
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--warmup", "1"],
                       capture_output=True, text=True, timeout=120, cwd=ROOT)
    assert r.returncode != 0 and "warmup" in r.stderr
