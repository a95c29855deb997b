"""bench.py's reference arm (the oracle timed on the host) for each kind of workload:
one JSON line with the contract's keys, on the GPU arm's metric and workload."""

import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

KEYS = {"metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
        "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "impl", "config",
        "cpu_baseline", "e2e"}


@pytest.mark.parametrize("workload,metric_word", [("tiny", "chunk-attention"),
                                                  ("convtiny", "convolution"),
                                                  ("block1p3b", "DiT-block")])
def test_reference_arm_prints_one_contract_line(workload, metric_word):
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--workload", workload,
                        "--steps", "2", "--warmup", "3", "--ref-seconds", "1"],
                       cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert KEYS <= set(d), KEYS - set(d)
    assert d["impl"] == "reference" and metric_word in d["metric"]
    assert d["config"]["workload"].startswith(workload + ":")
    assert d["value"] > 0 and d["cpu_baseline"]["value"] == d["value"]
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] >= 1
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}
    assert d["steps"] == 2 and d["warmup"] == 3
