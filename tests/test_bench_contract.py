"""The benchmark's reference leg (the CPU oracle) prints the one JSON line
the measurement contract asks for; CPU only."""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

KEYS = {"impl", "metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
        "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config",
        "cpu_baseline", "e2e"}


def _run(*args, env=None):
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *args],
                         capture_output=True, text=True, timeout=600, cwd=ROOT,
                         env=dict(os.environ, **(env or {})))
    assert out.returncode == 0, out.stderr[-2000:]
    return [ln for ln in out.stdout.splitlines() if ln.strip()]


@pytest.mark.parametrize("workload", [None, "dsnn_784_1000_1000_10_T25_B128",
                                      "rleaky_T25_B128_N1000",
                                      "csnn_12c5_mp2_64c5_mp2_10_T25_B128"])
def test_reference_leg_prints_one_contract_line(workload):
    args = ["--impl", "reference", "--steps", "2", "--warmup", "1", "--reference-seconds", "3"]
    if workload:
        args += ["--workload", workload]
    lines = _run(*args)
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert KEYS <= set(d)
    assert d["impl"] == "reference" and d["value"] > 0 and d["steps"] == 2
    assert d["higher_is_better"] is True and d["vs_baseline"] is None
    assert d["config"]["workload"] == (workload or "leaky_bf16_T500_B64_N8192")
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"]
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}


def test_reference_leg_other_ranks_print_nothing():
    lines = _run("--impl", "reference", "--steps", "1", "--warmup", "0",
                 "--reference-seconds", "1", env={"RANK": "1", "WORLD_SIZE": "2"})
    assert lines == []
