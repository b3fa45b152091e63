"""The whole-model decode step of bench.py (random Qwen3-style blocks around
the library's attention and pool, Sec. 4.1 / Sec. 3.2) runs on the paper's
model shape and leaves no device status set."""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.gpu
@pytest.mark.parametrize("workload", ["paper_k8", "tiny_f32"])
def test_model_mode_runs(workload):
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--mode", "model",
                        "--workload", workload, "--steps", "3", "--warmup", "3"],
                       cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    line = json.loads([l for l in r.stdout.splitlines() if l.startswith("{")][-1])
    assert line["value"] > 0 and line["config"]["mode"] == "model"
    assert 0.0 < line["whitematter_share"] < 1.0
