"""bench.py keeps its output contract: one JSON line with the keys the benchmark harness reads."""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
BASE_KEYS = {"metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better", "scaling",
             "vs_baseline", "dtype", "data", "config", "e2e"}


def _run(args, timeout=600):
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *args], capture_output=True, text=True,
                       timeout=timeout, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.strip().splitlines() if l.startswith("{")]
    assert len(lines) == 1, r.stdout
    return json.loads(lines[0])


def test_reference_arm_line():
    j = _run(["--impl", "reference", "--workload", "flat1m", "--steps", "1", "--warmup", "0"])
    assert BASE_KEYS <= set(j)
    assert j["impl"] == "reference" and j["value"] > 0 and j["higher_is_better"] is True
    assert j["cpu_baseline"]["kind"] == "oracle" and j["cpu_baseline"]["cores"] >= 1
    assert j["e2e"] == {"value": j["value"], "unit": j["unit"], "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
    assert j["config"]["workload"].startswith("flat1m")


@pytest.mark.gpu
def test_gpu_line_has_roofline_e2e_clocks():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    j = _run(["--workload", "flat1m", "--steps", "3", "--warmup", "3", "--no-cpu-baseline"])
    assert BASE_KEYS <= set(j)
    r = j["roofline"]
    assert r["bound"] == "hbm" and r["unit"] == "GB/s" and 0 < r["frac"] < 2 and r["peak"] > 0
    assert j["e2e"]["value"] > 0 and j["e2e"]["h2d_bytes_per_step"] > 0 and j["e2e"]["d2h_bytes_per_step"] > 0
    assert j["gpu_launches"] == 3 * (2 * 4 + 1)          # fused round: tau fills, tau-1 local steps, K6, K5
    assert j["n_gpus"] == 1 and j["scaling"] == "weak" and j["value"] > 0
    assert "clocks" in j
