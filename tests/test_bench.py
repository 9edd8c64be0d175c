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


def _wl(key, **hp_changes):
    import dataclasses
    import workloads as W
    wl = W.WORKLOADS[key]
    return dataclasses.replace(wl, hp=dataclasses.replace(wl.hp, **hp_changes)) if hp_changes else wl


def test_algorithmic_byte_counts():
    """The byte counts behind every roofline fraction, against the counts written out by hand from what
    each kernel reads and writes (4-byte states, 4- or 2-byte gradients)."""
    sys.path.insert(0, ROOT)
    import bench
    import workloads as W
    fused = W.FLAG_FUSED_ROUND
    s = _wl("gpt2s", flags=fused)                     # AdamW, fp32 g, n = 4
    m = _wl("gpt2m", flags=fused)                     # AdamW, bf16 g, n = 8
    lg = _wl("gpt2l", flags=fused)                    # SGD-momentum, fp32 g, n = 8
    # local step per worker-element: x, states, g read; x, states written
    assert bench.bytes_per_elem_local(s) == 4 + 8 + 4 + 4 + 8 == 28
    assert bench.bytes_per_elem_local(m) == 26
    assert bench.bytes_per_elem_local(lg) == 20
    assert bench.bytes_per_elem_local(s, zero_state=True) == 20      # states written, not read
    assert bench.bytes_per_elem_local(lg, zero_state=True) == 16
    # a whole launch; from x: x read once per tile, not once per worker
    assert bench.local_step_bytes(s) == 4 * s.d * 28
    assert bench.local_step_bytes(s, from_x=True) == 4 * s.d * 24 + s.d * 4
    # separate global step: x, m and n replicas read and written (the replicas not written when deferred)
    assert bench.bytes_per_param_global(s) == 8 * (4 + 2) == 48
    assert bench.bytes_per_param_global(m) == 80
    assert bench.bytes_per_param_global(_wl("gpt2s", global_mode=W.GLOBAL_ADAMW)) == 56
    assert bench.bytes_per_param_global(s, lazy_reset=True) == 48 - 16
    # fused last step + global step: per worker x_i, states and g read, states written; x, m read and written
    assert bench.bytes_per_param_fused_last(s) == 4 * (4 + 16 + 4) + 16 == 112
    assert bench.bytes_per_param_fused_last(m) == 8 * (4 + 16 + 2) + 16 == 192
    assert bench.bytes_per_param_fused_last(lg) == 8 * (4 + 8 + 4) + 16 == 144
    assert bench.bytes_per_param_fused_last(_wl("gpt2s", flags=fused, global_mode=W.GLOBAL_ADAMW)) == 120
    assert bench.bytes_per_param_fused_last(s, from_x=True) == 4 * (16 + 4) + 16
    reset = _wl("gpt2s", flags=fused | W.FLAG_RESET_LOCAL_STATE)
    assert bench.bytes_per_param_fused_last(reset) == 4 * (4 + 8 + 4) + 16            # states not written
    assert bench.bytes_per_param_fused_last(reset, from_x=True, zero_state=True) == 4 * 4 + 16
    # the rounds' totals quoted for the workloads (gradient fill excluded), unfused and fused
    for key, unfused, fused_total in (("gpt2s", 1392, 1332), ("gpt2m", 5072, 4948), ("gpt2l", 2000, 1876),
                                      ("gpt2xl", 2544, 2484)):
        w = _wl(key, flags=fused)
        u = w.tau * w.n * bench.bytes_per_elem_local(w) + bench.bytes_per_param_global(w)
        f = (w.tau - 2) * w.n * bench.bytes_per_elem_local(w) + bench.local_step_bytes(w, from_x=True) / w.d \
            + bench.bytes_per_param_fused_last(w)
        assert (u, f) == (unfused, fused_total), key


def test_workload_selection_names_only_changes():
    sys.path.insert(0, ROOT)
    import argparse
    import bench
    args = argparse.Namespace(workload="gpt2s", n_workers=None, tau=None, global_mode=None, fused=True,
                              reset_local_state=False, max_params=None, flat_params=None)
    import workloads as W
    assert bench.select_workload(args).name == W.WORKLOADS["gpt2s"].name
    args.tau, args.reset_local_state = 2, True
    name = bench.select_workload(args).name
    assert "tau=2" in name and "restarted" in name
    args.flat_params = 1000
    wl = bench.select_workload(args)
    assert wl.d == 1000 and len(wl.tensors) == 1 and "flat tensor of 1000" in wl.name


def test_clock_records_that_call_for_a_second_measurement():
    """hw_slowdown, hw_thermal_slowdown and sw_thermal_slowdown reject a timed region, and so do SM clocks
    well below their maximum with no reason given; sw_power_cap alone is kept."""
    sys.path.insert(0, ROOT)
    import bench
    ok = {"reasons": [], "sm_mhz": 2070.0, "sm_max_mhz": 2070.0}
    assert not bench.clocks_rejected(None) and not bench.clocks_rejected(ok)
    assert not bench.clocks_rejected(dict(ok, reasons=["sw_power_cap"], sm_mhz=1750.0))
    for reason in ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown"):
        assert bench.clocks_rejected(dict(ok, reasons=[reason]))
    assert bench.clocks_rejected(dict(ok, sm_mhz=1500.0))
    assert bench.any_rank(True, 1) and not bench.any_rank(False, 1)
