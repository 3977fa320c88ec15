"""bench.py's output line on the GPU: one JSON object with every key of the
measurement contract, for NormPre-G and NormPre-L on the single 256 x 1024
workload (a few steps, no CPU baseline, no Muon pass)."""
import json
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.parametrize("variant", ["G", "L"])
def test_bench_line_contract(variant):
    cmd = [sys.executable, os.path.join(ROOT, "bench.py"), "--steps", "4", "--warmup", "3",
           "--no-cpu-baseline", "--no-muon", "--config", "single_256x1024", "--variant", variant]
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, r.stdout[-2000:]
    d = json.loads(lines[0])
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
              "scaling", "vs_baseline", "dtype", "data", "config", "e2e", "gpu_launches", "roofline",
              "clocks", "step_ms"):
        assert k in d, k
    assert d["n_gpus"] == 1 and d["steps"] == 4 and d["warmup"] >= 3
    assert d["higher_is_better"] is False and d["unit"] == "ms" and d["value"] > 0
    assert d["config"]["workload"] == "single_256x1024" and d["config"]["variant"] == variant
    assert d["gpu_launches"] > 0
    e2e = d["e2e"]
    assert e2e["value"] > 0 and e2e["h2d_bytes_per_step"] > 0 and e2e["d2h_bytes_per_step"] > 0
    roof = d["roofline"]
    assert roof["bound"] == ("tensor" if variant == "G" else "hbm")
    assert roof["unit"] == ("TFLOP/s" if variant == "G" else "GB/s")
    assert roof["achieved"] > 0 and roof["peak"] > 0
    assert abs(roof["frac"] - roof["achieved"] / roof["peak"]) <= 1e-9 * max(1.0, roof["frac"])
    st = d["step_ms"]
    assert 0 < st["p10"] <= st["p50"] <= st["p90"] and st["steps"] == 4
    assert "sm_mhz" in d["clocks"] and "reasons" in d["clocks"]


def test_bench_line_both_variants():
    """Without --variant the workload's variants all run: NormPre-G on the
    line's own keys, NormPre-L under variants.L with its own roofline (the
    sketch contractions against HBM) and end-to-end number."""
    cmd = [sys.executable, os.path.join(ROOT, "bench.py"), "--steps", "4", "--warmup", "3",
           "--no-cpu-baseline", "--no-muon", "--config", "single_256x1024"]
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, r.stdout[-2000:]
    d = json.loads(lines[0])
    assert d["config"]["variant"] == "G" and d["roofline"]["bound"] == "tensor"
    lv = d["variants"]["L"]
    assert lv["config"]["variant"] == "L" and lv["value"] > 0 and lv["gpu_launches"] > 0
    assert lv["roofline"]["bound"] == "hbm" and lv["roofline"]["achieved"] > 0
    assert lv["e2e"]["value"] > 0
    # the launch counts of the timed region are per step, not doubled by the
    # untimed passes around it
    for e in (d, lv):
        ph = e["phases"]
        assert ph["normalize"]["launches_per_step"] >= 1
        assert e["gpu_launches"] == round(sum(v["launches_per_step"] for v in ph.values()) * 4)
