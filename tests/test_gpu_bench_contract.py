"""bench.py's JSON line on a tiny stream: one line on stdout with the
contract's keys and consistent values (the launch clock and the events time
the same kernel; the step count and launch count follow the workload)."""
import json
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_bench_json_line_tiny_stream():
    out = subprocess.run([sys.executable, "bench.py", "--config", "tiny", "--steps", "6",
                          "--warmup", "3", "--pool", "2", "--no-cpu-baseline"],
                         cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert out.returncode == 0, out.stderr[-2000:]
    lines = [l for l in out.stdout.splitlines() if l.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
                "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config",
                "roofline", "gpu_launches", "clocks", "e2e"):
        assert key in d, key
    assert d["n_gpus"] == 1 and d["steps"] == 6 and d["warmup"] == 3
    assert d["value"] > 0 and d["higher_is_better"] is True
    assert abs(d["value"] - 1e3 / d["ms_per_step"]) <= 1e-2 * d["value"]  # ms_per_step is rounded
    r = d["roofline"]
    assert r["bound"] == "tensor" and r["unit"] == "TFLOP/s" and r["peak"] > 0
    assert r["achieved"] > 0 and abs(r["frac"] - r["achieved"] / r["peak"]) < 1e-3
    # 1 layer x 6 frames: every attention launch is clocked
    assert r["launches"] == r["launches_total"] == 6
    # three kernels per layer-frame at most (attention, merge, saliency with the admission),
    # plus the anchor copy on the first frame
    assert 6 <= d["gpu_launches"] <= 3 * 6 + 1
    e = d["e2e"]
    assert e["value"] > 0 and e["h2d_bytes_per_step"] > 0 and e["d2h_bytes_per_step"] > 0
    assert "sm_mhz" in d["clocks"] and "reasons" in d["clocks"]
    # the paper's figures as context, and this stream's bank at its end by the
    # memory law of Eq. 6: 69 rows at frame 1, one per head per later frame
    pc = d["paper_context"]
    assert pc["hardware"].startswith("NVIDIA RTX 3090") and pc["saliency_latency_ms"]["ds 2x2 (default)"] == 8.29
    assert pc["this_workload_bank_rows_per_layer_at_stream_end"] == 69 + 7
