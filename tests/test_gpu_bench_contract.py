"""bench.py's GPU arm prints one JSON line with every key of the benchmark contract,
consistent with itself: whole-job tokens/s from the step time, the roofline fraction
from its own numbers, the library's launch count over the timed steps, the end-to-end
number with its copied bytes, the oracle's CPU baseline and the sampled clocks."""
import json
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def run_bench(*extra):
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--shape",
                          "2048,1024,2816,8192,2", "--steps", "3", "--warmup", "3",
                          "--cpu-tokens", "4", *extra],
                         capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert out.returncode == 0, out.stderr[-3000:]
    lines = [l for l in out.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    return json.loads(lines[0])


def test_gpu_arm_prints_the_contract_line():
    d = run_bench()
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
              "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config",
              "roofline", "cpu_baseline", "e2e", "gpu_launches", "clocks"):
        assert k in d, k
    assert d["n_gpus"] == 1 and d["steps"] == 3 and d["warmup"] == 3
    assert d["higher_is_better"] is True and d["scaling"] == "weak" and d["dtype"] == "bf16"
    T = d["config"]["T"]
    assert T == 2048 and d["config"]["workload"]
    assert abs(d["value"] - T / (d["ms_per_step"] / 1e3)) < 1e-6 * d["value"]
    r = d["roofline"]
    for k in ("bound", "achieved", "peak", "unit", "frac", "traffic"):
        assert k in r, k
    assert r["bound"] == "tensor" and r["unit"] == "TFLOP/s"
    assert abs(r["frac"] - r["achieved"] / r["peak"]) < 1e-9
    c = d["cpu_baseline"]
    assert c["kind"] == "oracle" and c["value"] > 0 and c["cores"] >= 1 and c["sample"]
    e = d["e2e"]
    assert e["value"] > 0 and e["unit"] == d["unit"]
    # h (T x d bf16), targets (T int32) and every A_l (T x d_ff bf16) each step
    assert e["h2d_bytes_per_step"] == T * 1024 * 2 + T * 4 + 2 * T * 2816 * 2
    assert e["d2h_bytes_per_step"] == 4
    # the library's own count: the same kernels every step, 11 or 12 per step (the
    # projection's split tail adds one when its last wave is split)
    assert d["gpu_launches"] % 3 == 0 and 33 <= d["gpu_launches"] <= 36
    assert e["gpu_launches"] >= d["gpu_launches"]   # plus the input copies
    assert {"sm_mhz", "sm_max_mhz", "reasons"} <= set(d["clocks"])
    assert d["direct_fixup_rows_last_chunk"] == 0


def test_window_stress_goes_through_the_fixup():
    d = run_bench("--window-stress", "--no-e2e", "--no-cpu")
    assert d["direct_fixup_rows_last_chunk"] > 2048 // 2
    assert d["config"]["inputs"].startswith("window stress")


@pytest.mark.parametrize("mode,parts", [("sm1", 1), ("sm", 2)])
def test_e2e_copy_schedules_launch_one_copy_per_part(mode, parts):
    """The end-to-end loop issues, every step, the step's kernels plus one input-copy
    launch per part: one for `sm1`; for `sm` one per long GEMM phase of the error signal,
    i.e. the logits pass and the projection of the shape's single token chunk."""
    d = run_bench("--no-cpu", "--e2e-copy", mode)
    e = d["e2e"]
    assert e["gpu_launches"] - d["gpu_launches"] == parts * d["steps"]
    assert e["h2d_bytes_per_step"] == 2048 * 1024 * 2 + 2048 * 4 + 2 * 2048 * 2816 * 2
