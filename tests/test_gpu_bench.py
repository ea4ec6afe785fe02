"""bench.py end to end on the small single-block workload: one JSON line with
the keys the measurement contract asks for (metric, value, roofline,
cpu_baseline, e2e with both copy directions, clocks, launch count), every
leg of the run completing."""
import json
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_bench_line_on_the_single_block_workload(cuda_ok, tmp_path):
    out = tmp_path / "line.json"
    trace = tmp_path / "trace.jsonl"
    cmd = [sys.executable, os.path.join(ROOT, "bench.py"), "--config", "c1", "--steps", "4", "--warmup", "3",
           "--no-dit", "--cpu-budget-s", "2", "--out", str(out), "--trace", str(trace), "--nvtx"]
    res = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert res.returncode == 0, res.stderr[-2000:]
    lines = [ln for ln in res.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, res.stdout[-2000:]
    line = json.loads(lines[0])
    assert line == json.loads(out.read_text())
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
              "scaling", "vs_baseline", "dtype", "data", "config", "roofline", "cpu_baseline", "e2e",
              "e2e_unpadded", "clocks", "gpu_launches", "q_delta_roofline", "ms_per_step_serial",
              "always_refresh_ms_per_step"):
        assert k in line, k
    assert line["value"] > 0 and line["steps"] == 4 and line["warmup"] == 3 and line["n_gpus"] == 1
    assert line["higher_is_better"] is False and line["config"]["name"] == "c1"
    assert line["gpu_launches"] > 0 and line["roofline"]["achieved"] > 0
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["value"] > 0
    e2e = line["e2e"]
    assert e2e["value"] > 0 and e2e["h2d_bytes_per_step"] > 0 and e2e["d2h_bytes_per_step"] > 0, e2e
    assert line["e2e_unpadded"]["value"] > 0
    # the observation record of the trajectory: one line per (step, block)
    recs = [json.loads(x) for x in trace.read_text().splitlines()]
    cfg = line["config"]
    assert len(recs) == cfg["trajectory_steps"] * cfg["blocks"]
    assert {tuple(sorted(r)) for r in recs} == {("a_b", "b", "gbar", "m_bar_read", "mode", "t")}
    by_t = {r["t"]: r["mode"][0] for r in recs if r["b"] == 0}
    assert [by_t[int(t)] for t in sorted(line["modes_per_step"], key=int)] == \
        [line["modes_per_step"][t][0] for t in sorted(line["modes_per_step"], key=int)]


def test_bench_separate_cache_update_schedule(cuda_ok):
    """--separate-cache-update adds one refadapt_ref_cache_update launch per
    block and step to the count; the same trajectory's modes either way."""
    def line(extra):
        cmd = [sys.executable, os.path.join(ROOT, "bench.py"), "--config", "c1", "--steps", "4", "--warmup", "3",
               "--no-dit", "--no-e2e", "--no-cpu-baseline", "--no-refresh-baseline", "--no-graph", "--no-serial",
               "--no-nested"] + extra
        res = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600)
        assert res.returncode == 0, res.stderr[-2000:]
        return json.loads([ln for ln in res.stdout.splitlines() if ln.startswith("{")][-1])

    fused, separate = line([]), line(["--separate-cache-update"])
    assert fused["modes_per_step"] == separate["modes_per_step"]
    blocks = fused["config"]["blocks"]
    assert separate["gpu_launches"] - fused["gpu_launches"] == blocks * fused["steps"]
