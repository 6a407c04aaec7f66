"""Host-side logic of bench.py (no GPU): the clocks summary taken from the
nvidia-smi samples, and the JSON contract of the reference arm (the oracle
timed on the host cores), alone and under torchrun with two ranks."""
import json
import os
import subprocess
import sys

import pytest

from conftest import ROOT

sys.path.insert(0, ROOT)
import bench  # noqa: E402

SAMPLES = [
    "0, 2070, 2070, 610.5, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active\n",
    "1, 1200, 2070, 100.0, 0x0000000000000004, Not Active, Not Active, Not Active, Active\n",
    "0, 1965, 2070, 1390.0, 0x0000000000000004, Not Active, Not Active, Not Active, Active\n",
    "0, 2070, 2070, 700.0, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active\n",
    "garbage line\n",
]


def test_clock_summary_median_and_reasons():
    c = bench.summarise_clocks(SAMPLES, 0)
    assert c == {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "samples": 3, "reasons": ["sw_power_cap"]}
    c1 = bench.summarise_clocks(SAMPLES, 1)
    assert c1["sm_mhz"] == 1200.0 and c1["samples"] == 1
    assert bench.summarise_clocks(["x\n"], 0) is None
    hot = ["0, 1500, 2070, 900, 0x48, Active, Active, Not Active, Not Active\n"]
    assert bench.summarise_clocks(hot, 0)["reasons"] == ["hw_slowdown", "hw_thermal_slowdown"]


def test_clock_sampler_stop_reads_and_removes_its_file():
    s = bench.ClockSampler()
    s.proc = subprocess.Popen(["sleep", "30"])
    with open(s.path, "w") as fh:
        fh.writelines(SAMPLES)
    c = s.stop(0)
    assert c["samples"] == 3 and c["reasons"] == ["sw_power_cap"]
    assert not os.path.exists(s.path)


def _reference_line(out):
    lines = [ln for ln in out.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, out
    return json.loads(lines[0])


def _check_reference(d, n):
    assert d["impl"] == "reference"
    assert d["metric"] == bench.METRIC and d["unit"] == bench.UNIT
    assert d["higher_is_better"] is True and d["n_gpus"] == n
    assert d["value"] > 0 and d["ms_per_step"] > 0
    assert d["config"]["workload"] == bench.WORKLOAD["workload"]
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"] and cb["sample"]
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}


def test_reference_arm_json_line():
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--steps", "1", "--warmup", "3"],
                       cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    _check_reference(_reference_line(r.stdout), 1)


def _free_port():
    import socket
    with socket.socket(socket.AF_INET, socket.SOCK_STREAM) as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def test_reference_arm_under_torchrun_prints_once():
    pytest.importorskip("torch.distributed.run")
    r = subprocess.run([sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
                        "--master-addr", "127.0.0.1", "--master-port", str(_free_port()), "bench.py", "--impl",
                        "reference", "--gpus", "2", "--steps", "1", "--warmup", "3"],
                       cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    _check_reference(_reference_line(r.stdout), 2)


def test_cpu_baseline_leg_is_bounded():
    import time
    t0 = time.perf_counter()
    cb = bench.cpu_baseline(budget_s=0.5)
    assert time.perf_counter() - t0 < 60
    assert cb["kind"] == "oracle" and cb["unit"] == bench.UNIT and cb["value"] > 0 and cb["cores"] >= 1
    assert "output rows" in cb["sample"]


def test_oracle_sample_ops_scale_with_rows():
    from concurrent.futures import ThreadPoolExecutor
    with ThreadPoolExecutor(max_workers=2) as pool:
        s = bench.OracleSample(pool)
        per_row = 2 * bench.Q_ * bench.CO_ * bench.R_ * bench.S_ * bench.C_
        assert s.run(1) == per_row and s.run(3) == 3 * per_row
        assert 1 <= s.rows_for_budget(0.001) <= s.rows_for_budget(1.0) <= bench.N_ * bench.P_
