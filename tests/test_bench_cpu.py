"""Host logic of bench.py that decides whether a timing is kept: the clock
summary (throttle reasons must be reported) and the workload bookkeeping."""
import bench


def test_clock_summary_reports_throttling():
    lines = [
        "0, 2070, 2070, 900.5, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active",
        "0, 1995, 2070, 1390.0, 0x0000000000000004, Not Active, Not Active, Not Active, Active",
        "0, 2070, 2070, 1010.2, 0x0000000000000000, Not Active, Active, Not Active, Not Active",
        "garbage line",
        "0, [N/A], 2070, 0, 0x0, Not Active, Not Active, Not Active, Not Active",
    ]
    s = bench.ClockSampler.summarize(lines)
    assert s["samples"] == 3
    assert s["sm_mhz"] == 2070.0 and s["sm_max_mhz"] == 2070.0
    assert s["reasons"] == ["hw_thermal_slowdown", "sw_power_cap"]


def test_clock_summary_clean_and_empty():
    clean = ["0, 2070, 2070, 800, 0x0, Not Active, Not Active, Not Active, Not Active"] * 4
    assert bench.ClockSampler.summarize(clean) == {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": [],
                                                    "samples": 4}
    assert bench.ClockSampler.summarize([])["sm_mhz"] is None


def test_clock_sampler_queries_the_gpu_in_use():
    """nvidia-smi numbers every GPU of the machine; CUDA only the visible ones."""
    assert bench.smi_gpu_id(0, None) == "0" and bench.smi_gpu_id(3, "") == "3"
    assert bench.smi_gpu_id(0, "5") == "5"
    assert bench.smi_gpu_id(1, "4, 6,7") == "6"
    assert bench.smi_gpu_id(0, "GPU-1a2b") == "GPU-1a2b"


def test_default_workload_is_the_conv2x_layer():
    wl = bench.workload_by_name("conv2x", None)
    assert (wl["N"], wl["C"], wl["H"], wl["W"], wl["K"], wl["R"], wl["S"]) == (32, 64, 56, 56, 64, 3, 3)
    assert wl["terms"] == 32 * 64 * 56 * 56 * 64 * 9 == 3_699_376_128
    assert 32 % bench.E2E_CHUNKS == 0


def _run_bench(args, env_extra=None):
    import json
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    env = dict(os.environ, **(env_extra or {}))
    r = subprocess.run([sys.executable, os.path.join(root, "bench.py"), *args], capture_output=True, text=True,
                       env=env, cwd=root, timeout=300)
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    return r.returncode, [json.loads(ln) for ln in lines], r.stderr


def test_reference_arm_prints_the_contract_line():
    """--impl reference times the oracle on the host (no GPU) and prints one JSON line with the base keys."""
    rc, lines, err = _run_bench(["--impl", "reference", "--steps", "1", "--warmup", "1"])
    assert rc == 0, err
    assert len(lines) == 1
    d = lines[0]
    assert d["impl"] == "reference" and d["value"] > 0 and d["unit"] == d["metric"]
    for key in ("n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better", "scaling", "vs_baseline", "dtype",
                "data", "config"):
        assert key in d, key
    assert d["steps"] == 1 and d["warmup"] == 1 and d["higher_is_better"] is True
    assert d["config"]["workload"] == "resnet18_conv2x_convshift_3x3"
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"] and cb["sample"]
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}


def test_reference_arm_runs_on_rank_zero_only():
    rc, lines, err = _run_bench(["--impl", "reference", "--steps", "1", "--warmup", "1"],
                                {"RANK": "1", "WORLD_SIZE": "2", "LOCAL_RANK": "1"})
    assert rc == 0, err
    assert lines == []


def test_all_cores_oracle_timing_covers_the_batch():
    """The all-cores CPU baseline splits the batch over spawned processes and times the whole of it."""
    wl = dict(name="tiny", N=5, C=3, H=6, W=5, K=4, R=3, S=3, stride=1, pad=1, terms=5 * 4 * 6 * 5 * 3 * 9)
    r = bench.cpu_baseline_all_cores(wl, cores=2)
    assert r["kind"] == "oracle" and r["cores"] == 2 and r["value"] > 0 and r["unit"] == bench.METRIC
    assert "all 5 images" in r["sample"]
