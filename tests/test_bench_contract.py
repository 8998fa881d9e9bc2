"""The bench's JSON line (CPU): the reference arm, which times the fp64 oracle on the host,
prints one line with the contract's keys; the workload config and the oracle sample are
described in it."""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_reference_arm_prints_one_contract_line():
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--config", "tiny",
                        "--steps", "2", "--warmup", "1"], capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.strip().splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
                "scaling", "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert key in d, key
    assert d["impl"] == "reference" and d["steps"] == 2 and d["warmup"] == 1 and d["n_gpus"] == 1
    assert d["value"] > 0 and d["higher_is_better"] is True and d["unit"] == "candidate-steps/s"
    assert d["config"]["workload"] == "tiny" and d["config"]["N"] == 4
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"] and cb["sample"]
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
    # the measured time of a sample step, and the whole-step time the value is scaled from
    assert 0 < d["ms_per_step"] < 600e3 and d["ms_per_full_step_extrapolated"] > 0


def test_clock_summary_parses_nvidia_smi_samples():
    """The bench's `clocks` key: median SM clock under load, the maximum, and every
    throttle reason seen active in any sample (what decides whether a run is kept)."""
    sys.path.insert(0, ROOT)
    import bench
    clk = bench.ClockSampler(0)
    clk.out = "\n".join([
        "1920, 2070, 1100.5, Not Active, Not Active, Not Active, Active",
        "1935, 2070, 1180.0, Not Active, Not Active, Not Active, Active",
        "1890, 2070, 1200.2, Not Active, Active, Not Active, Not Active",
        "garbage line",
        "",
    ])
    s = clk.summary()
    assert s["sm_mhz"] == 1920 and s["sm_max_mhz"] == 2070 and s["samples"] == 3
    assert s["reasons"] == ["hw_thermal_slowdown", "sw_power_cap"]
    empty = bench.ClockSampler(0)
    empty.out = ""
    assert empty.summary()["reasons"] == ["unsampled"]


def test_committed_kernel_counters_parse_and_track_their_source(tmp_path):
    """The roofline's ncu evidence comes from profiles/kernel_counters.txt: every capture
    line names its class, units, DRAM bytes and tensor-pipe activity, and a capture whose
    kernel source hash no longer matches is reported as stale (its figures are dropped)."""
    sys.path.insert(0, ROOT)
    import bench
    rec = bench.kernel_counters("self_attention")
    assert rec is not None and rec["units"] > 0 and rec["dram_bytes"] > 0 and 0 < rec["tensor_active"] <= 100
    assert os.path.exists(os.path.join(ROOT, "profiles", rec["summary"]))
    # every committed capture was taken on the kernel sources as they are now
    for cls in ("self_attention", "cross_attention", "gemm", "gemm_ffn_down"):
        r = bench.kernel_counters(cls)
        assert r is not None and r["stale"] is False, cls
    fake = tmp_path / "c.txt"
    fake.write_text("# comment\nclass=self_attention kernel=k units=2 dram_bytes=1e6 tensor_active=50 sm_mhz=1900 "
                    "src=attention.cu:0000000000000000 summary=x.md\n")
    old = bench.kernel_counters("self_attention", path=str(fake))
    assert old["stale"] is True and old["units"] == 2.0
    assert bench.kernel_counters("no_such_class", path=str(fake)) is None
