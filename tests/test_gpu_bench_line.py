"""The bench's own arm on the GPU (tiny workload, a few steps): one JSON line with the
contract's keys, the kernel launches counted, the end-to-end number through the host-buffer
entry point, and the second timed region that runs one complete search."""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.gpu
def test_bench_line_on_the_tiny_workload():
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--config", "tiny", "--steps", "4",
                        "--warmup", "3", "--no-cpu-baseline"], capture_output=True, text=True, timeout=900, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-3000:]
    lines = [ln for ln in r.stdout.strip().splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
                "scaling", "vs_baseline", "dtype", "data", "config", "roofline", "e2e", "gpu_launches", "clocks",
                "kernels", "full_search"):
        assert key in d, key
    assert d["steps"] == 4 and d["warmup"] == 3 and d["n_gpus"] == 1 and d["value"] > 0
    assert d["gpu_launches"] > 0 and d["config"]["workload"] == "tiny"
    assert d["roofline"]["bound"] == "tensor" and d["roofline"]["achieved"] > 0
    assert d["e2e"]["value"] > 0 and d["e2e"]["h2d_bytes_per_step"] > 0 and d["e2e"]["d2h_bytes_per_step"] > 0
    f = d["full_search"]
    assert f["T"] == d["config"]["T"] and f["value"] > 0 and 0 < f["computed_fraction"] <= 1
    assert f["cache_update"]["launches"] > 0 and f["unit"] == d["unit"]
    cases = d["cache_alone"]["cases"]
    assert [(c["N"], c["latent"]) for c in cases[:4]] == [(16, "16x21x60x104")] * 2 + [(32, "16x9x60x104")] * 2
    assert all(c["gbs"] > 0 and 0 <= c["skipped"] <= c["N"] for c in cases)


@pytest.mark.gpu
@pytest.mark.parametrize("extra", [["--search", "pruned"], ["--search", "static"], ["--search", "commit"],
                                   ["--search", "cfg"], ["--mask", "paper-density"], ["--tau", "0"]])
def test_bench_search_modes_on_the_tiny_workload(extra):
    """Every search mode the bench can time runs through its own arm and prints one line."""
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--config", "tiny", "--steps", "10",
                        "--warmup", "3", "--no-cpu-baseline", "--no-cache-alone", *extra],
                       capture_output=True, text=True, timeout=900, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-3000:]
    lines = [ln for ln in r.stdout.strip().splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["value"] > 0 and d["gpu_launches"] > 0 and 0 < d["computed_fraction"] <= 1
    assert d["full_search"]["value"] > 0
    if "--search" in extra:
        assert d["config"]["search"] == extra[1]
    if extra == ["--search", "commit"]:
        assert d["config"]["N"] == 1 and d["computed_fraction"] == 1.0
    if extra == ["--tau", "0"]:
        assert d["computed_fraction"] == 1.0
