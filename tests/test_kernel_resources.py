"""Resource use of every kernel as ptxas reports it for sm_103a (CPU: nvcc cross-compiles).

No kernel spills registers to local memory: the bandwidth-bound kernels keep their loads in
registers and the tensor-core kernels keep their accumulator hand-offs there, and a spill
would put local-memory traffic on paths whose rooflines assume none.  The skip update of
the carried cache step runs one 288-thread CTA per SM, so its registers must also fit that
block on one SM.
"""
import os
import re
import shutil
import subprocess
import tempfile
from concurrent.futures import ThreadPoolExecutor

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2607_23159_gb300", "csrc")
NVCC = shutil.which("nvcc") or ("/usr/local/cuda/bin/nvcc" if os.path.exists("/usr/local/cuda/bin/nvcc") else None)
ENTRY = re.compile(r"Compiling entry function '([^']+)' for 'sm_103a'.*?(\d+) bytes spill stores, (\d+) bytes spill "
                   r"loads.*?Used (\d+) registers", re.S)


def _ptxas_report(src: str) -> str:
    with tempfile.TemporaryDirectory() as tmp:
        cmd = [NVCC, "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-std=c++17", "-Xcompiler", "-fPIC",
               "--expt-relaxed-constexpr", "-I", os.path.join(ROOT, "include"), "-Xptxas", "-v", "-c",
               os.path.join(CSRC, src), "-o", os.path.join(tmp, "k.o")]
        r = subprocess.run(cmd, capture_output=True, text=True, timeout=600)
        assert r.returncode == 0, r.stderr[-2000:]
        return r.stdout + r.stderr


@pytest.fixture(scope="module")
def kernels():
    if NVCC is None:
        pytest.skip("nvcc not available")
    sources = sorted(f for f in os.listdir(CSRC) if f.endswith(".cu"))
    with ThreadPoolExecutor(max_workers=len(sources)) as pool:
        reports = list(pool.map(_ptxas_report, sources))
    found = {}
    for src, rep in zip(sources, reports):
        for name, st, ld, regs in ENTRY.findall(rep):
            found[name] = (src, int(st), int(ld), int(regs))
    return found


def test_no_kernel_spills_registers(kernels):
    assert len(kernels) >= 40, sorted(kernels)
    spilling = {n: v for n, v in kernels.items() if v[1] or v[2]}
    assert not spilling, spilling


def test_carried_skip_update_fits_one_cta_per_sm(kernels):
    skip = {n: v for n, v in kernels.items() if "carry_skip_kernel" in n}
    assert len(skip) == 4, sorted(skip)            # <score, decide> in {0, 1}^2
    for name, (_, _, _, regs) in skip.items():
        assert 288 * regs <= 65536, (name, regs)
