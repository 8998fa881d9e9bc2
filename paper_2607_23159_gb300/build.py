"""Build the C-ABI library ``lib/libcachedsearch.so`` from ``csrc/*.cu`` for sm_103a.

Each translation unit compiles in parallel with nvcc; the objects link into one shared
library with no dependency on torch.  Run ``python -m paper_2607_23159_gb300.build``.
``--debug`` builds ``lib/libcachedsearch_debug.so`` with CS_DEBUG_CHECKS (device-side
index checks; see cs_build_flags in include/cachedsearch.h); the binding loads it when
the environment sets CS_LIBRARY_VARIANT=debug.
"""
from __future__ import annotations

import fcntl
import os
import shutil
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
LIB_DIR = os.path.join(HERE, "lib")
VARIANTS = {   # name -> (object directory, library, extra nvcc flags)
    "release": (os.path.join(HERE, "_build"), os.path.join(LIB_DIR, "libcachedsearch.so"), []),
    "debug": (os.path.join(HERE, "_build_debug"), os.path.join(LIB_DIR, "libcachedsearch_debug.so"),
              ["-DCS_DEBUG_CHECKS"]),
}
BUILD, LIB, _ = VARIANTS["release"]

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "--expt-relaxed-constexpr",
         "-I", os.path.join(ROOT, "include")]


def nvcc() -> str:
    for c in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if c and os.path.exists(c):
            return c
    raise RuntimeError("nvcc not found")


def sources():
    return sorted(os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith(".cu"))


def _compile(src: str, build_dir: str, extra) -> str:
    obj = os.path.join(build_dir, os.path.basename(src)[:-3] + ".o")
    cmd = [nvcc(), *ARCH, *FLAGS, *extra, "-c", src, "-o", obj]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc failed on {os.path.basename(src)}:\n{r.stdout}\n{r.stderr}")
    return obj


def build(verbose_ptxas: bool = False, force: bool = False, debug: bool = False) -> str:
    """Compile every kernel source and link the library (the index-checking variant
    with ``debug``); returns its path.  Processes that build at the same time (one per
    GPU rank) take turns on a lock file, so the later ones find the library up to date."""
    build_dir, lib, flags = VARIANTS["debug" if debug else "release"]
    os.makedirs(build_dir, exist_ok=True)
    os.makedirs(LIB_DIR, exist_ok=True)
    with open(os.path.join(build_dir, ".lock"), "w") as lock:
        fcntl.flock(lock, fcntl.LOCK_EX)
        try:
            return _build_locked(verbose_ptxas, force, build_dir, lib, flags)
        finally:
            fcntl.flock(lock, fcntl.LOCK_UN)


def _build_locked(verbose_ptxas: bool, force: bool, build_dir: str, lib: str, flags) -> str:
    srcs = sources()
    headers = [os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith((".cuh", ".h"))]
    headers += [os.path.join(ROOT, "include", f) for f in os.listdir(os.path.join(ROOT, "include"))]
    if not force and os.path.exists(lib):
        t = os.path.getmtime(lib)
        if all(os.path.getmtime(p) < t for p in srcs + headers + [__file__]):
            return lib
    extra = list(flags) + (["-Xptxas", "-v"] if verbose_ptxas else [])
    with ThreadPoolExecutor(max(1, min(len(srcs), os.cpu_count() or 1))) as ex:
        objs = list(ex.map(lambda s: _compile(s, build_dir, extra), srcs))
    tmp = lib + ".tmp"
    cmd = [nvcc(), *ARCH, "-shared", "-o", tmp, *objs, "-lcudart"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, lib)
    return lib


if __name__ == "__main__":
    print(build(verbose_ptxas="-v" in sys.argv, force="-f" in sys.argv, debug="--debug" in sys.argv))
