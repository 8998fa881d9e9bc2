"""Host-side checks of the C-ABI library (no GPU needed): it loads, exports every
symbol the public headers declare, and its host-only queries agree with the layout
the input generator uses."""
import os
import re

import pytest

from paper_2607_23159_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    names = set()
    for h in os.listdir(os.path.join(ROOT, "include")):
        src = open(os.path.join(ROOT, "include", h)).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        names |= set(re.findall(r"^[A-Za-z_][\w \*]*?\b(cs_\w+)\s*\(", src, flags=re.M))
    return names


@pytest.fixture(scope="module")
def b():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_23159_gb300 import binding
    return binding


def test_exports_every_declared_symbol(b):
    decl = _declared()
    assert len(decl) >= 20
    missing = [n for n in decl if not hasattr(b.lib, n)]
    assert not missing, missing
    assert decl <= set(b.EXPORTED) | {"cs_last_error"}


def test_param_count_matches_generator_layout(b):
    for m in (synth.TINY, synth.WAN_1_3B, synth.WAN_14B):
        assert b.param_count(m) == synth.param_count(m)


def test_workspace_and_version(b):
    assert b.lib.cs_version().startswith(b"cachedsearch")
    # the default library has no index checks (that is lib/libcachedsearch_debug.so)
    assert b.lib.cs_build_flags() == (1 if os.environ.get("CS_LIBRARY_VARIANT") == "debug" else 0)
    # partials (drift, score), then the single-pass step's arrival counter and skipped list [N + 1]
    assert b.cache_workspace_bytes(4, 2096640) == 4 * 256 * 12 + 4 + 5 * 4 + 256
    assert b.cache_workspace_bytes(0, 10) == 0


def test_invalid_config_rejected_on_host(b):
    import ctypes as C
    cfg = b.model_config(synth.replace_model(synth.TINY, H=7), 4)   # odd height: no 1x2x2 patches
    h = C.c_void_p()
    st = b.lib.cs_init_model(C.byref(cfg), C.byref(h))
    assert st == b.CS_ERR_ARG and not h.value
    assert "invalid" in b.last_error()
    cfg = b.model_config(synth.replace_model(synth.TINY, heads=2), 4)   # head dim 64
    assert b.lib.cs_init_model(C.byref(cfg), C.byref(h)) == b.CS_ERR_UNSUPPORTED


def test_streamed_generator_matches_flat_layout(b):
    import ctypes as C
    import numpy as np
    m = synth.replace_model(synth.TINY, blocks=3)
    flat, _ = synth.make_params(m)
    parts = list(synth.iter_params(m, threads=3, window=4))
    assert [i for i, _ in parts] == list(range(len(parts)))
    assert len(parts) == b.lib.cs_param_tensor_count(C.byref(b.model_config(m, 1)))
    assert np.array_equal(np.concatenate([a.reshape(-1) for _, a in parts]), flat)


def test_failure_selftest_rejects_a_null_error_word_on_the_host(b):
    st = b.lib.cs_selftest_bounded_wait(None, None)   # checked before any launch
    assert st == b.CS_ERR_ARG and "null" in b.last_error()


def test_index_checking_build_reports_its_flag():
    """The --debug build variant compiles (cross-compiled here, no GPU needed), lands at its
    own path and reports bit 0 of cs_build_flags; the default library does not."""
    import subprocess
    import sys
    from paper_2607_23159_gb300 import build as bld
    path = bld.build(debug=True)
    assert path.endswith("libcachedsearch_debug.so") and os.path.exists(path)
    code = ("import ctypes, sys; lib = ctypes.CDLL(sys.argv[1]); print(lib.cs_build_flags())")
    out = subprocess.run([sys.executable, "-c", code, path], capture_output=True, text=True, timeout=120)
    assert out.returncode == 0, out.stderr
    assert out.stdout.strip() == "1"


_NOT_STATUS = {"cs_build_flags", "cs_param_tensor_count", "cs_destroy_model"}


def test_every_entry_point_rejects_empty_arguments_on_the_host(b):
    """Every call that returns a cs_status checks its pointers and sizes before any device
    work: with null pointers and zero sizes it returns CS_ERR_ARG and leaves a message
    (no GPU is touched, so this runs here)."""
    import ctypes as C
    zero = {C.c_int: 0, C.c_longlong: 0, C.c_size_t: 0, C.c_float: 0.0, C.c_double: 0.0}
    checked = []
    for name, (res, args) in b._SIGS.items():
        if res is not C.c_int or name in _NOT_STATUS:
            continue
        call = [zero.get(a) for a in args]   # pointers of every kind -> None
        st = getattr(b.lib, name)(*call)
        assert st == b.CS_ERR_ARG, f"{name} returned {st}"
        assert b.last_error(), name
        checked.append(name)
    assert len(checked) >= 25
    # destroying a null model is a no-op, like free(NULL)
    assert b.lib.cs_destroy_model(None) == b.CS_OK


def test_product_path_has_no_fallback():
    """The package never imports the oracle, and its binding refuses to import without
    the compiled library (no CPU or PyTorch fallback to fall back on)."""
    import subprocess
    import sys
    pkg = os.path.join(ROOT, "paper_2607_23159_gb300")
    for f in os.listdir(pkg):
        if f.endswith(".py"):
            src = open(os.path.join(pkg, f)).read()
            assert not re.search(r"^\s*(from|import)\s+oracle\b", src, flags=re.M), f
    code = ("import os, sys\n"
            "real = os.path.exists\n"
            "os.path.exists = lambda p: False if str(p).endswith('.so') else real(p)\n"
            "try:\n"
            "    import paper_2607_23159_gb300.binding\n"
            "except ImportError as e:\n"
            "    print('refused:', e)\n")
    out = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, cwd=ROOT, timeout=120)
    assert out.returncode == 0 and out.stdout.startswith("refused:") and "build" in out.stdout, out.stdout + out.stderr


def test_step_workspace_size_of_the_carried_form(b):
    """cs_cache_step_bytes: 0 for latents the token-layout update does not handle (odd H,
    W not a multiple of 4) and for N <= 0; otherwise it covers at least the carried sums
    (two float2 per candidate, by step parity), the unit and token-row partial pairs and
    the drift-pass partials, and grows with N."""
    from paper_2607_23159_gb300 import synth
    assert b.cache_step_bytes(4, 16, 21, 60, 102) == 0
    assert b.cache_step_bytes(4, 16, 21, 59, 104) == 0
    assert b.cache_step_bytes(0, 16, 21, 60, 104) == 0
    m = synth.WAN_1_3B
    units = -(-m.D // 4096)
    rows = m.F * m.H // 2
    chunks = -(-m.D // 8192)
    for N in (1, 4, 16):
        got = b.cache_step_bytes(N, m.C, m.F, m.H, m.W)
        assert got % 256 == 0
        assert got >= N * (2 * 8 + max(units, rows) * 8 + chunks * 8 + units * 4 + rows * 4)
    assert b.cache_step_bytes(16, m.C, m.F, m.H, m.W) > b.cache_step_bytes(4, m.C, m.F, m.H, m.W)
    t = synth.TINY
    assert b.cache_step_bytes(4, t.C, t.F, t.H, t.W) > 0
