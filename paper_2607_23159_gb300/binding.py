"""Thin ctypes binding of ``libcachedsearch.so`` (argument marshalling only).

Every computation happens in the library's CUDA kernels; this module turns torch
tensors into raw pointers and sizes, passes the current CUDA stream, and raises
:class:`CSError` on a non-zero status.  There is no fallback: if the library is not
built, importing this module raises.
"""
from __future__ import annotations

import ctypes as C
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
# CS_LIBRARY_VARIANT=debug selects the build with device-side index checks
# (`python -m paper_2607_23159_gb300.build --debug`); anything else the normal build
_VARIANT = os.environ.get("CS_LIBRARY_VARIANT", "release")
LIB_PATH = os.path.join(_HERE, "lib", "libcachedsearch_debug.so" if _VARIANT == "debug" else "libcachedsearch.so")

if not os.path.exists(LIB_PATH):
    raise ImportError(f"{LIB_PATH} is missing: build it with `python -m paper_2607_23159_gb300.build"
                      f"{' --debug' if _VARIANT == 'debug' else ''}` (or __graft_entry__.build())")
lib = C.CDLL(LIB_PATH)

(CS_OK, CS_ERR_ARG, CS_ERR_CUDA, CS_ERR_NONFINITE, CS_ERR_TIMEOUT, CS_ERR_NOMEM, CS_ERR_UNSUPPORTED,
 CS_ERR_BOUNDS) = range(8)
EPI_F32, EPI_BF16, EPI_GELU_BF16, EPI_RESID_F32, EPI_QKV = range(5)
KC_SELF_ATTN, KC_CROSS_ATTN, KC_GEMM, KC_CACHE, KC_OTHER = range(5)


class CSError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__(f"cachedsearch status {status}: {msg}")
        self.status = status


class ModelConfig(C.Structure):
    _fields_ = [(n, C.c_int) for n in
                ("C", "F", "H", "W", "d", "heads", "ffn", "blocks", "f_dim", "d_text", "Lt", "max_batch")]


P, I, LL, F, D, SZ = C.c_void_p, C.c_int, C.c_longlong, C.c_float, C.c_double, C.c_size_t

_SIGS = {
    "cs_selftest_bounded_wait": (I, [P, P]),
    "cs_last_error": (C.c_char_p, []),
    "cs_version": (C.c_char_p, []),
    "cs_build_flags": (I, []),
    "cs_param_count": (SZ, [C.POINTER(ModelConfig)]),
    "cs_init_model": (I, [C.POINTER(ModelConfig), C.POINTER(P)]),
    "cs_destroy_model": (I, [P]),
    "cs_load_weights": (I, [P, P, SZ, I, P]),
    "cs_param_tensor_count": (I, [C.POINTER(ModelConfig)]),
    "cs_load_param": (I, [P, I, P, SZ, I, P]),
    "cs_set_text_context": (I, [P, P, P]),
    "cs_set_null_text_context": (I, [P, P, P]),
    "cs_dit_forward": (I, [P, P, P, I, F, P, P]),
    "cs_cache_decide_cfg": (I, [P, P, P, P, I, LL, I, I, F, I, I, P, P, P, P, P, P, P]),
    "cs_cache_apply_cfg": (I, [P, P, P, P, P, I, LL, F, F, F, P, P, P, P]),
    "cs_search_step_cfg": (I, [P, P, P, P, P, P, I, I, I, F, F, F, I, I, F, P, P, P, P, P, P]),
    "cs_cache_workspace_bytes": (SZ, [I, LL]),
    "cs_cache_decide": (I, [P, P, P, P, I, LL, I, I, F, I, I, P, P, P, P, P, P, P]),
    "cs_cache_decide_noalloc": (I, [P, P, P, P, I, LL, I, I, F, I, I, P, P, P, P, P, P]),
    "cs_cache_apply": (I, [P, P, P, P, P, I, LL, F, F, P, P, P, P]),
    "cs_cache_decide_skip": (I, [P, P, P, P, P, I, LL, I, I, F, F, F, I, I, P, P, P, P, P, P, P, P]),
    "cs_cache_apply_computed": (I, [P, P, P, P, P, I, LL, F, F, P, P, P, P]),
    "cs_cache_apply_tokens": (I, [P, P, P, P, P, P, P, P, I, I, I, I, I, I, F, F, P, P, P, P, P, P]),
    "cs_cache_step_bytes": (SZ, [I, I, I, I, I]),
    "cs_cache_decide_skip_carry": (I, [P, P, P, P, P, I, I, I, I, I, I, I, F, F, F, I, I, P, P, P, P, P, I, P, P,
                                       P]),
    "cs_cache_apply_tokens_carry": (I, [P, P, P, P, P, P, P, P, I, I, I, I, I, I, I, F, F, P, P, P, P, P]),
    "cs_search_step": (I, [P, P, P, P, P, P, I, I, I, F, F, F, I, I, P, P, P, P, P, P]),
    "cs_search_step_host": (I, [P, P, P, P, P, P, I, I, I, F, F, F, I, I, P, P, P]),
    "cs_score": (I, [P, P, I, LL, P, P, P]),
    "cs_select_topk": (I, [P, I, I, P, P]),
    "cs_beam_refill": (I, [P, P, P, P, P, P, P, P, P, P, P, I, I, F, P, LL, P]),
    "cs_device_error": (I, [P, C.POINTER(I), P]),
    "cs_set_profiling": (I, [P, I]),
    "cs_kernel_stats": (I, [P, I, C.POINTER(LL), C.POINTER(D), C.POINTER(D)]),
    "cs_reset_kernel_stats": (I, [P]),
    "cs_launch_count": (LL, []),
    "cs_gemm_bf16": (I, [P, P, I, I, I, I, P, P, P, I, P, P]),
    "cs_gemm_qkv": (I, [P, P, I, I, I, P, I, I, I, I, P, P, P, I, P, P]),
    "cs_attention": (I, [P, P, P, P, I, I, I, I, I, I, I, P, P]),
    "cs_layernorm_modulate": (I, [P, P, P, P, I, I, P]),
}
for _name, (_res, _args) in _SIGS.items():
    _f = getattr(lib, _name)
    _f.restype = _res
    _f.argtypes = _args

EXPORTED = tuple(_SIGS)


def last_error() -> str:
    return lib.cs_last_error().decode()


def check(status: int):
    if status != CS_OK:
        raise CSError(status, last_error())


def launch_count() -> int:
    return int(lib.cs_launch_count())


def index_checks() -> bool:
    """True when the loaded library is the build with device-side index checks."""
    return bool(lib.cs_build_flags() & 1)


# ---------------------------------------------------------------- helpers --

def _ptr(t):
    """Raw pointer of a torch tensor / numpy array / None."""
    if t is None:
        return None
    if isinstance(t, np.ndarray):
        return t.ctypes.data
    return t.data_ptr()


def _stream(stream=None):
    import torch
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


def model_config(m, max_batch: int) -> ModelConfig:
    return ModelConfig(m.C, m.F, m.H, m.W, m.d, m.heads, m.ffn, m.blocks, m.f_dim, m.d_text, m.Lt, max_batch)


def param_count(m) -> int:
    cfg = model_config(m, 1)
    return int(lib.cs_param_count(C.byref(cfg)))


def cache_workspace_bytes(N: int, D: int) -> int:
    return int(lib.cs_cache_workspace_bytes(N, D))


# ------------------------------------------------------------- kernel ops --

def gemm(A, B, epi, out, bias=None, gate=None, err=None, stream=None):
    M, K = A.shape
    N = B.shape[0]
    check(lib.cs_gemm_bf16(_ptr(A), _ptr(B), M, N, K, epi, _ptr(bias), _ptr(gate), _ptr(out), out.shape[1],
                           _ptr(err), _stream(stream)))


def gemm_qkv(A, B, bias, L, d, heads, which_base, q, k, vt, Lv, err=None, stream=None):
    M, K = A.shape
    N = B.shape[0]
    check(lib.cs_gemm_qkv(_ptr(A), _ptr(B), M, N, K, _ptr(bias), L, d, heads, which_base, _ptr(q), _ptr(k),
                          _ptr(vt), Lv, _ptr(err), _stream(stream)))


def attention(q, k, vt, o, B, heads, Lq, Lk, hd, Lkv_stride, kv_shared, err=None, stream=None):
    check(lib.cs_attention(_ptr(q), _ptr(k), _ptr(vt), _ptr(o), B, heads, Lq, Lk, hd, Lkv_stride, int(kv_shared),
                           _ptr(err), _stream(stream)))


def layernorm_modulate(x, shift, scale, out, stream=None):
    M, d = x.shape
    check(lib.cs_layernorm_modulate(_ptr(x), _ptr(shift), _ptr(scale), _ptr(out), M, d, _stream(stream)))


def cache_decide(x, x_ref, accum, has_ref, step_k, T, tau, K_w, K_c, skip_mask, compute_idx, n_compute, workspace,
                 force=None, err=None, stream=None):
    N = x.shape[0]
    Dn = x[0].numel()
    check(lib.cs_cache_decide(_ptr(x), _ptr(x_ref), _ptr(accum), _ptr(has_ref), N, Dn, step_k, T, tau, K_w, K_c,
                              _ptr(force), _ptr(skip_mask), _ptr(compute_idx), _ptr(n_compute), _ptr(workspace),
                              _ptr(err), _stream(stream)))


def cache_decide_noalloc(x, x_ref, accum, has_ref, step_k, T, tau, K_w, K_c, skip_mask, compute_idx, n_compute,
                         force=None, err=None, stream=None):
    """cs_cache_decide without a workspace (fixed scratch inside the library)."""
    N = x.shape[0]
    Dn = x[0].numel()
    check(lib.cs_cache_decide_noalloc(_ptr(x), _ptr(x_ref), _ptr(accum), _ptr(has_ref), N, Dn, step_k, T, tau, K_w,
                                      K_c, _ptr(force), _ptr(skip_mask), _ptr(compute_idx), _ptr(n_compute),
                                      _ptr(err), _stream(stream)))


def cache_apply_tokens(st, skip_mask, hout, compute_idx, n_c, C, F, H, W, t_cur, t_next, workspace=None,
                       target=None, scores=None, tile_partials=None, err=None, stream=None):
    """cs_cache_apply_tokens: the computed candidates' update from the head's token output
    ``hout`` [n_c * L, 4C] (state dict ``st`` as from :func:`new_state`)."""
    N = st["x"].shape[0]
    check(lib.cs_cache_apply_tokens(_ptr(st["x"]), _ptr(st["x_ref"]), _ptr(st["delta"]), _ptr(st["accum"]),
                                    _ptr(st["has_ref"]), _ptr(skip_mask), _ptr(hout), _ptr(compute_idx), n_c, N, C,
                                    F, H, W, t_cur, t_next, _ptr(target), _ptr(scores), _ptr(workspace),
                                    _ptr(tile_partials), _ptr(err), _stream(stream)))


def cache_step_bytes(N: int, C: int, F: int, H: int, W: int) -> int:
    return int(lib.cs_cache_step_bytes(N, C, F, H, W))


def cache_decide_skip_carry(st, lat, step_k, T, t_cur, t_next, tau, K_w, K_c, skip_mask, compute_idx, n_compute,
                            step_ws, carried, force=None, target=None, err=None, stream=None):
    """cs_cache_decide_skip_carry on state dict ``st``; ``lat`` = (C, F, H, W)."""
    N = st["x"].shape[0]
    C_, F_, H_, W_ = lat
    check(lib.cs_cache_decide_skip_carry(_ptr(st["x"]), _ptr(st["x_ref"]), _ptr(st["delta"]), _ptr(st["accum"]),
                                         _ptr(st["has_ref"]), N, C_, F_, H_, W_, step_k, T, t_cur, t_next, tau, K_w,
                                         K_c, _ptr(force), _ptr(skip_mask), _ptr(compute_idx), _ptr(n_compute),
                                         _ptr(target), 1 if carried else 0, _ptr(step_ws), _ptr(err),
                                         _stream(stream)))


def cache_apply_tokens_carry(st, skip_mask, hout, compute_idx, n_c, lat, step_k, t_cur, t_next, step_ws,
                             target=None, scores=None, err=None, stream=None):
    """cs_cache_apply_tokens_carry: the computed update that also leaves the next step's drift."""
    N = st["x"].shape[0]
    C_, F_, H_, W_ = lat
    check(lib.cs_cache_apply_tokens_carry(_ptr(st["x"]), _ptr(st["x_ref"]), _ptr(st["delta"]), _ptr(st["accum"]),
                                          _ptr(st["has_ref"]), _ptr(skip_mask), _ptr(hout), _ptr(compute_idx), n_c,
                                          N, C_, F_, H_, W_, step_k, t_cur, t_next, _ptr(target), _ptr(scores),
                                          _ptr(step_ws), _ptr(err), _stream(stream)))


def cache_apply(x, x_ref, delta, v, skip_mask, t_cur, t_next, workspace=None, target=None, scores=None,
                stream=None):
    N = x.shape[0]
    Dn = x[0].numel()
    check(lib.cs_cache_apply(_ptr(x), _ptr(x_ref), _ptr(delta), _ptr(v), _ptr(skip_mask), N, Dn, t_cur, t_next,
                             _ptr(target), _ptr(scores), _ptr(workspace), _stream(stream)))


def cache_decide_skip(x, x_ref, delta, accum, has_ref, step_k, T, t_cur, t_next, tau, K_w, K_c, skip_mask,
                      compute_idx, n_compute, workspace, force=None, target=None, err=None, stream=None):
    N = x.shape[0]
    check(lib.cs_cache_decide_skip(_ptr(x), _ptr(x_ref), _ptr(delta), _ptr(accum), _ptr(has_ref), N, x[0].numel(),
                                   step_k, T, t_cur, t_next, tau, K_w, K_c, _ptr(force), _ptr(skip_mask),
                                   _ptr(compute_idx), _ptr(n_compute), _ptr(target), _ptr(workspace), _ptr(err),
                                   _stream(stream)))


def cache_apply_computed(x, x_ref, delta, v, skip_mask, t_cur, t_next, workspace=None, target=None, scores=None,
                         stream=None):
    N = x.shape[0]
    check(lib.cs_cache_apply_computed(_ptr(x), _ptr(x_ref), _ptr(delta), _ptr(v), _ptr(skip_mask), N,
                                      x[0].numel(), t_cur, t_next, _ptr(target), _ptr(scores), _ptr(workspace),
                                      _stream(stream)))


def score(x, target, scores, workspace, stream=None):
    N = x.shape[0]
    check(lib.cs_score(_ptr(x), _ptr(target), N, x[0].numel(), _ptr(scores), _ptr(workspace), _stream(stream)))


def select_topk(scores, k, idx, stream=None):
    check(lib.cs_select_topk(_ptr(scores), scores.numel(), k, _ptr(idx), _stream(stream)))


def beam_refill(src, dst, survivors, children, sigma, noise, stream=None):
    """src/dst: dicts with x, x_ref, delta, accum, has_ref tensors."""
    keep = survivors.numel()
    Dn = src["x"][0].numel()
    check(lib.cs_beam_refill(_ptr(src["x"]), _ptr(src["x_ref"]), _ptr(src["delta"]), _ptr(src["accum"]),
                             _ptr(src["has_ref"]), _ptr(dst["x"]), _ptr(dst["x_ref"]), _ptr(dst["delta"]),
                             _ptr(dst["accum"]), _ptr(dst["has_ref"]), _ptr(survivors), keep, children, sigma,
                             _ptr(noise), Dn, _stream(stream)))


# ------------------------------------------------------------------ model --

class Model:
    """Owner of a ``cs_model*`` (device weights + workspace for ``max_batch`` candidates)."""

    def __init__(self, mcfg, max_batch: int):
        self.mcfg = mcfg
        self.max_batch = max_batch
        self._cfg = model_config(mcfg, max_batch)
        h = C.c_void_p()
        check(lib.cs_init_model(C.byref(self._cfg), C.byref(h)))
        self.h = h

    def close(self):
        if self.h:
            lib.cs_destroy_model(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def load_weights(self, flat, stream=None):
        """flat: float32 numpy array (host) or torch CUDA tensor in the cs_param_count layout."""
        on_dev = not isinstance(flat, np.ndarray)
        if not on_dev:
            flat = np.ascontiguousarray(flat, dtype=np.float32)
        check(lib.cs_load_weights(self.h, _ptr(flat), flat.size if not on_dev else flat.numel(), int(on_dev),
                                  _stream(stream)))

    def load_param(self, index, arr, stream=None):
        """One tensor of the layout (numpy float32, host)."""
        arr = np.ascontiguousarray(arr, dtype=np.float32)
        check(lib.cs_load_param(self.h, index, _ptr(arr), arr.size, 0, _stream(stream)))

    def load_streamed(self, seed=None, threads=None):
        """Generate the seeded synthetic parameters tensor by tensor and load each."""
        from . import synth
        for i, arr in synth.iter_params(self.mcfg, **({} if seed is None else {"seed": seed}), threads=threads):
            self.load_param(i, arr)

    def set_text_context(self, ctx, stream=None):
        check(lib.cs_set_text_context(self.h, _ptr(ctx), _stream(stream)))

    def set_null_text_context(self, ctx, stream=None):
        check(lib.cs_set_null_text_context(self.h, _ptr(ctx), _stream(stream)))

    def search_step_cfg(self, st, k, T, t_cur, t_next, tau, K_w, K_c, w, skip_mask, force=None, target=None,
                        scores=None, stream=None) -> int:
        """Guided step; st from new_state_cfg (x [N, D], branch states [2N, ...])."""
        n = C.c_int(0)
        N = st["x"].shape[0]
        check(lib.cs_search_step_cfg(self.h, _ptr(st["x"]), _ptr(st["x_ref"]), _ptr(st["delta"]),
                                     _ptr(st["accum"]), _ptr(st["has_ref"]), N, k, T, t_cur, t_next, tau, K_w, K_c,
                                     w, _ptr(force), _ptr(skip_mask), _ptr(target), _ptr(scores), C.byref(n),
                                     _stream(stream)))
        return n.value

    def dit_forward(self, x, idx, n_c, t, v, stream=None):
        check(lib.cs_dit_forward(self.h, _ptr(x), _ptr(idx), n_c, t, _ptr(v), _stream(stream)))

    def search_step(self, st, k, T, t_cur, t_next, tau, K_w, K_c, skip_mask, force=None, target=None, scores=None,
                    stream=None) -> int:
        """st: dict of device tensors x, x_ref, delta, accum, has_ref.  Returns n_computed."""
        n = C.c_int(0)
        N = st["x"].shape[0]
        check(lib.cs_search_step(self.h, _ptr(st["x"]), _ptr(st["x_ref"]), _ptr(st["delta"]), _ptr(st["accum"]),
                                 _ptr(st["has_ref"]), N, k, T, t_cur, t_next, tau, K_w, K_c, _ptr(force),
                                 _ptr(skip_mask), _ptr(target), _ptr(scores), C.byref(n), _stream(stream)))
        return n.value

    def search_step_host(self, x_host, st, k, T, t_cur, t_next, tau, K_w, K_c, skip_host, stream=None) -> int:
        n = C.c_int(0)
        N = x_host.shape[0]
        check(lib.cs_search_step_host(self.h, _ptr(x_host), _ptr(st["x_ref"]), _ptr(st["delta"]),
                                      _ptr(st["accum"]), _ptr(st["has_ref"]), N, k, T, t_cur, t_next, tau, K_w,
                                      K_c, _ptr(skip_host), C.byref(n), _stream(stream)))
        return n.value

    def device_error(self, stream=None) -> int:
        code = C.c_int(0)
        check(lib.cs_device_error(self.h, C.byref(code), _stream(stream)))
        return code.value

    def set_profiling(self, on: bool):
        check(lib.cs_set_profiling(self.h, int(on)))

    def kernel_stats(self, cls: int):
        n, ms, work = C.c_longlong(0), C.c_double(0), C.c_double(0)
        check(lib.cs_kernel_stats(self.h, cls, C.byref(n), C.byref(ms), C.byref(work)))
        return n.value, ms.value, work.value

    def reset_kernel_stats(self):
        check(lib.cs_reset_kernel_stats(self.h))


def new_state_cfg(N: int, D: int, device="cuda"):
    """Zeroed guided-search state: latents [N, D]; two branch cache states per candidate
    (rows i and N + i)."""
    import torch
    st = new_state(2 * N, D, device)
    st["x"] = torch.zeros(N, D, dtype=torch.float32, device=device)
    return st


def new_state(N: int, D: int, device="cuda"):
    """Zeroed cache state for a fresh search (has_ref = 0: every candidate computes first)."""
    import torch
    return {
        "x": torch.zeros(N, D, dtype=torch.float32, device=device),
        "x_ref": torch.zeros(N, D, dtype=torch.float32, device=device),
        "delta": torch.zeros(N, D, dtype=torch.float32, device=device),
        "accum": torch.zeros(N, dtype=torch.float32, device=device),
        "has_ref": torch.zeros(N, dtype=torch.uint8, device=device),
    }


def selftest_bounded_wait(err, stream=None):
    """Queue the failure-path self-test: a bounded wait that nothing satisfies; after
    ~2 s of GPU time err[0] holds CS_ERR_TIMEOUT."""
    check(lib.cs_selftest_bounded_wait(_ptr(err), _stream(stream)))
