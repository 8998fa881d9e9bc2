"""Seeded synthetic inputs for the cached-search denoising step.

This module is the only code shared by the CUDA path's callers (tests, bench,
smoke) and the CPU oracle.  It draws random numbers and lays them out; it holds
none of the method's arithmetic (no model, no cache rule, no sampler).

Recipe (every draw is a numpy ``Philox`` stream, key = the seed named below):

* DiT weights: Xavier-uniform, ``U(-a, a)`` with ``a = sqrt(6 / (fan_in + fan_out))``
  in float32.  By default each is rounded to the nearest bf16 value (round-half-even),
  so that a bf16 device copy holds exactly the values the oracle sees and a parity
  difference measures the kernels alone; ``round_bf16=False`` keeps the float32 draws,
  which the library then rounds itself (parity then includes the weight rounding).
  Biases and the per-block modulation offsets are 0.  One stream per parameter
  tensor, keyed ``(42, tensor index)``.
* Initial noise ``x_1`` of candidate ``i``: ``N(0, 1)`` float32 from key ``i``
  (the paper draws each candidate's noise from a generator seeded with the
  candidate's seed, Sec. Reproducibility).
* Text context ``[Lt, d_text]``: ``N(0, 1)`` from key 7.
* Target latent ``y*``: ``N(0, 1)`` from key 11 (stands in for the verifier).
* Beam-refill perturbation of round ``r``, parent rank ``p``, child ``j``:
  ``N(0, 1)`` from key ``1_000_000 + 1000 r + 10 p + j``.
"""
from __future__ import annotations

from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, field
import os

import numpy as np

WEIGHT_SEED = 42
TEXT_SEED = 7
TARGET_SEED = 11


@dataclass(frozen=True)
class ModelConfig:
    """Shape of the DiT velocity model and its latent."""
    C: int            # latent channels
    F: int            # latent frames
    H: int            # latent height
    W: int            # latent width
    d: int            # model width
    heads: int        # attention heads
    ffn: int          # FFN hidden width
    blocks: int       # transformer blocks
    f_dim: int        # timestep sinusoid features
    d_text: int       # raw text-embedding width
    Lt: int           # text tokens

    @property
    def hd(self) -> int:
        return self.d // self.heads

    @property
    def P(self) -> int:           # features per 1x2x2 patch
        return self.C * 4

    @property
    def L(self) -> int:           # video tokens
        return self.F * (self.H // 2) * (self.W // 2)

    @property
    def D(self) -> int:           # latent elements per candidate
        return self.C * self.F * self.H * self.W


@dataclass(frozen=True)
class SearchConfig:
    name: str
    model: ModelConfig
    N: int
    T: int
    tau: float
    K_w: int
    K_c: int
    taus: tuple = field(default_factory=tuple)
    beam_every: int = 0      # re-score cadence (0: best-of-N only)
    beam_keep: int = 0
    beam_children: int = 0
    beam_sigma: float = 0.0


TINY = ModelConfig(C=4, F=3, H=8, W=8, d=128, heads=4, ffn=512, blocks=2,
                   f_dim=64, d_text=128, Lt=16)
WAN_1_3B = ModelConfig(C=16, F=21, H=60, W=104, d=1536, heads=12, ffn=8960,
                       blocks=30, f_dim=256, d_text=4096, Lt=512)
# 33 frames at 480x832: latent 16 x 9 x 60 x 104, 14040 tokens after 1x2x2 patching
WAN_1_3B_SHORT = ModelConfig(C=16, F=9, H=60, W=104, d=1536, heads=12, ffn=8960,
                             blocks=30, f_dim=256, d_text=4096, Lt=512)
WAN_14B = ModelConfig(C=16, F=21, H=60, W=104, d=5120, heads=40, ffn=13824,
                      blocks=40, f_dim=256, d_text=4096, Lt=512)

CONFIGS = {
    "tiny": SearchConfig("tiny", TINY, N=4, T=10, tau=0.1, K_w=1, K_c=1),
    "wan1.3b-best-of-4": SearchConfig("wan1.3b-best-of-4", WAN_1_3B, N=4, T=50, tau=0.1,
                                      K_w=5, K_c=5, taus=(0.0, 0.05, 0.1, 0.2)),
    "wan1.3b-beam16": SearchConfig("wan1.3b-beam16", WAN_1_3B, N=16, T=50, tau=0.1, K_w=5,
                                   K_c=5, beam_every=10, beam_keep=4, beam_children=3,
                                   beam_sigma=0.1),
    "wan1.3b-short32": SearchConfig("wan1.3b-short32", WAN_1_3B_SHORT, N=32, T=30, tau=0.15,
                                    K_w=3, K_c=3),
    "wan14b-best-of-4": SearchConfig("wan14b-best-of-4", WAN_14B, N=4, T=50, tau=0.1,
                                     K_w=5, K_c=5),
}


def replace_model(m: ModelConfig, **kw) -> ModelConfig:
    """A copy of ``m`` with some fields changed (e.g. fewer blocks)."""
    d = dict(m.__dict__)
    d.update(kw)
    return ModelConfig(**d)


# ---------------------------------------------------------------------------
# parameter layout: (name, shape, kind) in the order of the flat buffer the C ABI
# takes (``cs_load_weights``).  kind: "w" Xavier weight, "b" zero bias/offset.
# Linear layers follow y = x W^T + b with W stored [out, in].
# ---------------------------------------------------------------------------

def param_layout(m: ModelConfig):
    d, P, F = m.d, m.P, m.ffn
    lay = [
        ("patch_w", (d, P), "w"), ("patch_b", (d,), "b"),
        ("time_w1", (d, m.f_dim), "w"), ("time_b1", (d,), "b"),
        ("time_w2", (d, d), "w"), ("time_b2", (d,), "b"),
        ("mod_w", (6 * d, d), "w"), ("mod_b", (6 * d,), "b"),
        ("text_w1", (d, m.d_text), "w"), ("text_b1", (d,), "b"),
        ("text_w2", (d, d), "w"), ("text_b2", (d,), "b"),
        ("head_mod_w", (2 * d, d), "w"), ("head_mod_b", (2 * d,), "b"),
        ("head_w", (P, d), "w"), ("head_b", (P,), "b"),
    ]
    for b in range(m.blocks):
        lay += [
            (f"blk{b}.mod_off", (6, d), "b"),
            (f"blk{b}.qkv_w", (3 * d, d), "w"), (f"blk{b}.qkv_b", (3 * d,), "b"),
            (f"blk{b}.o_w", (d, d), "w"), (f"blk{b}.o_b", (d,), "b"),
            (f"blk{b}.cq_w", (d, d), "w"), (f"blk{b}.cq_b", (d,), "b"),
            (f"blk{b}.ckv_w", (2 * d, d), "w"), (f"blk{b}.ckv_b", (2 * d,), "b"),
            (f"blk{b}.co_w", (d, d), "w"), (f"blk{b}.co_b", (d,), "b"),
            (f"blk{b}.ff1_w", (F, d), "w"), (f"blk{b}.ff1_b", (F,), "b"),
            (f"blk{b}.ff2_w", (d, F), "w"), (f"blk{b}.ff2_b", (d,), "b"),
        ]
    return lay


def param_count(m: ModelConfig) -> int:
    return int(sum(np.prod(s) for _, s, _ in param_layout(m)))


def round_to_bf16(a: np.ndarray) -> np.ndarray:
    """Nearest bf16 value (ties to even) of each float32, kept as float32."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32)
    u = (u + (np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1)))) & np.uint32(0xFFFF0000)
    return u.view(np.float32)


def _one_param(idx: int, shape, kind: str, seed: int, out: np.ndarray, round_bf16: bool = True):
    if kind == "b":
        out[...] = 0.0
        return
    fan_out, fan_in = shape
    a = np.float32(np.sqrt(6.0 / (fan_in + fan_out)))
    g = np.random.Generator(np.random.Philox(key=[seed, idx]))
    u = g.random(out.size, dtype=np.float32)
    w = (u * np.float32(2.0) - np.float32(1.0)) * a
    out[...] = (round_to_bf16(w) if round_bf16 else w).reshape(shape)


def make_params(m: ModelConfig, seed: int = WEIGHT_SEED, threads: int | None = None, round_bf16: bool = True):
    """All DiT parameters as (flat float32 buffer, {name: view into it}); weights rounded
    to bf16 values unless ``round_bf16`` is False."""
    lay = param_layout(m)
    flat = np.empty(param_count(m), dtype=np.float32)
    views, off = {}, 0
    for name, shape, _ in lay:
        n = int(np.prod(shape))
        views[name] = flat[off:off + n].reshape(shape)
        off += n
    jobs = [(i, s, k, views[n]) for i, (n, s, k) in enumerate(lay)]
    nthr = threads or min(16, os.cpu_count() or 1)
    with ThreadPoolExecutor(nthr) as ex:
        list(ex.map(lambda j: _one_param(j[0], j[1], j[2], seed, j[3], round_bf16), jobs))
    return flat, views


def iter_params(m: ModelConfig, seed: int = WEIGHT_SEED, threads: int | None = None, window: int = 32):
    """Yield (tensor index, float32 array) in layout order, the same values as
    :func:`make_params`, generated a bounded window of tensors ahead on a thread pool."""
    lay = param_layout(m)
    nthr = threads or min(16, os.cpu_count() or 1)

    def gen(i):
        name, shape, kind = lay[i]
        out = np.empty(shape, dtype=np.float32)
        _one_param(i, shape, kind, seed, out)
        return out

    with ThreadPoolExecutor(nthr) as ex:
        futs = {}
        for i in range(len(lay)):
            for j in range(i, min(len(lay), i + window)):
                if j not in futs:
                    futs[j] = ex.submit(gen, j)
            yield i, futs.pop(i).result()


def normal(seed: int, shape) -> np.ndarray:
    g = np.random.Generator(np.random.Philox(key=seed))
    return g.standard_normal(int(np.prod(shape)), dtype=np.float32).reshape(shape)


def initial_noise(m: ModelConfig, seeds) -> np.ndarray:
    """``x_1`` for each seed, [N, C, F, H, W] float32."""
    return np.stack([normal(int(s), (m.C, m.F, m.H, m.W)) for s in seeds])


def text_context(m: ModelConfig) -> np.ndarray:
    return normal(TEXT_SEED, (m.Lt, m.d_text))


def target_latent(m: ModelConfig) -> np.ndarray:
    return normal(TARGET_SEED, (m.C, m.F, m.H, m.W))


def beam_noise_seed(round_idx: int, parent_rank: int, child: int) -> int:
    return 1_000_000 + 1000 * round_idx + 10 * parent_rank + child


def beam_noise(m: ModelConfig, round_idx: int, keep: int, children: int) -> np.ndarray:
    """Perturbations for every child of one refill, [keep*children, C, F, H, W]."""
    return np.stack([normal(beam_noise_seed(round_idx, p, j), (m.C, m.F, m.H, m.W))
                     for p in range(keep) for j in range(children)])


def uniform(seed: int, shape, lo=-1.0, hi=1.0) -> np.ndarray:
    g = np.random.Generator(np.random.Philox(key=seed))
    return (g.random(int(np.prod(shape)), dtype=np.float32) * np.float32(hi - lo)
            + np.float32(lo)).reshape(shape)
