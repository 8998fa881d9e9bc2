"""CPU oracle for the CachedSearch denoising step (arxiv 2607.23159).

TEST INFRASTRUCTURE, NOT PRODUCT CODE.  Only ``tests/``, ``__graft_entry__.smoke()``
and the CPU-baseline leg of ``bench.py`` may import this module.  It shares no
code with the CUDA path and imports nothing from it.

Plain, slow, float64 numpy, written from the paper:

* flow-matching Euler sampler on the grid ``1 = t_1 > ... > t_{T+1} = 0``  (Sec. 2, Eq. euler)
* transformation-vector cache ``Delta = v(x_ref) - x_ref``                   (Sec. 3.1, Eq. delta)
* skipped call returns ``x + Delta``                                         (Sec. 3.1, Eq. skip)
* accumulated relative drift ``a += ||x - x_ref||_F / ||x_ref||_F``; skip while
  ``a <= tau``; compute, refresh ``(Delta, x_ref)`` and reset ``a`` once ``a > tau``;
  warmup/cooldown windows and the empty cache always compute   (Sec. 3.1, Eq. indicator;
  App. Reproducibility, cache wrapper)
* CachedSearch: N cached rollouts, score, argmax                             (Algorithm 1)

The paper does not define the DiT block; the velocity model here is the block the
workload names (adaLN-modulated LayerNorm, full self-attention over video tokens,
cross-attention to a text context, GELU FFN).  Readings of points the paper leaves
open are stated where they are used.

Parity status: the cache rule, sampler, search and selection are pinned by closed
forms and invariants in ``tests/test_oracle_pins.py``; each DiT primitive is pinned
against textbook special cases, the block against an independent composition and the
forward by token-permutation invariants.  The conditioning MLPs (``DiT.modulation``:
timestep sinusoid to the six adaLN vectors per block and the head's two;
``DiT.text_kv``: text projection to per-block K/V) are pinned by closed-form values
through identity weights (SiLU at +-ln 3, the odd/even identities of GELU), by the
role each adaLN vector plays in the block and head, and by an independent torch.nn
composition.  The DiT forward as a whole has no printed value in the paper to pin
against (pinned per part and by invariants, not as a whole).
``tests/test_oracle_mutants.py`` checks that planted mistakes in the functions above
fail the pins.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

LN_EPS = 1e-6


# ---------------------------------------------------------------------------
# sampler (Sec. 2, Eq. euler)
# ---------------------------------------------------------------------------

def time_grid(T: int) -> np.ndarray:
    """``t_k = 1 - (k-1)/T`` for k = 1..T+1 (a decreasing grid from 1 to 0, Sec. 2)."""
    return 1.0 - np.arange(T + 1, dtype=np.float64) / T


def euler(x, t_cur, t_next, v):
    """``x_{t_{k+1}} = x_{t_k} + (t_{k+1} - t_k) v`` (Eq. euler)."""
    return x + (t_next - t_cur) * v


# ---------------------------------------------------------------------------
# DiT primitives
# ---------------------------------------------------------------------------

def linear(x, w, b):
    """``y = x W^T + b`` with ``W`` stored [out, in]."""
    return x @ np.asarray(w, np.float64).T + np.asarray(b, np.float64)


def layer_norm(x, eps=LN_EPS):
    """LayerNorm over the last axis, no affine: ``(x - mean) / sqrt(var + eps)``."""
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps)


def gelu_tanh(x):
    """GELU, tanh form (Hendrycks & Gimpel 2016): 0.5 x (1 + tanh(sqrt(2/pi)(x + 0.044715 x^3)))."""
    return 0.5 * x * (1.0 + np.tanh(np.sqrt(2.0 / np.pi) * (x + 0.044715 * x ** 3)))


def silu(x):
    return x / (1.0 + np.exp(-x))


def softmax_rows(s):
    s = s - s.max(axis=-1, keepdims=True)
    e = np.exp(s)
    return e / e.sum(axis=-1, keepdims=True)


def attention(q, k, v):
    """Scaled dot-product attention of one head, ``softmax(q k^T / sqrt(hd)) v``.

    q [Lq, hd], k [Lk, hd], v [Lk, hd]; no mask.  Rows are independent, so long
    query sets are taken a slab of rows at a time (the definition per row is unchanged).
    """
    hd = q.shape[-1]
    out = np.empty((q.shape[0], v.shape[1]), dtype=np.float64)
    step = max(1, int(2 ** 24 // max(1, k.shape[0])))
    for r0 in range(0, q.shape[0], step):
        s = (q[r0:r0 + step] @ k.T) / np.sqrt(hd)
        out[r0:r0 + step] = softmax_rows(s) @ v
    return out


def multi_head_attention(q, k, v, heads):
    """q [Lq, d], k/v [Lk, d]; heads are contiguous hd-wide column groups."""
    hd = q.shape[1] // heads
    return np.concatenate([attention(q[:, h * hd:(h + 1) * hd], k[:, h * hd:(h + 1) * hd],
                                     v[:, h * hd:(h + 1) * hd]) for h in range(heads)], axis=1)


def patchify(x):
    """[C, F, H, W] -> tokens [F * H/2 * W/2, C*4].

    Patch (1, 2, 2); tokens in (f, h/2, w/2) row-major order; inside a token the
    feature index is ``c*4 + ph*2 + pw``.
    """
    C, F, H, W = x.shape
    t = x.reshape(C, F, H // 2, 2, W // 2, 2).transpose(1, 2, 4, 0, 3, 5)
    return t.reshape(F * (H // 2) * (W // 2), C * 4)


def unpatchify(tok, C, F, H, W):
    """Inverse of :func:`patchify`."""
    t = tok.reshape(F, H // 2, W // 2, C, 2, 2).transpose(3, 0, 1, 4, 2, 5)
    return t.reshape(C, F, H, W)


def timestep_sinusoid(t, f_dim):
    """Sinusoid of ``1000 t``: ``[cos(1000 t f_j), sin(1000 t f_j)]``,
    ``f_j = exp(-ln(10^4) j / (f_dim/2))`` for j = 0..f_dim/2-1."""
    half = f_dim // 2
    freqs = np.exp(-np.log(10000.0) * np.arange(half, dtype=np.float64) / half)
    arg = 1000.0 * float(t) * freqs
    return np.concatenate([np.cos(arg), np.sin(arg)])


# ---------------------------------------------------------------------------
# the velocity model v_theta(x, t, c)  (Sec. 2; block as named by the workload)
# ---------------------------------------------------------------------------

class DiT:
    """float64 DiT velocity model over a parameter dict from the shared generator."""

    def __init__(self, cfg, params: dict):
        self.cfg = cfg
        self.p = {k: np.asarray(v, dtype=np.float64) for k, v in params.items()}

    # -- conditioning shared by every candidate ----------------------------
    def text_kv(self, ctx):
        """Per-block cross-attention K, V of the projected text (computed once per prompt).

        text = W2 GELU(W1 ctx + b1) + b2 ; [K | V] = text W_ckv^T + b_ckv.
        """
        p, d = self.p, self.cfg.d
        txt = linear(gelu_tanh(linear(np.asarray(ctx, np.float64), p["text_w1"], p["text_b1"])),
                     p["text_w2"], p["text_b2"])
        kv = []
        for b in range(self.cfg.blocks):
            y = linear(txt, p[f"blk{b}.ckv_w"], p[f"blk{b}.ckv_b"])
            kv.append((y[:, :d], y[:, d:]))
        return kv

    def modulation(self, t):
        """adaLN vectors for time t: per block (shift1, scale1, gate1, shift2, scale2, gate2)
        and the head's (shift, scale).

        e = W2 SiLU(W1 sin(t) + b1) + b2 ; m = W_mod SiLU(e) + b_mod (6 d, shared) plus a
        per-block [6, d] offset ; head = W_hm SiLU(e) + b_hm (2 d).
        """
        p, d = self.p, self.cfg.d
        e = linear(silu(linear(timestep_sinusoid(t, self.cfg.f_dim), p["time_w1"], p["time_b1"])),
                   p["time_w2"], p["time_b2"])
        m = linear(silu(e), p["mod_w"], p["mod_b"]).reshape(6, d)
        blocks = [m + p[f"blk{b}.mod_off"] for b in range(self.cfg.blocks)]
        hm = linear(silu(e), p["head_mod_w"], p["head_mod_b"]).reshape(2, d)
        return blocks, hm

    def block(self, b, x, mod, kv):
        """One transformer block on tokens x [L, d] (float64)."""
        p, H = self.p, self.cfg.heads
        shift1, scale1, gate1, shift2, scale2, gate2 = mod
        d = self.cfg.d
        h = layer_norm(x) * (1.0 + scale1) + shift1
        qkv = linear(h, p[f"blk{b}.qkv_w"], p[f"blk{b}.qkv_b"])
        sa = multi_head_attention(qkv[:, :d], qkv[:, d:2 * d], qkv[:, 2 * d:], H)
        x = x + gate1 * linear(sa, p[f"blk{b}.o_w"], p[f"blk{b}.o_b"])
        h = layer_norm(x)
        qc = linear(h, p[f"blk{b}.cq_w"], p[f"blk{b}.cq_b"])
        ca = multi_head_attention(qc, kv[0], kv[1], H)
        x = x + linear(ca, p[f"blk{b}.co_w"], p[f"blk{b}.co_b"])
        h = layer_norm(x) * (1.0 + scale2) + shift2
        f = linear(gelu_tanh(linear(h, p[f"blk{b}.ff1_w"], p[f"blk{b}.ff1_b"])),
                   p[f"blk{b}.ff2_w"], p[f"blk{b}.ff2_b"])
        return x + gate2 * f

    def block_rows(self, b, x, rows, mod, kv):
        """The block's output for the token rows ``rows`` only, x [L, d] being every token
        of the input.  Attention is the only step that mixes tokens, and it does so through
        the keys and values alone: K and V come from every row of x, everything else (the
        queries, projections, cross-attention, FFN) from the selected rows, so each selected
        row equals the same row of :meth:`block`."""
        p, H, d = self.p, self.cfg.heads, self.cfg.d
        shift1, scale1, gate1, shift2, scale2, gate2 = mod
        kv_self = linear(layer_norm(x) * (1.0 + scale1) + shift1, p[f"blk{b}.qkv_w"][d:], p[f"blk{b}.qkv_b"][d:])
        xr = x[rows]
        q = linear(layer_norm(xr) * (1.0 + scale1) + shift1, p[f"blk{b}.qkv_w"][:d], p[f"blk{b}.qkv_b"][:d])
        sa = multi_head_attention(q, kv_self[:, :d], kv_self[:, d:], H)
        xr = xr + gate1 * linear(sa, p[f"blk{b}.o_w"], p[f"blk{b}.o_b"])
        qc = linear(layer_norm(xr), p[f"blk{b}.cq_w"], p[f"blk{b}.cq_b"])
        xr = xr + linear(multi_head_attention(qc, kv[0], kv[1], H), p[f"blk{b}.co_w"], p[f"blk{b}.co_b"])
        h = layer_norm(xr) * (1.0 + scale2) + shift2
        f = linear(gelu_tanh(linear(h, p[f"blk{b}.ff1_w"], p[f"blk{b}.ff1_b"])), p[f"blk{b}.ff2_w"], p[f"blk{b}.ff2_b"])
        return xr + gate2 * f

    def velocity_rows(self, x, t, kv, rows):
        """Velocity of a one-block model at the token rows ``rows``, in token layout
        [len(rows), 4C] (feature ``4c + 2 ph + pw`` of token l, as :func:`patchify`): the
        rows of ``patchify(velocity(x, t, kv))``.  Only the last block may be evaluated on
        a subset of rows, so the model must have exactly one block."""
        if self.cfg.blocks != 1:
            raise ValueError("velocity_rows needs a one-block model (the next block would need every row)")
        mods, hm = self.modulation(t)
        tok = linear(patchify(np.asarray(x, np.float64)), self.p["patch_w"], self.p["patch_b"])
        out = self.block_rows(0, tok, rows, mods[0], kv[0])
        h = layer_norm(out) * (1.0 + hm[1]) + hm[0]
        return linear(h, self.p["head_w"], self.p["head_b"])

    def velocity(self, x, t, kv):
        """v_theta(x, t, c) for one latent x [C, F, H, W] -> [C, F, H, W]."""
        c = self.cfg
        mods, hm = self.modulation(t)
        tok = linear(patchify(np.asarray(x, np.float64)), self.p["patch_w"], self.p["patch_b"])
        for b in range(c.blocks):
            tok = self.block(b, tok, mods[b], kv[b])
        h = layer_norm(tok) * (1.0 + hm[1]) + hm[0]
        out = linear(h, self.p["head_w"], self.p["head_b"])
        return unpatchify(out, c.C, c.F, c.H, c.W)


# ---------------------------------------------------------------------------
# transformation-vector cache wrapper (Sec. 3.1)
# ---------------------------------------------------------------------------

@dataclass
class CacheState:
    """Per-candidate (single-branch) cache state: (Delta, x_ref, a) plus whether a
    Delta exists yet (Sec. 3.1; two latent-sized tensors and one scalar, Sec. 3.3)."""
    delta: np.ndarray | None = None
    x_ref: np.ndarray | None = None
    a: float = 0.0

    @property
    def has_ref(self) -> bool:
        return self.x_ref is not None


def relative_drift(x, x_ref):
    """``||x - x_ref||_F / ||x_ref||_F`` (Eq. indicator)."""
    return float(np.sqrt(np.sum((x - x_ref) ** 2)) / np.sqrt(np.sum(x_ref ** 2)))


def forced_compute(k, T, K_w, K_c, has_ref):
    """Warmup steps k <= K_w, cooldown steps k > T - K_c, and any step with an empty
    cache always compute (Sec. 3.1; App. Reproducibility)."""
    return k <= K_w or k > T - K_c or not has_ref


def wrapper_call(st: CacheState, x, k, T, tau, K_w, K_c, velocity_fn, force=None):
    """One intercepted transformer call at step k (1-based) on input x.

    Reading: on a forced step no drift is evaluated (the step computes and resets
    ``a``, so the drift would be discarded).  ``tau <= 0`` is the paper's "off"
    mode: every call computes, which makes ``G_0 = G`` exactly.  ``force`` (None, or
    a bool) replaces the skip decision after the drift has been accumulated; it is
    how a replayed mask keeps two implementations on the same schedule.

    Returns (velocity used, computed?, drift added this call or None).
    """
    x = np.asarray(x, np.float64)
    drift = None
    if forced_compute(k, T, K_w, K_c, st.has_ref):
        compute = True
    else:
        drift = relative_drift(x, st.x_ref)
        st.a += drift
        compute = (tau <= 0.0) or (st.a > tau)
    if force is not None:
        if not force and not st.has_ref:
            raise ValueError("cannot skip a call before the first Delta exists")
        compute = bool(force)
    if compute:
        v = np.asarray(velocity_fn(x), np.float64)
        st.delta = v - x          # Eq. delta
        st.x_ref = x.copy()
        st.a = 0.0
    else:
        v = x + st.delta          # Eq. skip
    return v, compute, drift


def rollout(x1, T, tau, K_w, K_c, velocity_fn_t, force_mask=None):
    """Cached rollout G_tau from noise x1: returns (x_{T+1}, computed[T], a after each step).

    ``velocity_fn_t(x, t)`` is the model; ``force_mask[k-1]`` optionally fixes step k's
    decision.  A fresh cache state per rollout (Algorithm 1 resets it per candidate).
    """
    t = time_grid(T)
    st = CacheState()
    x = np.asarray(x1, np.float64)
    computed, acc = [], []
    for k in range(1, T + 1):
        f = None if force_mask is None else bool(force_mask[k - 1])
        v, c, _ = wrapper_call(st, x, k, T, tau, K_w, K_c, lambda z: velocity_fn_t(z, t[k - 1]), f)
        x = euler(x, t[k - 1], t[k], v)
        computed.append(c)
        acc.append(st.a)
    return x, np.array(computed), np.array(acc)


def rollout_uncached(x1, T, velocity_fn_t):
    """Plain sampler G (no wrapper): T Euler steps on the model velocity (Eq. euler)."""
    t = time_grid(T)
    x = np.asarray(x1, np.float64)
    for k in range(1, T + 1):
        x = euler(x, t[k - 1], t[k], velocity_fn_t(x, t[k - 1]))
    return x


# ---------------------------------------------------------------------------
# batched step over N candidates (the unit the GPU path advances per call)
# ---------------------------------------------------------------------------

def search_step(states, xs, k, T, tau, K_w, K_c, velocity_fn_t, force=None, target=None):
    """Advance every candidate one Euler step under its own cache state.

    xs [N, ...] latents at t_k.  Returns (x_next [N, ...], skipped [N] bool,
    v_used [N, ...], scores or None).  With ``target`` given, each candidate is scored
    on the x0 estimate ``x_{k+1} - t_{k+1} v`` (equal to ``x_{T+1}`` on the last step).
    """
    t = time_grid(T)
    out, skipped, vs = [], [], []
    for i, st in enumerate(states):
        f = None if force is None else bool(force[i])
        v, c, _ = wrapper_call(st, xs[i], k, T, tau, K_w, K_c,
                               lambda z: velocity_fn_t(z, t[k - 1]), f)
        out.append(euler(np.asarray(xs[i], np.float64), t[k - 1], t[k], v))
        skipped.append(not c)
        vs.append(v)
    out = np.stack(out)
    scores = None
    if target is not None:
        x0 = out - t[k] * np.stack(vs)
        scores = np.array([score(x0[i], target) for i in range(len(states))])
    return out, np.array(skipped), np.stack(vs), scores


# ---------------------------------------------------------------------------
# scoring and selection (Algorithm 1; the verifier is replaced by L2-to-target)
# ---------------------------------------------------------------------------

def score(x0, target):
    """``-||x0 - y*||_2`` (stand-in verifier V(y, c))."""
    return -float(np.sqrt(np.sum((np.asarray(x0, np.float64) - np.asarray(target, np.float64)) ** 2)))


def topk(scores, k):
    """Indices of the k largest scores, descending; equal scores -> lower index first;
    NaN ranks below every number."""
    s = np.asarray(scores, np.float64)
    key = [(-np.inf if np.isnan(v) else v, i) for i, v in enumerate(s)]
    order = sorted(range(len(s)), key=lambda i: (-key[i][0], i))
    return np.array(order[:k], dtype=np.int32)


def cached_search(x1s, T, tau, K_w, K_c, velocity_fn_t, target):
    """Algorithm 1 exploration: N cached rollouts (fresh state each), score, argmax.

    Returns (i_star, scores, final latents, computed masks [N, T])."""
    finals, masks = [], []
    for x1 in x1s:
        xf, comp, _ = rollout(x1, T, tau, K_w, K_c, velocity_fn_t)
        finals.append(xf)
        masks.append(comp)
    scores = np.array([score(xf, target) for xf in finals])
    return int(topk(scores, 1)[0]), scores, np.stack(finals), np.stack(masks)


def beam_refill(states, xs, survivors, children, sigma, noise):
    """Beam refill: new slot ``p*(1+children)`` holds survivor ``survivors[p]`` unchanged;
    slots ``p*(1+children) + 1 + j`` hold its j-th child ``x + sigma * noise[p*children + j]``
    with a copy of the parent's cache state (Delta, x_ref, a)."""
    new_states, new_x = [], []
    for p, src in enumerate(survivors):
        st = states[src]
        for j in range(children + 1):
            cp = CacheState(None if st.delta is None else st.delta.copy(),
                            None if st.x_ref is None else st.x_ref.copy(), st.a)
            x = np.asarray(xs[src], np.float64).copy()
            if j > 0:  # children only exist when children > 0
                x = x + sigma * np.asarray(noise[p * children + j - 1], np.float64)
            new_states.append(cp)
            new_x.append(x)
    return new_states, np.stack(new_x)


# ---------------------------------------------------------------------------
# search variants built on the same step
# ---------------------------------------------------------------------------

def static_schedule(k, T, K_w, K_c, every):
    """Static uniform-schedule baseline (Sec. 3.1, Properties): warmup and cooldown steps
    compute; between them a step computes when (k - K_w) is a multiple of ``every``."""
    if k <= K_w or k > T - K_c:
        return True
    return (k - K_w) % every == 0


def rollout_static(x1, T, K_w, K_c, every, velocity_fn_t):
    """Cached rollout whose decisions follow :func:`static_schedule` (the indicator is
    still accumulated but does not decide)."""
    mask = np.array([static_schedule(k, T, K_w, K_c, every) for k in range(1, T + 1)])
    return rollout(x1, T, 1e30, K_w, K_c, velocity_fn_t, force_mask=mask)


def commit(x1, T, velocity_fn_t):
    """Algorithm 1, commit branch: regenerate the chosen seed at full compute, G(c, s)."""
    return rollout_uncached(x1, T, velocity_fn_t)


def beam_search(x1s, T, tau, K_w, K_c, velocity_fn_t, target, every, keep, children, sigma, noise_for_round):
    """Beam-style cached search (workload reading; the paper's closest step is the
    prune-and-continue composition of Sec. abl-stack): every ``every`` steps (before the
    last) score the x0 estimate, keep the top ``keep`` and refill each with ``children``
    perturbed copies (:func:`beam_refill`).  Returns (final scores, final latents, masks)."""
    states = [CacheState() for _ in range(len(x1s))]
    xs = np.asarray(x1s, np.float64)
    masks, r = [], 0
    for k in range(1, T + 1):
        rescore = (k % every == 0 and k < T) or k == T
        xs, skipped, _, sc = search_step(states, xs, k, T, tau, K_w, K_c, velocity_fn_t,
                                         target=target if rescore else None)
        masks.append(skipped)
        if k % every == 0 and k < T:
            surv = topk(sc, keep)
            states, xs = beam_refill(states, xs, list(surv), children, sigma, noise_for_round(r))
            r += 1
    return sc, xs, np.array(masks)


def pruned_search(x1s, T, tau, K_w, K_c, velocity_fn_t, target, prune_step, keep):
    """Cached search with mid-trajectory pruning (Sec. abl-stack): all candidates run
    cached to ``prune_step``, are scored on the sampler's x0 estimate, and only the top
    ``keep`` continue to step T.  Returns (winner's original index, final scores of the
    survivors, survivor original indices, final latents of the survivors)."""
    states = [CacheState() for _ in range(len(x1s))]
    xs = np.asarray(x1s, np.float64)
    ids = np.arange(len(x1s))
    for k in range(1, T + 1):
        prune = k == prune_step
        xs, _, _, sc = search_step(states, xs, k, T, tau, K_w, K_c, velocity_fn_t,
                                   target=target if (prune or k == T) else None)
        if prune:
            surv = topk(sc, keep)
            states, xs = beam_refill(states, xs, list(surv), 0, 0.0, None)
            ids = ids[surv]
    best = int(topk(sc, 1)[0])
    return int(ids[best]), sc, ids, xs


# ---------------------------------------------------------------------------
# classifier-free guidance with per-branch cache state (Eq. cfg; Sec. 3.1, per-branch state)
# ---------------------------------------------------------------------------

def cfg_combine(v_uncond, v_cond, w):
    """``v(x, t, 0) + w (v(x, t, c) - v(x, t, 0))`` (Eq. cfg)."""
    return v_uncond + w * (v_cond - v_uncond)


def search_step_cfg(states_c, states_u, xs, k, T, tau, K_w, K_c, vel_cond_t, vel_uncond_t, w,
                    force_c=None, force_u=None, target=None):
    """One guided Euler step of every candidate.  Each branch keeps its own cache state
    and takes its own decision on the same latent input (Sec. 3.1, per-branch cache
    state); the two velocities (computed or ``x + Delta_b``) are combined by Eq. cfg and
    the Euler step uses the combination.  Returns (x_next, skipped_c, skipped_u, scores)."""
    t = time_grid(T)
    out, sk_c, sk_u, vs = [], [], [], []
    for i in range(len(xs)):
        x = np.asarray(xs[i], np.float64)
        fc = None if force_c is None else bool(force_c[i])
        fu = None if force_u is None else bool(force_u[i])
        v_c, comp_c, _ = wrapper_call(states_c[i], x, k, T, tau, K_w, K_c, lambda z: vel_cond_t(z, t[k - 1]), fc)
        v_u, comp_u, _ = wrapper_call(states_u[i], x, k, T, tau, K_w, K_c, lambda z: vel_uncond_t(z, t[k - 1]), fu)
        v = cfg_combine(v_u, v_c, w)
        out.append(euler(x, t[k - 1], t[k], v))
        vs.append(v)
        sk_c.append(not comp_c)
        sk_u.append(not comp_u)
    out = np.stack(out)
    scores = None
    if target is not None:
        x0 = out - t[k] * np.stack(vs)
        scores = np.array([score(x0[i], target) for i in range(len(xs))])
    return out, np.array(sk_c), np.array(sk_u), scores
