"""Pins of the CPU oracle against what the paper and the mathematics fix (no GPU).

Each test checks the oracle against something other than itself: a worked example
derived by hand, a closed form, an invariant of the method, or an independent
library routine (torch / scipy) for a textbook primitive.
"""
import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as TF

from oracle import cachedsearch_oracle as O
from paper_2607_23159_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _tiny_model(blocks=2):
    cfg = synth.replace_model(synth.TINY, blocks=blocks)
    _, params = synth.make_params(cfg)
    return cfg, O.DiT(cfg, params)


def _read_golden(name):
    out = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            key, *vals = line.split()
            out[key] = np.array([float(v) for v in vals])
    return out


# ---------------------------------------------------------------- sampler -----

def test_time_grid_endpoints_and_spacing():
    t = O.time_grid(50)
    assert t[0] == 1.0 and t[-1] == 0.0 and len(t) == 51
    assert np.all(np.diff(t) < 0)
    np.testing.assert_allclose(np.diff(t), -1 / 50, rtol=0, atol=1e-15)


def test_euler_linear_field_closed_form():
    # v(x) = lam x  =>  x_{T+1} = prod_k (1 + h_k lam) x_1 exactly (Eq. euler)
    lam, T = -0.7, 13
    x1 = np.array([1.5, -2.0, 0.25])
    x = O.rollout_uncached(x1, T, lambda x, t: lam * x)
    t = O.time_grid(T)
    np.testing.assert_allclose(x, np.prod(1 + np.diff(t) * lam) * x1, rtol=1e-14)


def test_euler_constant_field_reaches_x1_minus_v():
    # constant velocity c on the grid 1 -> 0: x_0 = x_1 - c (sum of steps is -1)
    c = np.array([0.3, -1.1])
    x = O.rollout_uncached(np.array([2.0, 5.0]), 7, lambda x, t: c)
    np.testing.assert_allclose(x, np.array([2.0, 5.0]) - c, rtol=0, atol=1e-14)


# --------------------------------------------------------------- cache rule ---

def test_cache_rule_worked_example():
    g = _read_golden("cache_rule_1d.txt")
    xf, comp, acc = O.rollout(np.array([1.0]), 10, 0.25, 0, 0, lambda x, t: np.array([-1.0]))
    np.testing.assert_array_equal(comp.astype(int), g["computed"].astype(int))
    np.testing.assert_allclose(acc, g["accum_after_step"], rtol=0, atol=1e-12)
    np.testing.assert_allclose(xf, g["x_final"], rtol=0, atol=1e-12)


def test_tau_zero_is_uncached_sampling_bitwise():
    # "off" mode recovers G exactly (Sec. 3.1 Properties; bit-exact no-cache control)
    cfg, m = _tiny_model()
    kv = m.text_kv(synth.text_context(cfg))
    x1 = synth.initial_noise(cfg, [3])[0]
    vel = lambda x, t: m.velocity(x, t, kv)
    xc, comp, _ = O.rollout(x1, 10, 0.0, 1, 1, vel)
    xu = O.rollout_uncached(x1, 10, vel)
    assert comp.all()
    assert np.array_equal(xc, xu)


def test_huge_tau_skips_every_step_after_the_first_closed_form():
    # K_w = K_c = 0: step 1 computes (empty cache), every later step skips.  With
    # u_k = x_k + Delta a skip gives u_{k+1} = (1 + h_k) u_k, so
    # x_{T+1} = -Delta + prod_{k>=2}(1 + h_k) (x_2 + Delta), Delta = v(x_1) - x_1.
    cfg, m = _tiny_model()
    kv = m.text_kv(synth.text_context(cfg))
    x1 = synth.initial_noise(cfg, [1])[0].astype(np.float64)
    T = 10
    vel = lambda x, t: m.velocity(x, t, kv)
    xf, comp, _ = O.rollout(x1, T, 1e30, 0, 0, vel)
    assert comp[0] and not comp[1:].any()
    t = O.time_grid(T)
    v1 = m.velocity(x1, t[0], kv)
    delta = v1 - x1
    x2 = x1 + (t[1] - t[0]) * v1
    expect = -delta + np.prod(1 + np.diff(t)[1:]) * (x2 + delta)
    np.testing.assert_allclose(xf, expect, rtol=1e-12, atol=1e-12)


def test_warmup_cooldown_windows_force_compute():
    # v = 0 keeps x fixed, so the drift is 0 and every free step skips; only the
    # warmup (k <= K_w) and cooldown (k > T - K_c) windows compute.
    _, comp, _ = O.rollout(np.ones(4), 12, 0.1, 3, 2, lambda x, t: np.zeros(4))
    assert comp.astype(int).tolist() == [1, 1, 1, 0, 0, 0, 0, 0, 0, 0, 1, 1]


def test_forced_decision_replays_mask():
    f = np.array([1, 0, 0, 1, 0, 1, 0, 0, 0, 1], bool)
    _, comp, _ = O.rollout(np.array([1.0]), 10, 0.25, 0, 0, lambda x, t: np.array([-1.0]), f)
    assert np.array_equal(comp, f)
    with pytest.raises(ValueError):
        O.rollout(np.array([1.0]), 3, 0.25, 0, 0, lambda x, t: x, np.array([0, 1, 1], bool))


def test_search_step_equals_per_candidate_rollout():
    # batched advance of N candidates = N independent rollouts (batch invariance)
    cfg, m = _tiny_model()
    kv = m.text_kv(synth.text_context(cfg))
    x1s = synth.initial_noise(cfg, range(3)).astype(np.float64)
    vel = lambda x, t: m.velocity(x, t, kv)
    T = 6
    states = [O.CacheState() for _ in range(3)]
    xs = x1s.copy()
    masks = []
    for k in range(1, T + 1):
        xs, skipped, _, _ = O.search_step(states, xs, k, T, 0.5, 1, 1, vel)
        masks.append(~skipped)
    assert not np.array(masks).all()  # tau 0.5 skips steps 2 and 4: the states matter
    for i in range(3):
        xf, comp, _ = O.rollout(x1s[i], T, 0.5, 1, 1, vel)
        assert np.array_equal(xf, xs[i])
        assert np.array_equal(comp, np.array(masks)[:, i])


def test_x0_estimate_score_on_last_step_is_final_latent_score():
    cfg, m = _tiny_model()
    kv = m.text_kv(synth.text_context(cfg))
    x1s = synth.initial_noise(cfg, range(2)).astype(np.float64)
    y = synth.target_latent(cfg)
    vel = lambda x, t: m.velocity(x, t, kv)
    T = 3
    states = [O.CacheState() for _ in range(2)]
    xs = x1s
    for k in range(1, T + 1):
        xs, _, _, sc = O.search_step(states, xs, k, T, 0.5, 1, 1, vel, target=y)
    np.testing.assert_allclose(sc, [-np.linalg.norm(xs[i] - y) for i in range(2)], rtol=1e-15)


def test_x0_estimate_is_exact_for_a_constant_field():
    # v = c: every trajectory is the straight line x_t = x_1 - (1 - t) c, so the x0
    # estimate x_{k+1} - t_{k+1} v equals x_1 - c at every step, not only the last
    c = np.array([0.4, -0.2, 1.5])
    x1s = np.array([[1.0, 2.0, -1.0], [0.5, 0.0, 3.0]])
    y = np.array([0.1, 0.2, 0.3])
    T = 7
    states = [O.CacheState() for _ in range(2)]
    xs = x1s
    for k in range(1, T + 1):
        xs, _, _, sc = O.search_step(states, xs, k, T, 0.0, 0, 0, lambda x, t: c, target=y)
        np.testing.assert_allclose(sc, [-np.linalg.norm(x1s[i] - c - y) for i in range(2)], rtol=1e-13)


# --------------------------------------------------------- search / select ---

def test_topk_order_ties_and_nan():
    assert O.topk([1.0, 3.0, 3.0, 2.0], 2).tolist() == [1, 2]
    assert O.topk([np.nan, -5.0, 0.0], 3).tolist() == [2, 1, 0]
    rng = np.random.default_rng(0)
    for _ in range(50):
        s = rng.integers(-3, 3, size=9).astype(float)
        idx = O.topk(s, 9)
        # brute force: descending by value, ascending index among equals
        assert sorted(range(9), key=lambda i: (-s[i], i)) == idx.tolist()


def test_cached_search_brute_force_argmax():
    # Algorithm 1 on tiny inputs: argmax over independently scored rollouts
    cfg, m = _tiny_model(blocks=1)
    kv = m.text_kv(synth.text_context(cfg))
    x1s = synth.initial_noise(cfg, range(4))
    y = synth.target_latent(cfg)
    vel = lambda x, t: m.velocity(x, t, kv)
    i_star, scores, finals, comp = O.cached_search(x1s, 5, 0.5, 1, 1, vel, y)
    assert not comp.all()
    brute = [-np.sqrt(((O.rollout(x1s[i], 5, 0.5, 1, 1, vel)[0] - y) ** 2).sum()) for i in range(4)]
    np.testing.assert_allclose(scores, brute, rtol=1e-15)
    assert scores[i_star] == max(scores)


def test_beam_refill_layout_and_state_copy():
    st = [O.CacheState(np.full(2, i * 1.0), np.full(2, 10.0 + i), 0.01 * i) for i in range(4)]
    xs = np.arange(8, dtype=float).reshape(4, 2)
    noise = np.ones((2 * 2, 2))
    ns, nx = O.beam_refill(st, xs, [2, 0], 2, 0.1, noise)
    assert len(ns) == 6
    np.testing.assert_array_equal(nx[0], xs[2])
    np.testing.assert_allclose(nx[1], xs[2] + 0.1)
    np.testing.assert_array_equal(nx[3], xs[0])
    assert ns[1].a == st[2].a and np.array_equal(ns[4].x_ref, st[0].x_ref)


# --------------------------------------------------------------- primitives ---

def test_attention_special_cases():
    rng = np.random.default_rng(1)
    v = rng.standard_normal((5, 4))
    q = rng.standard_normal((3, 4))
    # one key -> output is that value row
    np.testing.assert_allclose(O.attention(q, rng.standard_normal((1, 4)), v[:1]), np.repeat(v[:1], 3, 0))
    # identical keys -> uniform weights -> mean of V
    k = np.repeat(rng.standard_normal((1, 4)), 5, 0)
    np.testing.assert_allclose(O.attention(q, k, v), np.repeat(v.mean(0, keepdims=True), 3, 0), atol=1e-14)
    # two keys with hand logits: q.k1/sqrt(4) = 0.5, q.k2 = 0 -> weights (s, 1-s), s = logistic(0.5)
    s = 1 / (1 + math.exp(-0.5))
    out = O.attention(np.ones((1, 4)), np.array([[1.0, 0, 0, 0], [0, 0, 0, 0]]), v[:2])
    np.testing.assert_allclose(out[0], s * v[0] + (1 - s) * v[1], rtol=1e-13, atol=1e-15)


def test_attention_rows_sum_to_one_and_match_torch_sdpa():
    rng = np.random.default_rng(2)
    q, k, v = (rng.standard_normal((37, 16)) for _ in range(3))
    p = O.softmax_rows(q @ k.T / 4.0)
    np.testing.assert_allclose(p.sum(1), 1.0, atol=1e-14)
    ref = TF.scaled_dot_product_attention(*(torch.from_numpy(a)[None] for a in (q, k, v)))[0]
    np.testing.assert_allclose(O.attention(q, k, v), ref.numpy(), atol=1e-12)


def test_layer_norm_gelu_linear_against_independent_routines():
    from scipy.special import erf
    rng = np.random.default_rng(3)
    x = rng.standard_normal((6, 10)) * 3 + 1
    ref = TF.layer_norm(torch.from_numpy(x), (10,), eps=1e-6).numpy()
    np.testing.assert_allclose(O.layer_norm(x), ref, atol=1e-12)
    np.testing.assert_allclose(O.layer_norm(np.array([[-1.0, 1.0]])), [[-1 / math.sqrt(1 + 1e-6), 1 / math.sqrt(1 + 1e-6)]])
    g = O.gelu_tanh(x)
    np.testing.assert_allclose(g, TF.gelu(torch.from_numpy(x), approximate="tanh").numpy(), atol=1e-13)
    # the tanh form stays within 1e-3 of the exact x Phi(x)
    np.testing.assert_allclose(g, 0.5 * x * (1 + erf(x / math.sqrt(2))), atol=1e-3)
    w = rng.standard_normal((3, 10))
    b = rng.standard_normal(3)
    np.testing.assert_allclose(O.linear(x, w, b), TF.linear(torch.from_numpy(x), torch.from_numpy(w), torch.from_numpy(b)).numpy(), atol=1e-12)
    # non-square hand case: y = x W^T + b
    np.testing.assert_allclose(O.linear(np.array([[1.0, 2.0]]), np.array([[1.0, 0.0], [0.0, 3.0], [1.0, 1.0]]), np.zeros(3)), [[1.0, 6.0, 3.0]])


def test_patchify_layout_and_inverse():
    C, F, H, W = 3, 2, 4, 6
    x = np.arange(C * F * H * W, dtype=float).reshape(C, F, H, W)
    tok = O.patchify(x)
    assert tok.shape == (F * 2 * 3, C * 4)
    for (c, f, h, w) in [(0, 0, 0, 0), (2, 1, 3, 5), (1, 0, 2, 1), (2, 1, 1, 4)]:
        assert tok[(f * 2 + h // 2) * 3 + w // 2, c * 4 + (h % 2) * 2 + (w % 2)] == x[c, f, h, w]
    np.testing.assert_array_equal(O.unpatchify(tok, C, F, H, W), x)


def test_timestep_sinusoid_values():
    e = O.timestep_sinusoid(0.0, 8)
    np.testing.assert_array_equal(e, [1, 1, 1, 1, 0, 0, 0, 0])
    e = O.timestep_sinusoid(0.5, 8)
    # j = 0 has frequency 1: cos(500), sin(500); j = 2 has 10^-2: cos(5), sin(5)
    np.testing.assert_allclose([e[0], e[4], e[2], e[6]], [math.cos(500), math.sin(500), math.cos(5), math.sin(5)], rtol=1e-12)


def _block_torch(p, b, x, mod, kv, heads):
    """The same block written with torch.nn.functional primitives (float64)."""
    T = lambda a: torch.from_numpy(np.asarray(a, np.float64))
    x = T(x)
    d = x.shape[1]
    hd = d // heads
    sh1, sc1, g1, sh2, sc2, g2 = (T(m) for m in mod)
    ln = lambda z: TF.layer_norm(z, (d,), eps=1e-6)

    def mha(q, k, v):
        sp = lambda z: z.reshape(z.shape[0], heads, hd).transpose(0, 1)
        return TF.scaled_dot_product_attention(sp(q), sp(k), sp(v)).transpose(0, 1).reshape(q.shape[0], d)

    h = ln(x) * (1 + sc1) + sh1
    q, k, v = TF.linear(h, T(p[f"blk{b}.qkv_w"]), T(p[f"blk{b}.qkv_b"])).split(d, dim=1)
    x = x + g1 * TF.linear(mha(q, k, v), T(p[f"blk{b}.o_w"]), T(p[f"blk{b}.o_b"]))
    qc = TF.linear(ln(x), T(p[f"blk{b}.cq_w"]), T(p[f"blk{b}.cq_b"]))
    x = x + TF.linear(mha(qc, T(kv[0]), T(kv[1])), T(p[f"blk{b}.co_w"]), T(p[f"blk{b}.co_b"]))
    h = ln(x) * (1 + sc2) + sh2
    f = TF.linear(TF.gelu(TF.linear(h, T(p[f"blk{b}.ff1_w"]), T(p[f"blk{b}.ff1_b"])), approximate="tanh"),
                  T(p[f"blk{b}.ff2_w"]), T(p[f"blk{b}.ff2_b"]))
    return (x + g2 * f).numpy()


def test_block_against_torch_functional_composition():
    cfg, m = _tiny_model(blocks=1)
    rng = np.random.default_rng(4)
    # random (non-zero) biases and offsets so that every term is exercised
    for k in list(m.p):
        if k.endswith("_b") or k.endswith("mod_off"):
            m.p[k] = rng.standard_normal(m.p[k].shape) * 0.3
    kv = m.text_kv(synth.text_context(cfg))
    mods, _ = m.modulation(0.37)
    x = rng.standard_normal((cfg.L, cfg.d))
    np.testing.assert_allclose(m.block(0, x, mods[0], kv[0]),
                               _block_torch(m.p, 0, x, mods[0], kv[0], cfg.heads), atol=1e-10)


def test_dit_token_permutation_equivariance():
    # no positional encoding: permuting video tokens permutes the velocity tokens
    cfg, m = _tiny_model()
    kv = m.text_kv(synth.text_context(cfg))
    x = synth.initial_noise(cfg, [0])[0].astype(np.float64)
    tok = O.patchify(x)
    perm = np.random.default_rng(5).permutation(cfg.L)
    v = O.patchify(m.velocity(x, 0.6, kv))
    vp = O.patchify(m.velocity(O.unpatchify(tok[perm], cfg.C, cfg.F, cfg.H, cfg.W), 0.6, kv))
    np.testing.assert_allclose(vp, v[perm], atol=1e-11)


def test_dit_text_token_permutation_invariance():
    # cross-attention sums over the text tokens: reordering them (keys and values
    # together) leaves the velocity unchanged
    cfg, m = _tiny_model()
    ctx = synth.text_context(cfg)
    perm = np.random.default_rng(6).permutation(cfg.Lt)
    x = synth.initial_noise(cfg, [1])[0].astype(np.float64)
    v = m.velocity(x, 0.4, m.text_kv(ctx))
    np.testing.assert_allclose(m.velocity(x, 0.4, m.text_kv(np.asarray(ctx)[perm])), v, atol=1e-11)


def test_dit_zero_blocks_reduce_to_head_of_embedding():
    # all block weights 0 (and biases 0): every block is the identity, so
    # v = head(LN(embed(x)) (1 + scale_h) + shift_h)
    cfg, m = _tiny_model()
    for k in list(m.p):
        if k.startswith("blk"):
            m.p[k] = np.zeros_like(m.p[k])
    kv = m.text_kv(synth.text_context(cfg))
    x = synth.initial_noise(cfg, [2])[0].astype(np.float64)
    t = 0.25
    _, hm = m.modulation(t)
    tok = O.patchify(x) @ m.p["patch_w"].T
    mu = tok.mean(1, keepdims=True)
    sd = np.sqrt(tok.var(1, keepdims=True) + 1e-6)
    out = ((tok - mu) / sd * (1 + hm[1]) + hm[0]) @ m.p["head_w"].T
    np.testing.assert_allclose(O.patchify(m.velocity(x, t, kv)), out, atol=1e-12)


def test_row_subset_forms_equal_the_full_forward():
    # the block and the one-block velocity evaluated on a subset of token rows are the
    # same rows of the full evaluation (attention mixes tokens only through K and V)
    cfg, m = _tiny_model(blocks=1)
    rng = np.random.default_rng(27)
    for k in list(m.p):
        if k.endswith("_b") or k.endswith("mod_off"):
            m.p[k] = rng.standard_normal(m.p[k].shape) * 0.3
    kv = m.text_kv(synth.text_context(cfg))
    mods, _ = m.modulation(0.55)
    x = rng.standard_normal((cfg.L, cfg.d))
    rows = np.array([0, 5, 17, cfg.L - 1])
    np.testing.assert_allclose(m.block_rows(0, x, rows, mods[0], kv[0]), m.block(0, x, mods[0], kv[0])[rows],
                               atol=1e-11)
    lat = synth.initial_noise(cfg, [3])[0].astype(np.float64)
    np.testing.assert_allclose(m.velocity_rows(lat, 0.55, kv, rows), O.patchify(m.velocity(lat, 0.55, kv))[rows],
                               atol=1e-11)
    with pytest.raises(ValueError):
        _tiny_model(blocks=2)[1].velocity_rows(lat, 0.5, kv, rows)


# ---------------------------------------------------- conditioning MLPs ---
# The adaLN modulation MLP and the text projection are the workload architecture's
# conditioning (Sec. 2 names a DiT conditioned on t and the text c; the block is fixed
# by the workload).  Their pins: closed-form values through identity weights, the
# roles of the six adaLN vectors and of the head's two inside the block, and an
# independent torch.nn composition with every bias and offset non-zero.

def _eye_stack(reps, d):
    return np.concatenate([np.eye(d)] * reps, axis=0)


def test_modulation_closed_form_through_identity_weights():
    # time_w2 = 0 makes e = time_b2 exactly; with e = (ln 3, -ln 3, 0, ...) the SiLU
    # has the closed forms SiLU(ln 3) = 3/4 ln 3, SiLU(-ln 3) = -1/4 ln 3, SiLU(0) = 0.
    # mod_w / head_mod_w = stacked identities pass SiLU(e) to every vector, so chunk j
    # of block b is SiLU(e) + b_mod[j] + offset_b[j] and the head's is SiLU(e) + b_hm[j].
    cfg, m = _tiny_model(blocks=3)
    d = cfg.d
    rng = np.random.default_rng(21)
    ln3 = math.log(3.0)
    e0 = np.resize(np.array([ln3, -ln3, 0.0]), d)
    silu_e0 = np.resize(np.array([0.75 * ln3, -0.25 * ln3, 0.0]), d)
    m.p["time_w2"] = np.zeros((d, d))
    m.p["time_b2"] = e0
    m.p["mod_w"] = _eye_stack(6, d)
    m.p["mod_b"] = rng.standard_normal(6 * d)
    m.p["head_mod_w"] = _eye_stack(2, d)
    m.p["head_mod_b"] = rng.standard_normal(2 * d)
    for b in range(cfg.blocks):
        m.p[f"blk{b}.mod_off"] = rng.standard_normal((6, d))
    for t in (0.0, 0.3, 1.0):          # e does not depend on t here
        mods, hm = m.modulation(t)
        assert len(mods) == cfg.blocks
        for b in range(cfg.blocks):
            for j in range(6):         # shift1, scale1, gate1, shift2, scale2, gate2
                np.testing.assert_allclose(mods[b][j], silu_e0 + m.p["mod_b"][j * d:(j + 1) * d]
                                           + m.p[f"blk{b}.mod_off"][j], rtol=0, atol=1e-14)
        for j in range(2):             # head shift, scale
            np.testing.assert_allclose(hm[j], silu_e0 + m.p["head_mod_b"][j * d:(j + 1) * d], rtol=0, atol=1e-14)


def test_modulation_sinusoid_path_closed_form():
    # time_w1 = [I; 0], time_w2 = I and zero biases: e = SiLU(sinusoid(t)) on the first
    # f_dim features and 0 after them; mod_w = stacked identities: every adaLN vector is
    # SiLU(e).  At t = 0 the sinusoid is (1, ..., 1, 0, ..., 0), so the first half holds
    # SiLU(SiLU(1)) with SiLU(1) = e/(e+1); at t = 1/2 its first cosine is cos(500).
    cfg, m = _tiny_model(blocks=1)
    d, f = cfg.d, cfg.f_dim
    w1 = np.zeros((d, f))
    w1[:f, :f] = np.eye(f)
    m.p["time_w1"], m.p["time_b1"] = w1, np.zeros(d)
    m.p["time_w2"], m.p["time_b2"] = np.eye(d), np.zeros(d)
    m.p["mod_w"], m.p["mod_b"] = _eye_stack(6, d), np.zeros(6 * d)
    m.p["blk0.mod_off"] = np.zeros((6, d))
    silu = lambda z: z / (1.0 + math.exp(-z))
    s1 = math.e / (math.e + 1.0)
    mods, _ = m.modulation(0.0)
    for j in range(6):
        np.testing.assert_allclose(mods[0][j][:f // 2], silu(s1), rtol=1e-14)
        np.testing.assert_array_equal(mods[0][j][f // 2:], 0.0)
    mods, _ = m.modulation(0.5)
    np.testing.assert_allclose(mods[0][0][0], silu(silu(math.cos(500.0))), rtol=1e-13)
    np.testing.assert_allclose(mods[0][3][f // 2], silu(silu(math.sin(500.0))), rtol=1e-13)


def _block_with(m, cfg, b, mod, zero):
    for k in zero:
        m.p[f"blk{b}.{k}"] = np.zeros_like(m.p[f"blk{b}.{k}"])
    rng = np.random.default_rng(23)
    x = rng.standard_normal((cfg.L, cfg.d))
    kv = m.text_kv(synth.text_context(cfg))
    return x, m.block(b, x, mod, kv[b])


def test_adaln_vectors_play_their_roles_in_the_block():
    # scale = -1 cancels the normalised input, leaving h = shift for every token; with
    # the other branches' weights zero the block then adds the same vector to every
    # token.  A gate of 0 removes its branch whatever the branch computes.
    rng = np.random.default_rng(22)
    cfg, m = _tiny_model(blocks=1)
    d = cfg.d
    mod = [rng.standard_normal(d) * 0.5 for _ in range(6)]
    mod[1] = -np.ones(d)                                   # scale1
    x, y = _block_with(m, cfg, 0, mod, ["cq_w", "co_w", "ff1_w", "ff2_w"])
    r = y - x
    np.testing.assert_allclose(r, np.broadcast_to(r[0], r.shape), atol=1e-12)
    assert np.abs(r[0]).max() > 1e-3

    cfg, m = _tiny_model(blocks=1)
    mod = [rng.standard_normal(d) * 0.5 for _ in range(6)]
    mod[4] = -np.ones(d)                                   # scale2
    x, y = _block_with(m, cfg, 0, mod, ["qkv_w", "o_w", "cq_w", "co_w"])
    r = y - x
    np.testing.assert_allclose(r, np.broadcast_to(r[0], r.shape), atol=1e-12)
    assert np.abs(r[0]).max() > 1e-3

    # gates: with gate1 = gate2 = 0 the block is x + CA(LN(x)); random self-attention
    # and FFN weights then change nothing
    cfg, m = _tiny_model(blocks=1)
    mod = [rng.standard_normal(d) * 0.5 for _ in range(6)]
    mod[2] = np.zeros(d)
    mod[5] = np.zeros(d)
    kv = m.text_kv(synth.text_context(cfg))
    x = rng.standard_normal((cfg.L, d))
    y0 = m.block(0, x, mod, kv[0])
    for k in ("qkv_w", "o_w", "ff1_w", "ff2_w"):
        m.p[f"blk0.{k}"] = rng.standard_normal(m.p[f"blk0.{k}"].shape)
    np.testing.assert_allclose(m.block(0, x, mod, kv[0]), y0, atol=1e-12)


def test_head_modulation_roles():
    # head scale = -1 (through head_mod_b, with head_mod_w = 0): every token's head
    # input is the head shift, so the velocity is the same per-patch vector
    # head_w shift + head_b at every token, for any latent
    cfg, m = _tiny_model()
    d = cfg.d
    rng = np.random.default_rng(24)
    shift = rng.standard_normal(d)
    m.p["head_mod_w"] = np.zeros((2 * d, d))
    m.p["head_mod_b"] = np.concatenate([shift, -np.ones(d)])
    m.p["head_b"] = rng.standard_normal(cfg.P)
    kv = m.text_kv(synth.text_context(cfg))
    expect = m.p["head_w"] @ shift + m.p["head_b"]
    for s in (0, 1):
        x = synth.initial_noise(cfg, [s])[0].astype(np.float64)
        v = O.patchify(m.velocity(x, 0.45, kv))
        np.testing.assert_allclose(v, np.broadcast_to(expect, v.shape), atol=1e-12)


def test_text_kv_closed_form_through_identity_weights():
    # text_w1 = I, text_w2 = 2 I, text_b2 = beta, ckv_w = [I; 3 I]: per block b
    #   K_b(c) = 2 GELU(c) + beta + kb_b,   V_b(c) = 3 (2 GELU(c) + beta) + vb_b.
    # GELU(c) - GELU(-c) = c exactly (tanh form), and GELU(c) + GELU(-c) is within 2e-3
    # of its exact-erf value c erf(c / sqrt 2).
    cfg, m = _tiny_model(blocks=3)
    d = cfg.d
    assert cfg.d_text == d
    rng = np.random.default_rng(25)
    beta = rng.standard_normal(d)
    m.p["text_w1"], m.p["text_b1"] = np.eye(d), np.zeros(d)
    m.p["text_w2"], m.p["text_b2"] = 2.0 * np.eye(d), beta
    for b in range(cfg.blocks):
        m.p[f"blk{b}.ckv_w"] = np.concatenate([np.eye(d), 3.0 * np.eye(d)])
        m.p[f"blk{b}.ckv_b"] = rng.standard_normal(2 * d)
    c = rng.standard_normal((cfg.Lt, d)) * 1.5
    kv_p, kv_m = m.text_kv(c), m.text_kv(-c)
    even = c * np.vectorize(math.erf)(c / math.sqrt(2.0))     # GELU(c) + GELU(-c), exact-erf form
    for b in range(cfg.blocks):
        kb, vb = m.p[f"blk{b}.ckv_b"][:d], m.p[f"blk{b}.ckv_b"][d:]
        (K, V), (Km, Vm) = kv_p[b], kv_m[b]
        np.testing.assert_allclose(K - Km, 2.0 * c, atol=1e-12)
        np.testing.assert_allclose(K + Km, 2.0 * even + 2.0 * (beta + kb), atol=4e-3)
        np.testing.assert_allclose(V - 3.0 * K, np.broadcast_to(vb - 3.0 * kb, V.shape), atol=1e-12)


def test_conditioning_against_torch_nn_composition():
    """modulation() and text_kv() rebuilt from torch.nn.Linear modules, F.silu,
    F.gelu(approximate='tanh') and a torch sinusoid with 10000^(-j/half) frequencies,
    with every bias and offset random and non-zero."""
    cfg, m = _tiny_model(blocks=2)
    d, f = cfg.d, cfg.f_dim
    rng = np.random.default_rng(26)
    for k in list(m.p):
        if k.endswith("_b") or k.endswith("_b1") or k.endswith("_b2") or k.endswith("mod_off"):
            m.p[k] = rng.standard_normal(m.p[k].shape) * 0.3
    T = lambda a: torch.from_numpy(np.asarray(a, np.float64))

    def lin(wk, bk):
        layer = torch.nn.Linear(m.p[wk].shape[1], m.p[wk].shape[0], dtype=torch.float64)
        with torch.no_grad():
            layer.weight.copy_(T(m.p[wk]))
            layer.bias.copy_(T(m.p[bk]))
        return layer

    with torch.no_grad():
        for t in (0.0, 0.37, 0.9):
            half = f // 2
            freq = torch.pow(torch.tensor(10000.0, dtype=torch.float64),
                             -torch.arange(half, dtype=torch.float64) / half)
            ang = (1000.0 * t) * freq
            sinus = torch.cat([torch.cos(ang), torch.sin(ang)])
            e = lin("time_w2", "time_b2")(TF.silu(lin("time_w1", "time_b1")(sinus)))
            six = lin("mod_w", "mod_b")(TF.silu(e)).view(6, d)
            head = lin("head_mod_w", "head_mod_b")(TF.silu(e)).view(2, d)
            mods, hm = m.modulation(t)
            for b in range(cfg.blocks):
                np.testing.assert_allclose(np.asarray(mods[b]), (six + T(m.p[f"blk{b}.mod_off"])).numpy(),
                                           atol=1e-12)
            np.testing.assert_allclose(np.asarray(hm), head.numpy(), atol=1e-12)
        ctx = T(synth.text_context(cfg))
        txt = lin("text_w2", "text_b2")(TF.gelu(lin("text_w1", "text_b1")(ctx), approximate="tanh"))
        kv = m.text_kv(synth.text_context(cfg))
        for b in range(cfg.blocks):
            k_t, v_t = lin(f"blk{b}.ckv_w", f"blk{b}.ckv_b")(txt).split(d, dim=1)
            np.testing.assert_allclose(kv[b][0], k_t.numpy(), atol=1e-12)
            np.testing.assert_allclose(kv[b][1], v_t.numpy(), atol=1e-12)


# ------------------------------------------------------------ search variants ---

def test_static_schedule_hand_example_and_every_one_is_uncached():
    got = [O.static_schedule(k, 12, 2, 2, 3) for k in range(1, 13)]
    # warmup 1-2, cooldown 11-12, in between k - 2 in {3, 6} -> k = 5, 8
    assert [int(g) for g in got] == [1, 1, 0, 0, 1, 0, 0, 1, 0, 0, 1, 1]
    cfg, m = _tiny_model(blocks=1)
    kv = m.text_kv(synth.text_context(cfg))
    x1 = synth.initial_noise(cfg, [0])[0]
    vel = lambda x, t: m.velocity(x, t, kv)
    xs, comp, _ = O.rollout_static(x1, 6, 1, 1, 1, vel)
    assert comp.all() and np.array_equal(xs, O.rollout_uncached(x1, 6, vel))
    assert np.array_equal(O.commit(x1, 6, vel), O.rollout_uncached(x1, 6, vel))


def test_beam_and_pruned_search_degenerate_cases():
    cfg, m = _tiny_model(blocks=1)
    kv = m.text_kv(synth.text_context(cfg))
    x1s = synth.initial_noise(cfg, range(4))
    y = synth.target_latent(cfg)
    vel = lambda x, t: m.velocity(x, t, kv)
    T = 6
    i_star, sc, _, _ = O.cached_search(x1s, T, 0.5, 1, 1, vel, y)
    # keep everything, no children: the beam only permutes slots
    sb, _, _ = O.beam_search(x1s, T, 0.5, 1, 1, vel, y, every=2, keep=4, children=0, sigma=0.0,
                             noise_for_round=lambda r: None)
    np.testing.assert_allclose(np.sort(sb), np.sort(sc), rtol=1e-12)
    # sigma = 0 children are exact copies of their parent
    sb, xb, skipped = O.beam_search(x1s, T, 0.5, 1, 1, vel, y, every=3, keep=2, children=1, sigma=0.0,
                                    noise_for_round=lambda r: np.ones((2, *x1s.shape[1:])))
    assert skipped[3:].any()  # children skip on the cache state they inherited
    assert np.array_equal(xb[0], xb[1]) and np.array_equal(xb[2], xb[3])
    # pruning that keeps every candidate picks the same winner as the plain search
    win, sp, ids, _ = O.pruned_search(x1s, T, 0.5, 1, 1, vel, y, prune_step=3, keep=4)
    assert win == i_star
    np.testing.assert_allclose(np.sort(sp), np.sort(sc), rtol=1e-12)


def test_cfg_guidance_one_is_conditional_and_tau_zero_is_uncached_guided_sampling():
    cfg, m = _tiny_model(blocks=1)
    kv_c = m.text_kv(synth.text_context(cfg))
    kv_u = m.text_kv(np.zeros((cfg.Lt, cfg.d_text)))
    vc = lambda x, t: m.velocity(x, t, kv_c)
    vu = lambda x, t: m.velocity(x, t, kv_u)
    x1s = synth.initial_noise(cfg, range(2)).astype(np.float64)
    T = 5
    # w = 1: the combination is the conditional velocity exactly -> plain conditional sampling
    sc, su = [O.CacheState() for _ in range(2)], [O.CacheState() for _ in range(2)]
    xs = x1s
    for k in range(1, T + 1):
        xs, _, _, _ = O.search_step_cfg(sc, su, xs, k, T, 0.0, 1, 1, vc, vu, 1.0)
    for i in range(2):
        np.testing.assert_allclose(xs[i], O.rollout_uncached(x1s[i], T, vc), rtol=1e-12, atol=1e-12)
    # w = 0: the unconditional velocity alone
    sc, su = [O.CacheState() for _ in range(2)], [O.CacheState() for _ in range(2)]
    xs = x1s
    for k in range(1, T + 1):
        xs, _, _, _ = O.search_step_cfg(sc, su, xs, k, T, 0.0, 1, 1, vc, vu, 0.0)
    for i in range(2):
        np.testing.assert_allclose(xs[i], O.rollout_uncached(x1s[i], T, vu), rtol=1e-12, atol=1e-12)
    # w = 5, tau = 0: uncached guided Euler sampling (Eq. cfg + Eq. euler) written out
    sc, su = [O.CacheState() for _ in range(2)], [O.CacheState() for _ in range(2)]
    xs = x1s
    for k in range(1, T + 1):
        xs, skc, sku, _ = O.search_step_cfg(sc, su, xs, k, T, 0.0, 1, 1, vc, vu, 5.0)
        assert not skc.any() and not sku.any()
    t = O.time_grid(T)
    for i in range(2):
        x = x1s[i]
        for k in range(T):
            a, b = vu(x, t[k]), vc(x, t[k])
            x = x + (t[k + 1] - t[k]) * (a + 5.0 * (b - a))
        assert np.array_equal(xs[i], x)
    # branches keep separate state: with a huge tau each branch skips after its first call
    sc, su = [O.CacheState()], [O.CacheState()]
    xs = x1s[:1]
    for k in range(1, T + 1):
        xs, skc, sku, _ = O.search_step_cfg(sc, su, xs, k, T, 1e30, 0, 0, vc, vu, 5.0)
        assert skc[0] == (k > 1) and sku[0] == (k > 1)
    assert not np.array_equal(sc[0].delta, su[0].delta)
