"""End-to-end parity of the batched cached-search step (GPU) with the fp64 oracle.

* tiny configuration (2 blocks, d 128, 48 tokens, N 4, T 10, tau 0.1): the whole search,
  once free-running (masks must agree except where the oracle's indicator is within 1e-3
  of tau) and once replaying the oracle's masks (final latents within 2e-2 max relative
  error, top-1 identical);
* the 1.3B model width (d 1536, 12 x 128 heads, FFN 8960, 512 x 4096 text) with 2 blocks
  on a small latent, where the oracle still finishes in seconds;
* both with bf16-valued weights (the kernels alone) and with unrounded float32 weights
  that the library rounds on load (bf16 vs fp32, the weight rounding included);
* properties that hold at any size: batch invariance (a candidate's result is bitwise
  the same alone or inside any batch), run-to-run determinism, tau = 0 equals always
  computing, and the closed form of an all-skip rollout.
"""
import numpy as np
import pytest
import torch

from oracle import cachedsearch_oracle as O
from paper_2607_23159_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def B():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_23159_gb300 import binding
    return binding


def dev(a, dtype=torch.float32):
    return torch.from_numpy(np.ascontiguousarray(a)).to("cuda").to(dtype)


class Inputs:
    def __init__(self, m, N, seeds=None, round_bf16=True):
        self.m = m
        self.flat, self.params = synth.make_params(m, round_bf16=round_bf16)
        self.ctx = synth.text_context(m)
        self.x1 = synth.initial_noise(m, seeds if seeds is not None else range(N))
        self.y = synth.target_latent(m)


def gpu_search(B, inp, N, T, tau, K_w, K_c, force_masks=None, model=None, score=True):
    m = inp.m
    own = model is None
    if own:
        model = B.Model(m, N)
        model.load_weights(inp.flat)
        model.set_text_context(dev(inp.ctx))
    st = B.new_state(N, m.D)
    st["x"].copy_(dev(inp.x1.reshape(N, -1)))
    t = O.time_grid(T)
    skip = torch.zeros(N, dtype=torch.uint8, device="cuda")
    scores = torch.zeros(N, device="cuda")
    y = dev(inp.y.reshape(-1))
    masks, ncs = [], []
    for k in range(1, T + 1):
        force = None if force_masks is None else dev(force_masks[k - 1].astype(np.uint8), torch.uint8)
        n = model.search_step(st, k, T, float(t[k - 1]), float(t[k]), tau, K_w, K_c, skip, force=force,
                              target=y if (score and k == T) else None, scores=scores)
        masks.append(skip.cpu().numpy().astype(bool))
        ncs.append(n)
    torch.cuda.synchronize()
    assert model.device_error() == 0
    out = (st, np.array(masks), scores.cpu().numpy(), ncs)
    if own:
        model.close()
    return out


def oracle_search(inp, N, T, tau, K_w, K_c):
    m = inp.m
    dit = O.DiT(m, inp.params)
    kv = dit.text_kv(inp.ctx)
    vel = lambda z, tt: dit.velocity(z, tt, kv)
    states = [O.CacheState() for _ in range(N)]
    xs = inp.x1.astype(np.float64)
    masks, pres = [], []
    for k in range(1, T + 1):
        pre = [None if O.forced_compute(k, T, K_w, K_c, s.has_ref) else s.a + O.relative_drift(xs[i], s.x_ref)
               for i, s in enumerate(states)]
        xs, skipped, _, sc = O.search_step(states, xs, k, T, tau, K_w, K_c, vel,
                                           target=inp.y if k == T else None)
        masks.append(skipped)
        pres.append(pre)
    return xs, np.array(masks), sc, pres


def max_rel(g, o):
    return max(np.abs(g[i] - o[i]).max() / np.abs(o[i]).max() for i in range(len(o)))


# ------------------------------------------------------------- tiny config ----

@pytest.fixture(scope="module")
def tiny():
    cfg = synth.CONFIGS["tiny"]
    inp = Inputs(cfg.model, cfg.N)
    ref = oracle_search(inp, cfg.N, cfg.T, cfg.tau, cfg.K_w, cfg.K_c)
    return cfg, inp, ref


@pytest.fixture(scope="module")
def tiny_fp32():
    """The tiny workload with unrounded float32 weights: the oracle takes them as they
    are and the library rounds them to bf16 on load, so the parity includes the weight
    rounding (bf16 vs fp32)."""
    cfg = synth.CONFIGS["tiny"]
    inp = Inputs(cfg.model, cfg.N, round_bf16=False)
    assert not np.array_equal(inp.flat, synth.round_to_bf16(inp.flat))
    ref = oracle_search(inp, cfg.N, cfg.T, cfg.tau, cfg.K_w, cfg.K_c)
    return cfg, inp, ref


def test_tiny_dit_forward_matches_oracle_on_compacted_subset(B, tiny):
    cfg, inp, _ = tiny
    m = inp.m
    model = B.Model(m, cfg.N)
    model.load_weights(inp.flat)
    model.set_text_context(dev(inp.ctx))
    x = dev(inp.x1.reshape(cfg.N, -1))
    v = torch.full((cfg.N, m.D), 7.0, device="cuda")
    idx = torch.tensor([0, 2, 3], dtype=torch.int32, device="cuda")
    model.dit_forward(x, idx, 3, 0.7, v)
    got = v.cpu().numpy()
    dit = O.DiT(m, inp.params)
    kv = dit.text_kv(inp.ctx)
    for i in (0, 2, 3):
        ref = dit.velocity(inp.x1[i], 0.7, kv).reshape(-1)
        assert np.abs(got[i] - ref).max() / np.abs(ref).max() < 2e-2
    assert np.all(got[1] == 7.0)          # rows not in the subset are untouched
    assert model.device_error() == 0
    model.close()


@pytest.mark.parametrize("weights", ["bf16-valued", "fp32"])
def test_tiny_search_free_running_matches_oracle(B, tiny, tiny_fp32, weights):
    cfg, inp, (xo, mo, so, pres) = tiny if weights == "bf16-valued" else tiny_fp32
    st, mg, sg, _ = gpu_search(B, inp, cfg.N, cfg.T, cfg.tau, cfg.K_w, cfg.K_c)
    for k in range(cfg.T):
        diff = mg[k] != mo[k]
        if diff.any():
            near = [pres[k][i] is not None and abs(pres[k][i] - cfg.tau) < 1e-3 for i in range(cfg.N)]
            assert all(near[i] for i in np.flatnonzero(diff)), f"mask differs at step {k + 1} outside the tie zone"
            pytest.skip(f"tie-zone decision at step {k + 1}; latents are checked by the replay test")
    g = st["x"].cpu().numpy().reshape(xo.shape)
    assert max_rel(g, xo) < 2e-2
    assert 0 < mo.sum() < mo.size            # the configuration really skips, but not everything
    assert int(np.argmax(sg)) == int(O.topk(so, 1)[0])


@pytest.mark.parametrize("weights", ["bf16-valued", "fp32"])
def test_tiny_search_mask_replay_matches_oracle(B, tiny, tiny_fp32, weights):
    cfg, inp, (xo, mo, so, _) = tiny if weights == "bf16-valued" else tiny_fp32
    st, mg, sg, _ = gpu_search(B, inp, cfg.N, cfg.T, cfg.tau, cfg.K_w, cfg.K_c, force_masks=~mo)
    assert np.array_equal(mg, mo)
    g = st["x"].cpu().numpy().reshape(xo.shape)
    assert max_rel(g, xo) < 2e-2
    np.testing.assert_allclose(sg, so, rtol=2e-2)
    idx = torch.zeros(cfg.N, dtype=torch.int32, device="cuda")
    B.select_topk(dev(sg), cfg.N, idx)
    assert idx.cpu().tolist() == O.topk(so, cfg.N).tolist()


# --------------------------------------------------- 1.3B width, small latent ----

@pytest.mark.parametrize("round_bf16", [True, False])
def test_wan13b_width_small_latent_matches_oracle(B, round_bf16):
    m = synth.replace_model(synth.WAN_1_3B, F=2, H=16, W=16, blocks=2)
    N, T, tau = 2, 3, 0.1
    inp = Inputs(m, N, round_bf16=round_bf16)
    xo, mo, so, _ = oracle_search(inp, N, T, tau, 1, 1)
    st, mg, sg, _ = gpu_search(B, inp, N, T, tau, 1, 1, force_masks=~mo)
    g = st["x"].cpu().numpy().reshape(xo.shape)
    assert max_rel(g, xo) < 2e-2
    np.testing.assert_allclose(sg, so, rtol=2e-2)


# ------------------------------------------------------- any-size properties ----

def test_batch_invariance_and_determinism_tiny(B, tiny):
    cfg, inp, _ = tiny
    st, mg, _, _ = gpu_search(B, inp, cfg.N, cfg.T, cfg.tau, cfg.K_w, cfg.K_c)
    st2, mg2, _, _ = gpu_search(B, inp, cfg.N, cfg.T, cfg.tau, cfg.K_w, cfg.K_c)
    assert torch.equal(st["x"], st2["x"]) and np.array_equal(mg, mg2)
    for i in range(cfg.N):
        one = Inputs.__new__(Inputs)
        one.__dict__.update(inp.__dict__)
        one.x1 = inp.x1[i:i + 1]
        s1, m1, _, _ = gpu_search(B, one, 1, cfg.T, cfg.tau, cfg.K_w, cfg.K_c)
        assert np.array_equal(m1[:, 0], mg[:, i])
        assert torch.equal(s1["x"][0], st["x"][i]), f"candidate {i} differs alone vs in the batch"


def test_tau_zero_equals_always_compute(B, tiny):
    cfg, inp, _ = tiny
    s0, m0, _, n0 = gpu_search(B, inp, cfg.N, cfg.T, 0.0, cfg.K_w, cfg.K_c)
    sf, mf, _, _ = gpu_search(B, inp, cfg.N, cfg.T, cfg.tau, cfg.K_w, cfg.K_c,
                              force_masks=np.ones((cfg.T, cfg.N), bool))
    assert not m0.any() and all(n == cfg.N for n in n0)
    assert torch.equal(s0["x"], sf["x"])


def _all_skip_closed_form(B, inp, model, N, T):
    m = inp.m
    st = B.new_state(N, m.D)
    st["x"].copy_(dev(inp.x1.reshape(N, -1)))
    t = O.time_grid(T)
    skip = torch.zeros(N, dtype=torch.uint8, device="cuda")
    model.search_step(st, 1, T, float(t[0]), float(t[1]), 1e30, 0, 0, skip)
    x2 = st["x"].double().cpu().numpy()
    delta = st["delta"].double().cpu().numpy()
    assert np.isfinite(x2).all() and np.isfinite(delta).all()
    for k in range(2, T + 1):
        n = model.search_step(st, k, T, float(t[k - 1]), float(t[k]), 1e30, 0, 0, skip)
        assert n == 0
    torch.cuda.synchronize()
    expect = -delta + np.prod(1 + np.diff(t)[1:]) * (x2 + delta)
    got = st["x"].double().cpu().numpy()
    np.testing.assert_allclose(got, expect, rtol=0, atol=1e-5 * np.abs(expect).max())
    assert model.device_error() == 0


def _model(B, inp, N):
    model = B.Model(inp.m, N)
    model.load_weights(inp.flat)
    model.set_text_context(dev(inp.ctx))
    return model


def test_all_skip_closed_form_tiny(B):
    inp = Inputs(synth.TINY, 4)
    model = _model(B, inp, 4)
    _all_skip_closed_form(B, inp, model, 4, 10)
    model.close()


def test_wan13b_full_size_properties(B):
    """1.3B shape at full size (30 blocks, 32760 tokens): one computed step then
    all-skip steps follow the closed form; a candidate alone equals itself in a batch
    of 4, bitwise."""
    m = synth.WAN_1_3B
    inp = Inputs(m, 4)
    model = _model(B, inp, 4)
    _all_skip_closed_form(B, inp, model, 4, 5)
    x = dev(inp.x1.reshape(4, -1))
    v4 = torch.zeros(4, m.D, device="cuda")
    v1 = torch.zeros(4, m.D, device="cuda")
    model.dit_forward(x, torch.arange(4, dtype=torch.int32, device="cuda"), 4, 0.9, v4)
    model.dit_forward(x, torch.tensor([2], dtype=torch.int32, device="cuda"), 1, 0.9, v1)
    torch.cuda.synchronize()
    assert torch.isfinite(v4).all()
    assert torch.equal(v1[2], v4[2])
    assert float(v4.std()) > 0.05
    assert model.device_error() == 0
    model.close()


def test_streamed_weight_loading_equals_flat_loading(B):
    m = synth.TINY
    inp = Inputs(m, 2)
    a = _model(B, inp, 2)
    b = B.Model(m, 2)
    b.load_streamed()
    b.set_text_context(dev(inp.ctx))
    x = dev(inp.x1.reshape(2, -1))
    idx = torch.arange(2, dtype=torch.int32, device="cuda")
    va, vb = torch.zeros(2, m.D, device="cuda"), torch.zeros(2, m.D, device="cuda")
    a.dit_forward(x, idx, 2, 0.4, va)
    b.dit_forward(x, idx, 2, 0.4, vb)
    torch.cuda.synchronize()
    assert torch.equal(va, vb)
    a.close()
    b.close()


def test_host_buffer_step_equals_device_step_tiny(B, tiny):
    """cs_search_step_host (latents and mask in pinned host memory, the path the bench's
    end-to-end number takes) gives the device-buffer step's latents and masks bit for bit."""
    cfg, inp, _ = tiny
    st_d, m_d, _, n_d = gpu_search(B, inp, cfg.N, cfg.T, cfg.tau, cfg.K_w, cfg.K_c, score=False)
    model = B.Model(cfg.model, cfg.N)
    model.load_weights(inp.flat)
    model.set_text_context(dev(inp.ctx))
    xh = torch.from_numpy(inp.x1.reshape(cfg.N, -1).copy()).pin_memory()
    skip_h = torch.zeros(cfg.N, dtype=torch.uint8).pin_memory()
    st = B.new_state(cfg.N, cfg.model.D)
    t = O.time_grid(cfg.T)
    masks, ncs = [], []
    for k in range(1, cfg.T + 1):
        ncs.append(model.search_step_host(xh, st, k, cfg.T, float(t[k - 1]), float(t[k]), cfg.tau, cfg.K_w, cfg.K_c,
                                          skip_h))
        masks.append(skip_h.numpy().astype(bool).copy())
    assert model.device_error() == 0
    model.close()
    assert ncs == n_d and np.array_equal(np.array(masks), m_d)
    assert torch.equal(xh, st_d["x"].cpu())


def test_kernel_stats_count_the_algorithmic_work(B, tiny):
    """The per-class counters behind the bench's roofline: with every candidate forced to
    compute, the GEMM, self- and cross-attention work equal the closed-form FLOPs of the
    DiT per candidate-step (QKV 6Ld^2 ... per block), the cache class counts its
    algorithmic bytes, and every class records launches and time."""
    cfg, inp, _ = tiny
    m, N, T = cfg.model, cfg.N, cfg.T
    model = B.Model(m, N)
    model.load_weights(inp.flat)
    model.set_text_context(dev(inp.ctx))
    st = B.new_state(N, m.D)
    st["x"].copy_(dev(inp.x1.reshape(N, -1)))
    skip = torch.zeros(N, dtype=torch.uint8, device="cuda")
    force = torch.ones(N, dtype=torch.uint8, device="cuda")
    t = O.time_grid(T)
    model.reset_kernel_stats()
    model.set_profiling(True)
    for k in range(1, T + 1):
        assert model.search_step(st, k, T, float(t[k - 1]), float(t[k]), cfg.tau, cfg.K_w, cfg.K_c, skip,
                                 force=force) == N
    model.set_profiling(False)
    stats = {c: model.kernel_stats(c) for c in range(5)}
    assert model.device_error() == 0
    model.close()
    L, d, hd, H, Lt, ffn, nb = m.L, m.d, m.hd, m.heads, m.Lt, m.ffn, m.blocks
    P = 4 * m.C
    Kp = (P + 63) // 64 * 64          # the patch embedding runs on zero-padded 64-wide rows
    cs = N * T                        # computed candidate-steps
    gemm = 2.0 * L * (d * Kp + nb * (6 * d * d + 2 * d * ffn) + P * d)
    assert stats[B.KC_GEMM][2] == cs * gemm
    assert stats[B.KC_SELF_ATTN][2] == cs * nb * 4.0 * H * L * L * hd
    assert stats[B.KC_CROSS_ATTN][2] == cs * nb * 4.0 * H * L * Lt * hd
    assert stats[B.KC_SELF_ATTN][0] == T * nb and stats[B.KC_CROSS_ATTN][0] == T * nb
    # cache bytes: computed candidates read x, v and write x, Delta, x_ref (20 D); a free
    # step whose drift was not carried over from the previous step also reads x_ref for the
    # drift (24 D): only a free first step (this workload's step 1 lies in the window)
    assert cfg.K_w >= 1
    assert stats[B.KC_CACHE][2] == float(m.D * N * 20 * T)
    for c in range(5):
        assert stats[c][0] > 0 and stats[c][1] > 0.0, c


def test_searches_of_changing_sizes_on_one_model(B):
    """The single-pass cache step keeps its per-candidate arrival counters in the model
    between steps; a model that has run searches of other sizes (larger and smaller)
    gives each search the same bits as a fresh model."""
    inp = Inputs(synth.TINY, 8)
    shared = _model(B, inp, 8)
    for N in (4, 6, 2, 8, 3):
        sub = Inputs.__new__(Inputs)
        sub.__dict__.update(inp.__dict__)
        sub.x1 = inp.x1[:N]
        s1, m1, sc1, n1 = gpu_search(B, sub, N, 10, 0.1, 1, 1, model=shared)
        fresh = _model(B, inp, 8)
        s2, m2, sc2, n2 = gpu_search(B, sub, N, 10, 0.1, 1, 1, model=fresh)
        fresh.close()
        assert n1 == n2 and np.array_equal(m1, m2), N
        assert torch.equal(s1["x"], s2["x"]) and np.array_equal(sc1, sc2), N
        assert 0 < m1.sum() < m1.size, N        # both kinds of decision occur
    shared.close()
