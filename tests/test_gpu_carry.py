"""The carried form of the cache step (GPU): every update leaves the next step's drift sums
(Sec. 3.1, Eq. indicator), so that a step decides without reading x and x_ref.

* full 1.3B latent (N 4) and short-clip latent (N 8): a window step, then free steps
  whose decisions come from the carried sums, every element against the oracle's wrapper
  step and against the drift-pass form (cs_cache_decide_skip + cs_cache_apply_tokens) on
  a second copy of the state: the same masks and latent bits, accum to float32 rounding;
* a cached candidate without a carried drift (has_ref = 1): the carried call changes
  nothing and reports -1, the drift-pass call then gives the oracle's step;
* through the model: searches interleaved on one model (each call finds the other's
  buffers, so no drift is carried) equal the same searches run alone (carried), and an
  outside write that clears the carried bit equals the same write on a copied state.
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


def _tokens(m, k, i, scale):
    """Head output (token layout [L][4C]) of candidate i at step k."""
    return (synth.normal(1000 * k + i, (m.L, 4 * m.C)) * scale).astype(np.float32)


def _new(B, N, D, x):
    st = B.new_state(N, D)
    st["x"].copy_(dev(x))
    return st


@pytest.mark.parametrize("m,N", [(synth.WAN_1_3B, 4), (synth.WAN_1_3B_SHORT, 8)])
def test_carried_steps_match_oracle_and_drift_pass_form(B, m, N):
    T, tau, K = 50, 0.1, 5
    D, L = m.D, m.L
    lat = (m.C, m.F, m.H, m.W)
    t = O.time_grid(T)
    # velocity scales: drift of a just-computed candidate ~ |h| * scale = 0.02 * scale
    scale = np.tile([1.0, 8.0, 2.5, 12.0], N // 4)
    x0 = synth.normal(71, (N, D))
    y = synth.normal(72, (D,))
    gpu = [_new(B, N, D, x0), _new(B, N, D, x0)]     # carried form, drift-pass form
    ws = torch.zeros(B.cache_step_bytes(N, *lat) // 4 + 1, device="cuda")
    ws_old = torch.zeros(B.cache_workspace_bytes(N, D) // 4 + 1, device="cuda")
    tp = torch.zeros(N, m.F * m.H // 2, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    states = [O.CacheState() for _ in range(N)]
    xo = x0.astype(np.float64)
    computed_kinds = set()
    for k in range(K, K + 5):                        # step 5 in the warm-up window, then free steps
        score = k == K + 4
        tgt = dev(y) if score else None
        out = []
        for which, st in enumerate(gpu):
            skip = torch.zeros(N, dtype=torch.uint8, device="cuda")
            idx = torch.zeros(N, dtype=torch.int32, device="cuda")
            nc = torch.zeros(1, dtype=torch.int32, device="cuda")
            sc = torch.zeros(N, device="cuda")
            if which == 0:
                B.cache_decide_skip_carry(st, lat, k, T, float(t[k - 1]), float(t[k]), tau, K, K, skip, idx, nc, ws,
                                          carried=True, target=tgt, err=err)
            else:
                B.cache_decide_skip(st["x"], st["x_ref"], st["delta"], st["accum"], st["has_ref"], k, T,
                                    float(t[k - 1]), float(t[k]), tau, K, K, skip, idx, nc, ws_old, target=tgt,
                                    err=err)
            torch.cuda.synchronize()
            n_c = int(nc[0])
            assert n_c >= 0
            comp = idx[:n_c].cpu().numpy()
            hout = dev(np.concatenate([_tokens(m, k, i, scale[i]) for i in comp])) if n_c else \
                torch.zeros(1, device="cuda")
            if which == 0:
                B.cache_apply_tokens_carry(st, skip, hout, idx, n_c, lat, k, float(t[k - 1]), float(t[k]), ws,
                                           target=tgt, scores=sc if score else None, err=err)
            else:
                B.cache_apply_tokens(st, skip, hout, idx, n_c, *lat, float(t[k - 1]), float(t[k]), workspace=ws_old,
                                     target=tgt, scores=sc if score else None, tile_partials=tp, err=err)
            torch.cuda.synchronize()
            assert int(err[0]) == 0
            out.append((skip.cpu().numpy().astype(bool), sc.cpu().numpy()))
        (m0, sc0), (m1, sc1) = out
        # oracle: the wrapper step with the same per-candidate velocities
        pre = [None if O.forced_compute(k, T, K, K, s.has_ref) else s.a + O.relative_drift(xo[i], s.x_ref)
               for i, s in enumerate(states)]
        xs, so, sk = [], [], []
        for i in range(N):
            vi = O.unpatchify(_tokens(m, k, i, scale[i]).astype(np.float64), *lat).reshape(-1)
            vel, c, _ = O.wrapper_call(states[i], xo[i], k, T, tau, K, K, lambda z: vi)
            xn = O.euler(xo[i], t[k - 1], t[k], vel)
            xs.append(xn)
            sk.append(not c)
            so.append(O.score(xn - t[k] * vel, y))
        xo = np.stack(xs)
        for p in pre:
            assert p is None or abs(p - tau) > 1e-3, (k, pre)   # no decision inside the tie zone
        assert m0.tolist() == sk and np.array_equal(m0, m1), (k, m0, m1, sk)
        computed_kinds.update(sk)
        g0, g1 = gpu
        for key in ("x", "x_ref", "delta"):
            assert torch.equal(g0[key], g1[key]), (k, key)
        np.testing.assert_allclose(g0["x"].cpu().numpy(), xo, rtol=1e-5, atol=1e-5)
        np.testing.assert_allclose(g0["accum"].cpu().numpy(), [s.a for s in states], rtol=1e-5, atol=1e-7)
        np.testing.assert_allclose(g0["accum"].cpu().numpy(), g1["accum"].cpu().numpy(), rtol=1e-6, atol=1e-9)
        # every candidate now carries its drift; the drift-pass form leaves 1
        assert g0["has_ref"].cpu().tolist() == [3] * N and g1["has_ref"].cpu().tolist() == [1] * N
        if score:
            np.testing.assert_allclose(sc0, so, rtol=1e-5)
            np.testing.assert_allclose(sc0, sc1, rtol=1e-6)
    assert computed_kinds == {True, False}           # both decisions were taken on carried drifts


def test_missing_carried_drift_changes_nothing_then_drift_pass(B):
    m = synth.TINY
    N, T, tau, K = 4, 10, 0.1, 1
    D = m.D
    lat = (m.C, m.F, m.H, m.W)
    t = O.time_grid(T)
    x0 = synth.normal(81, (N, D))
    st = _new(B, N, D, x0)
    ws = torch.zeros(B.cache_step_bytes(N, *lat) // 4 + 1, device="cuda")
    skip = torch.zeros(N, dtype=torch.uint8, device="cuda")
    idx = torch.zeros(N, dtype=torch.int32, device="cuda")
    nc = torch.zeros(1, dtype=torch.int32, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    scale = [0.3, 10.0, 0.5, 12.0]   # drift at step 2 ~ 0.1 * scale: 0.03, 1.0, 0.05, 1.2
    hout = dev(np.concatenate([_tokens(m, 1, i, scale[i]) for i in range(N)]))
    # step 1 (window): every candidate computes and carries its drift
    B.cache_decide_skip_carry(st, lat, 1, T, float(t[0]), float(t[1]), tau, K, K, skip, idx, nc, ws, carried=True,
                              err=err)
    B.cache_apply_tokens_carry(st, skip, hout, idx, N, lat, 1, float(t[0]), float(t[1]), ws, err=err)
    torch.cuda.synchronize()
    st["has_ref"][2] = 1                                # candidate 2's state written outside the calls
    before = {k_: v.clone() for k_, v in st.items()}
    skip.fill_(7)
    B.cache_decide_skip_carry(st, lat, 2, T, float(t[1]), float(t[2]), tau, K, K, skip, idx, nc, ws, carried=True,
                              err=err)
    torch.cuda.synchronize()
    assert int(nc[0]) == -1 and int(err[0]) == 0
    for k_ in before:
        assert torch.equal(before[k_], st[k_]), k_
    assert skip.cpu().tolist() == [7] * N
    B.cache_decide_skip_carry(st, lat, 2, T, float(t[1]), float(t[2]), tau, K, K, skip, idx, nc, ws, carried=False,
                              err=err)
    torch.cuda.synchronize()
    assert int(err[0]) == 0
    # oracle: step 1 computes everything, step 2 decides from x and x_ref
    states = [O.CacheState() for _ in range(N)]
    want = []
    for i in range(N):
        v1 = O.unpatchify(_tokens(m, 1, i, scale[i]).astype(np.float64), *lat).reshape(-1)
        O.wrapper_call(states[i], x0[i], 1, T, tau, K, K, lambda z: v1)
        x1 = O.euler(x0[i].astype(np.float64), t[0], t[1], v1)
        _, c, _ = O.wrapper_call(states[i], x1, 2, T, tau, K, K, lambda z: None)
        want.append(not c)
    assert skip.cpu().numpy().astype(bool).tolist() == want
    assert want == [True, False, True, False]
    np.testing.assert_allclose(st["accum"].cpu().numpy(), [s.a for s in states], rtol=1e-5, atol=1e-7)
    assert st["has_ref"].cpu().tolist() == [3, 1, 3, 1]   # skipped ones carry again; computed ones wait for the update


# ------------------------------------------------------------- through the model ----

def _model(B, m, N):
    flat, _ = synth.make_params(m)
    model = B.Model(m, N)
    model.load_weights(flat)
    model.set_text_context(dev(synth.text_context(m)))
    return model


def test_interleaved_searches_equal_solo_runs(B):
    """Two searches alternating steps on one model never find their own buffers in the
    previous call, so every free step takes the drift pass; run alone, each carries its
    drift.  Masks and latents agree bit for bit."""
    cfg = synth.CONFIGS["tiny"]
    m, N, T = cfg.model, cfg.N, cfg.T
    t = O.time_grid(T)
    x1 = [synth.initial_noise(m, range(N)).reshape(N, -1), synth.initial_noise(m, range(N, 2 * N)).reshape(N, -1)]

    def run(model, sts, order):
        masks = [[], []]
        skip = torch.zeros(N, dtype=torch.uint8, device="cuda")
        for k in range(1, T + 1):
            for s in order:
                model.search_step(sts[s], k, T, float(t[k - 1]), float(t[k]), cfg.tau, cfg.K_w, cfg.K_c, skip)
                masks[s].append(skip.cpu().numpy().astype(bool))
        return [np.array(mk) for mk in masks]

    model = _model(B, m, N)
    inter = [_new(B, N, m.D, x1[0]), _new(B, N, m.D, x1[1])]
    mi = run(model, inter, (0, 1))
    solo = [_new(B, N, m.D, x1[0]), _new(B, N, m.D, x1[1])]
    ms = [run(model, [solo[0], None], (0,))[0], run(model, [None, solo[1]], (1,))[1]]
    assert model.device_error() == 0
    model.close()
    for s in (0, 1):
        assert np.array_equal(mi[s], ms[s]), s
        assert 0 < ms[s].sum() < ms[s].size, s                  # both decisions occur
        assert torch.equal(inter[s]["x"], solo[s]["x"]), s
        np.testing.assert_allclose(inter[s]["accum"].cpu().numpy(), solo[s]["accum"].cpu().numpy(), rtol=1e-6,
                                   atol=1e-9)


def test_outside_write_with_cleared_bit_equals_copied_state(B):
    """An outside change of one candidate's latent between steps, with bit 1 of its has_ref
    cleared as the contract asks, gives the same search as making that change on a copy of
    the state (new buffers: nothing is carried)."""
    cfg = synth.CONFIGS["tiny"]
    m, N, T = cfg.model, cfg.N, cfg.T
    t = O.time_grid(T)
    x1 = synth.initial_noise(m, range(N)).reshape(N, -1)
    bump = dev(synth.normal(91, (m.D,)) * 0.05)
    model = _model(B, m, N)
    skip = torch.zeros(N, dtype=torch.uint8, device="cuda")
    runs = []
    for copy in (False, True):
        st = _new(B, N, m.D, x1)
        masks = []
        for k in range(1, T + 1):
            if k == 5:
                if copy:
                    st = {k_: v.clone() for k_, v in st.items()}
                st["x"][2] += bump
                st["has_ref"][2] = st["has_ref"][2] & 1
            model.search_step(st, k, T, float(t[k - 1]), float(t[k]), cfg.tau, cfg.K_w, cfg.K_c, skip)
            masks.append(skip.cpu().numpy().astype(bool))
        runs.append((st, np.array(masks)))
    assert model.device_error() == 0
    model.close()
    (s0, m0), (s1, m1) = runs
    assert np.array_equal(m0, m1)
    for key in ("x", "x_ref", "delta", "accum", "has_ref"):
        assert torch.equal(s0[key], s1[key]), key


@pytest.mark.parametrize("m,N", [(synth.TINY, 4), (synth.WAN_1_3B_SHORT, 4)])
def test_both_decision_modes_give_drift_pass_latents(B, m, N):
    """One window step that leaves every candidate's drift, then a free step three ways:
    decisions from the carried drift (one launch), the drift pass followed by the carrying
    skip update, and the drift-pass form of cs_cache_decide_skip: the same masks and latent
    bits, and both carrying forms leave the same carried decisions for the next step."""
    T, tau, K = 10, 0.1, 1
    D = m.D
    lat = (m.C, m.F, m.H, m.W)
    t = O.time_grid(T)
    scale = [0.3, 10.0, 0.5, 12.0]
    x0 = synth.normal(85, (N, D))
    hout1 = dev(np.concatenate([_tokens(m, 1, i, scale[i]) for i in range(N)]))
    idx_all = torch.arange(N, dtype=torch.int32, device="cuda")
    sts, wss = [], []
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    for _ in range(3):
        st = _new(B, N, D, x0)
        ws = torch.zeros(B.cache_step_bytes(N, *lat) // 4 + 1, device="cuda")
        skip = torch.zeros(N, dtype=torch.uint8, device="cuda")
        B.cache_apply_tokens_carry(st, skip, hout1, idx_all, N, lat, 1, float(t[0]), float(t[1]), ws, err=err)
        sts.append(st)
        wss.append(ws)
    torch.cuda.synchronize()
    for st in sts[1:]:
        assert torch.equal(st["x"], sts[0]["x"])
    masks, ncs = [], []
    for which, (st, ws) in enumerate(zip(sts, wss)):
        skip = torch.zeros(N, dtype=torch.uint8, device="cuda")
        idx = torch.zeros(N, dtype=torch.int32, device="cuda")
        nc = torch.zeros(1, dtype=torch.int32, device="cuda")
        if which < 2:
            B.cache_decide_skip_carry(st, lat, 2, T, float(t[1]), float(t[2]), tau, K, K, skip, idx, nc, ws,
                                      carried=which == 0, err=err)
        else:
            st["has_ref"].fill_(1)
            old = torch.zeros(B.cache_workspace_bytes(N, D) // 4 + 1, device="cuda")
            B.cache_decide_skip(st["x"], st["x_ref"], st["delta"], st["accum"], st["has_ref"], 2, T, float(t[1]),
                                float(t[2]), tau, K, K, skip, idx, nc, old, err=err)
        torch.cuda.synchronize()
        assert int(err[0]) == 0, which
        masks.append(skip.cpu().tolist())
        ncs.append(int(nc[0]))
    assert masks[0] == masks[1] == masks[2] == [1, 0, 1, 0], masks
    assert ncs == [2, 2, 2]
    for which in (1, 2):
        assert torch.equal(sts[which]["x"], sts[0]["x"]), which
    assert sts[0]["has_ref"].cpu().tolist() == sts[1]["has_ref"].cpu().tolist() == [3, 1, 3, 1]
