"""Host orchestration of the search drivers (no GPU).

``paper_2607_23159_gb300.search.Search`` only sequences library calls: which step scores,
when the beam refills, how slots map back to original candidates, which buffer holds the
live state.  Here its three device calls (the step, top-k, beam refill) are replaced by
the CPU oracle working on the same state tensors, so that the drivers' bookkeeping can be
compared with the oracle's own search loops (Algorithm 1; beam and pruned search; the
static schedule; the commit branch).
"""
import numpy as np
import pytest
import torch

from oracle import cachedsearch_oracle as O

T, TAU, K_W, K_C = 12, 0.3, 2, 2
SHAPE = (2, 3, 4)              # a small latent [C, F, W]; the loops never look inside it
D = int(np.prod(SHAPE))


def velocity(x, t):
    """A smooth nonlinear field, so that drifts and scores differ between candidates."""
    return np.tanh(x) * (1.0 + t) - 0.5 * x + 0.2


@pytest.fixture(scope="module")
def S():
    import __graft_entry__
    __graft_entry__.build()             # the binding module loads the library on import
    from paper_2607_23159_gb300 import search
    return search


class _OracleModel:
    """Stands in for binding.Model: one oracle step over the state tensors, in place."""

    class mcfg:
        D = D

    def search_step(self, st, k, T_, t_cur, t_next, tau, K_w, K_c, skip, force=None, target=None, scores=None):
        n = st["x"].shape[0]
        states = [O.CacheState(st["delta"][i].numpy().reshape(SHAPE).copy() if st["has_ref"][i] else None,
                               st["x_ref"][i].numpy().reshape(SHAPE).copy() if st["has_ref"][i] else None,
                               float(st["accum"][i])) for i in range(n)]
        xs = st["x"].numpy().reshape(n, *SHAPE)
        f = None if force is None else force.numpy().astype(bool)
        tgt = None if target is None else target.numpy().reshape(SHAPE)
        out, skipped, _, sc = O.search_step(states, xs, k, T_, tau, K_w, K_c, velocity, force=f, target=tgt)
        for i, s in enumerate(states):
            st["x"][i] = torch.from_numpy(out[i].reshape(-1))
            st["x_ref"][i] = torch.from_numpy(s.x_ref.reshape(-1))
            st["delta"][i] = torch.from_numpy(s.delta.reshape(-1))
            st["accum"][i] = s.a
            st["has_ref"][i] = 1
        skip.copy_(torch.from_numpy(skipped.astype(np.uint8)))
        if scores is not None:
            scores.copy_(torch.from_numpy(sc))
        return int((~skipped).sum())


def _new_state(N, D_, device="cpu"):
    return {k: torch.zeros(N, D_, dtype=torch.float64) for k in ("x", "x_ref", "delta")} | {
        "accum": torch.zeros(N, dtype=torch.float64), "has_ref": torch.zeros(N, dtype=torch.uint8)}


def _select_topk(scores, k, idx, stream=None):
    idx[:k] = torch.from_numpy(O.topk(scores.numpy(), k).astype(np.int32))


def _beam_refill(src, dst, survivors, children, sigma, noise, stream=None):
    n = src["x"].shape[0]
    states = [O.CacheState(src["delta"][i].numpy().copy(), src["x_ref"][i].numpy().copy(), float(src["accum"][i]))
              for i in range(n)]
    surv = [int(s) for s in survivors]
    new_states, new_x = O.beam_refill(states, src["x"].numpy(), surv, children, sigma,
                                      None if noise is None else noise.numpy())
    for j, s in enumerate(new_states):
        dst["x"][j] = torch.from_numpy(new_x[j])
        dst["x_ref"][j] = torch.from_numpy(s.x_ref)
        dst["delta"][j] = torch.from_numpy(s.delta)
        dst["accum"][j] = s.a
        dst["has_ref"][j] = src["has_ref"][surv[j // (children + 1)]]


def _search(S, monkeypatch, max_n, target):
    monkeypatch.setattr(S.B, "new_state", _new_state)
    monkeypatch.setattr(S.B, "select_topk", _select_topk)
    monkeypatch.setattr(S.B, "beam_refill", _beam_refill)
    s = S.Search(_OracleModel(), max_n, target=torch.from_numpy(target.reshape(-1)), device="cpu")
    s.scores = torch.zeros(max_n, dtype=torch.float64)
    return s


def _inputs(n, seed=0):
    rng = np.random.default_rng(seed)
    return rng.standard_normal((n, *SHAPE)), rng.standard_normal(SHAPE)


def test_best_of_n_matches_algorithm_1(S, monkeypatch):
    x1, y = _inputs(5)
    s = _search(S, monkeypatch, 5, y)
    win, scores, masks = s.best_of_n(torch.from_numpy(x1.reshape(5, -1)), T, TAU, K_W, K_C)
    i_star, sc, _, comp = O.cached_search(x1, T, TAU, K_W, K_C, velocity, y)
    assert win == i_star
    np.testing.assert_allclose(scores, sc, rtol=1e-12)
    assert np.array_equal(masks, ~comp.T)
    assert masks.any() and not masks.all()


def test_static_schedule_and_forced_masks(S, monkeypatch):
    x1, y = _inputs(3, seed=1)
    s = _search(S, monkeypatch, 3, y)
    _, _, masks = s.best_of_n(torch.from_numpy(x1.reshape(3, -1)), T, TAU, K_W, K_C, schedule_every=3)
    for i in range(3):
        _, comp, _ = O.rollout_static(x1[i], T, K_W, K_C, 3, velocity)
        assert np.array_equal(masks[:, i], ~comp)
    # a replayed per-step mask is applied as given
    rng = np.random.default_rng(2)
    forces = rng.integers(0, 2, size=(T, 3)).astype(np.uint8)
    forces[0] = 1                                   # the first call must compute
    _, _, masks = s.best_of_n(torch.from_numpy(x1.reshape(3, -1)), T, TAU, K_W, K_C,
                              forces=[torch.from_numpy(f) for f in forces])
    assert np.array_equal(masks, forces == 0)


def test_beam_tracks_slots_like_the_oracle(S, monkeypatch):
    N, every, keep, children, sigma = 6, 4, 2, 2, 0.1
    x1, y = _inputs(N, seed=3)
    rounds = (T - 1) // every
    rng = np.random.default_rng(4)
    noise = [rng.standard_normal((keep * children, D)) for _ in range(rounds)]
    s = _search(S, monkeypatch, N, y)
    best, scores = s.beam(torch.from_numpy(x1.reshape(N, -1)), T, TAU, K_W, K_C, every, keep, children, sigma,
                          [torch.from_numpy(z) for z in noise])
    sc, xs, _ = O.beam_search(x1, T, TAU, K_W, K_C, velocity, y, every, keep, children, sigma,
                              lambda r: noise[r].reshape(keep * children, *SHAPE))
    assert s.n == keep * (children + 1)
    np.testing.assert_allclose(scores, sc, rtol=1e-12)
    assert best == int(O.topk(sc, 1)[0])
    np.testing.assert_allclose(s.st["x"].numpy(), xs.reshape(len(xs), -1), rtol=1e-12)
    # each final slot's original candidate: survivors' ancestors, repeated for their children
    states, xo, anc = [O.CacheState() for _ in range(N)], x1, np.arange(N)
    for k in range(1, T + 1):
        refill = k % every == 0 and k < T
        xo, _, _, sc_k = O.search_step(states, xo, k, T, TAU, K_W, K_C, velocity, target=y if refill else None)
        if refill:
            surv = last = O.topk(sc_k, keep)
            states, xo = O.beam_refill(states, xo, list(surv), children, sigma,
                                       noise[k // every - 1].reshape(keep * children, *SHAPE))
            anc = np.repeat(anc[surv], children + 1)
    assert rounds >= 2 and np.array_equal(s.ids, anc)
    assert not np.array_equal(anc, np.repeat(last, children + 1))   # the lineage is not the last round's slots


def test_pruned_search_maps_survivors_to_original_candidates(S, monkeypatch):
    N, prune_step, keep = 6, 5, 3
    x1, y = _inputs(N, seed=5)
    s = _search(S, monkeypatch, N, y)
    win, scores, ids = s.pruned(torch.from_numpy(x1.reshape(N, -1)), T, TAU, K_W, K_C, prune_step, keep)
    o_win, o_sc, o_ids, _ = O.pruned_search(x1, T, TAU, K_W, K_C, velocity, y, prune_step, keep)
    assert win == o_win
    assert np.array_equal(ids, o_ids)
    assert sorted(ids.tolist()) != list(range(keep))   # the survivors are not simply the first slots
    np.testing.assert_allclose(scores, o_sc, rtol=1e-12)


def test_commit_is_the_uncached_rollout(S, monkeypatch):
    x1, y = _inputs(1, seed=6)
    s = _search(S, monkeypatch, 1, y)
    x = s.commit(torch.from_numpy(x1.reshape(1, -1)), T, K_W, K_C)
    assert np.array_equal(x.numpy().reshape(SHAPE), O.commit(x1[0], T, velocity))
