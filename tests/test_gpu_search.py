"""Search variants on the GPU against the fp64 oracle (tiny configuration):
static every-k schedule, beam rescoring with refill, pruned search, and the
full-compute commit of the winner (bitwise equal to its tau = 0 batched rollout)."""
import numpy as np
import pytest
import torch

from oracle import cachedsearch_oracle as O
from paper_2607_23159_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def env():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_23159_gb300 import binding as B, search as S
    m = synth.TINY
    flat, params = synth.make_params(m)
    ctx = synth.text_context(m)
    model = B.Model(m, 8)
    model.load_weights(flat)
    model.set_text_context(torch.from_numpy(ctx).cuda())
    dit = O.DiT(m, params)
    kv = dit.text_kv(ctx)
    vel = lambda z, t: dit.velocity(z, t, kv)
    y = synth.target_latent(m)
    srch = S.Search(model, 8, target=torch.from_numpy(y.reshape(-1)).cuda())
    yield B, S, m, vel, y, srch
    model.close()


def _x1(m, n):
    return synth.initial_noise(m, range(n))


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a.reshape(a.shape[0], -1))).cuda()


def _rel(g, o):
    return np.abs(g - o).max() / np.abs(o).max()


def test_static_schedule_matches_oracle(env):
    B, S, m, vel, y, srch = env
    T, every = 10, 3
    x1 = _x1(m, 4)
    win, sc, masks = srch.best_of_n(_dev(x1), T, 0.1, 1, 1, schedule_every=every)
    want = np.array([S.static_schedule(k, T, 1, 1, every) for k in range(1, T + 1)])
    assert np.array_equal(~masks, np.repeat(want[:, None], 4, axis=1))
    for i in range(4):
        xo, comp, _ = O.rollout_static(x1[i], T, 1, 1, every, vel)
        assert np.array_equal(comp, want)
        assert _rel(srch.st["x"][i].cpu().numpy().reshape(xo.shape), xo) < 2e-2


def test_beam_search_matches_oracle(env):
    B, S, m, vel, y, srch = env
    T, every, keep, children, sigma = 10, 3, 2, 1, 0.1
    x1 = _x1(m, 4)
    rounds = [synth.beam_noise(m, r, keep, children) for r in range(3)]
    so, xo, mo = O.beam_search(x1, T, 0.1, 1, 1, vel, y, every, keep, children, sigma, lambda r: rounds[r])
    best, sg = srch.beam(_dev(x1), T, 0.1, 1, 1, every, keep, children, sigma,
                         [_dev(n) for n in rounds])
    np.testing.assert_allclose(sg, so, rtol=2e-2)
    assert best == int(O.topk(so, 1)[0])
    g = srch.st["x"].cpu().numpy().reshape(xo.shape)
    assert max(_rel(g[i], xo[i]) for i in range(len(xo))) < 2e-2


def test_pruned_search_matches_oracle(env):
    B, S, m, vel, y, srch = env
    T, prune_step, keep = 10, 4, 2
    x1 = _x1(m, 6)
    win_o, so, ids_o, xo = O.pruned_search(x1, T, 0.1, 1, 1, vel, y, prune_step, keep)
    win_g, sg, ids_g = srch.pruned(_dev(x1), T, 0.1, 1, 1, prune_step, keep)
    assert ids_g.tolist() == ids_o.tolist()
    assert win_g == win_o
    np.testing.assert_allclose(sg, so, rtol=2e-2)


def test_commit_regenerates_the_winner_bitwise(env):
    B, S, m, vel, y, srch = env
    T = 10
    x1 = _x1(m, 4)
    win, _, _ = srch.best_of_n(_dev(x1), T, 0.1, 1, 1)
    # the tau = 0 batched rollout of every candidate ...
    srch.best_of_n(_dev(x1), T, 0.0, 1, 1)
    batched = srch.st["x"][win].clone()
    # ... equals the winner regenerated alone at full compute, bit for bit
    alone = srch.commit(_dev(x1[win:win + 1]), T, 1, 1)
    assert torch.equal(alone, batched)
    xo = O.commit(x1[win], T, vel)
    assert _rel(alone.cpu().numpy().reshape(xo.shape), xo) < 2e-2
