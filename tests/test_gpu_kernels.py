"""Parity of the individual sm_103a kernels with the fp64 oracle (GPU).

Inputs are seeded and synthetic; GEMM operands are bf16-representable, so the GEMM is
compared with the oracle's exact Linear and only the fp32 accumulation / bf16 output
rounding separates them.  Sizes span several tiles and leave ragged tails."""
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
    torch.cuda.init()
    return binding


def bf(a):
    return synth.round_to_bf16(np.asarray(a, np.float32))


def dev(a, dtype=torch.float32):
    return torch.from_numpy(np.ascontiguousarray(a)).to("cuda").to(dtype)


def err_word():
    return torch.zeros(4, dtype=torch.int32, device="cuda")


# ------------------------------------------------------------------- GEMM ----

@pytest.mark.parametrize("M,N,K", [(300, 384, 128), (513, 640, 192), (128, 1536, 64), (77, 16, 128)])
def test_gemm_epilogues_match_oracle_linear(B, M, N, K):
    A = bf(synth.normal(100 + M, (M, K)))
    W = bf(synth.normal(200 + N, (N, K)) * 0.1)
    bias = synth.normal(300 + N, (N,))
    ref = O.linear(A, W, bias)
    scale = np.abs(ref).max()
    err = err_word()
    Ad, Wd = dev(A, torch.bfloat16), dev(W, torch.bfloat16)
    out = torch.empty(M, N, device="cuda")
    B.gemm(Ad, Wd, B.EPI_F32, out, bias=dev(bias), err=err)
    np.testing.assert_allclose(out.cpu().numpy(), ref, rtol=0, atol=2e-5 * scale)
    outb = torch.empty(M, N, device="cuda", dtype=torch.bfloat16)
    B.gemm(Ad, Wd, B.EPI_BF16, outb, bias=dev(bias), err=err)
    np.testing.assert_allclose(outb.float().cpu().numpy(), ref, rtol=2 ** -8, atol=1e-5 * scale)
    B.gemm(Ad, Wd, B.EPI_GELU_BF16, outb, bias=dev(bias), err=err)
    np.testing.assert_allclose(outb.float().cpu().numpy(), O.gelu_tanh(ref), rtol=2 ** -8, atol=1e-4 * scale)
    res0 = synth.normal(400, (M, N))
    gate = synth.normal(401, (N,))
    res = dev(res0)
    B.gemm(Ad, Wd, B.EPI_RESID_F32, res, bias=dev(bias), gate=dev(gate), err=err)
    np.testing.assert_allclose(res.cpu().numpy(), res0 + gate * ref, rtol=0, atol=4e-5 * scale * np.abs(gate).max())
    res = dev(res0)
    B.gemm(Ad, Wd, B.EPI_RESID_F32, res, bias=dev(bias), gate=None, err=err)
    np.testing.assert_allclose(res.cpu().numpy(), res0 + ref, rtol=0, atol=4e-5 * scale)
    torch.cuda.synchronize()
    assert int(err[0]) == 0


@pytest.mark.parametrize("M,N,K", [(1, 512, 64), (129, 544, 128), (257, 520, 64), (1000, 800, 320),
                                   (255, 1024, 64), (383, 2560, 128)])
def test_gemm_cluster_pairs_ragged_shapes(B, M, N, K):
    """N >= 512 runs on clusters of two CTAs (one M = 256 MMA per pair): odd tile counts leave
    the second CTA of the last pair without rows, N tails leave half a B tile out of range, and
    N % 32 != 0 takes the non-TMA epilogue.  float32 and residual outputs against the oracle."""
    A = bf(synth.normal(500 + M, (M, K)))
    W = bf(synth.normal(600 + N, (N, K)) * 0.1)
    bias = synth.normal(700 + N, (N,))
    ref = O.linear(A, W, bias)
    scale = np.abs(ref).max()
    err = err_word()
    Ad, Wd = dev(A, torch.bfloat16), dev(W, torch.bfloat16)
    out = torch.full((M, N), 7.0, device="cuda")
    B.gemm(Ad, Wd, B.EPI_F32, out, bias=dev(bias), err=err)
    np.testing.assert_allclose(out.cpu().numpy(), ref, rtol=0, atol=2e-5 * scale)
    res0 = synth.normal(800, (M, N))
    res = dev(res0)
    B.gemm(Ad, Wd, B.EPI_RESID_F32, res, bias=dev(bias), gate=None, err=err)
    np.testing.assert_allclose(res.cpu().numpy(), res0 + ref, rtol=0, atol=4e-5 * scale)
    torch.cuda.synchronize()
    assert int(err[0]) == 0


@pytest.mark.parametrize("hd,heads,L,nb", [(128, 2, 200, 3), (32, 4, 48, 2)])
def test_gemm_qkv_scatter_layout(B, hd, heads, L, nb):
    d = hd * heads
    M, K = nb * L, 128
    A = bf(synth.normal(11, (M, K)))
    W = bf(synth.normal(12, (3 * d, K)) * 0.1)
    bias = synth.normal(13, (3 * d,))
    ref = O.linear(A, W, bias)
    hds, Lv = max(hd, 64), (L + 7) // 8 * 8
    q = torch.zeros(nb * heads, L, hds, device="cuda", dtype=torch.bfloat16)
    k = torch.zeros_like(q)
    vt = torch.zeros(nb * heads, hd, Lv, device="cuda", dtype=torch.bfloat16)
    B.gemm_qkv(dev(A, torch.bfloat16), dev(W, torch.bfloat16), dev(bias), L, d, heads, 0, q, k, vt, Lv)
    r = ref.reshape(nb, L, 3, heads, hd)
    tol = dict(rtol=2 ** -8, atol=1e-5 * np.abs(ref).max())
    qe = r[:, :, 0].transpose(0, 2, 1, 3).reshape(nb * heads, L, hd)
    ke = r[:, :, 1].transpose(0, 2, 1, 3).reshape(nb * heads, L, hd)
    ve = r[:, :, 2].transpose(0, 2, 3, 1).reshape(nb * heads, hd, L)
    np.testing.assert_allclose(q.float().cpu().numpy()[:, :, :hd], qe, **tol)
    np.testing.assert_allclose(k.float().cpu().numpy()[:, :, :hd], ke, **tol)
    np.testing.assert_allclose(vt.float().cpu().numpy()[:, :, :L], ve, **tol)
    if hds > hd:   # padding columns stay zero
        assert float(q.float()[:, :, hd:].abs().max()) == 0.0


# -------------------------------------------------------------- attention ----

def _attn_case(B, hd, heads, nb, Lq, Lk, kv_shared, qscale, seed, kramp=0.0):
    hds = max(hd, 64)
    Lks = (Lk + 7) // 8 * 8
    nkv = heads if kv_shared else nb * heads
    q = np.zeros((nb * heads, Lq, hds), np.float32)
    k = np.zeros((nkv, Lk, hds), np.float32)
    q[:, :, :hd] = bf(synth.normal(seed, (nb * heads, Lq, hd)) * qscale)
    # kramp > 0 scales the keys up along the sequence, so that the running row max keeps
    # growing from tile to tile and the lazy O rescale fires on most tiles
    kscale = 1.0 + kramp * np.arange(Lk, dtype=np.float32)[None, :, None] / max(Lk, 1)
    k[:, :, :hd] = bf(synth.normal(seed + 1, (nkv, Lk, hd)) * kscale)
    v = bf(synth.normal(seed + 2, (nkv, Lk, hd)))
    vt = np.zeros((nkv, hd, Lks), np.float32)
    vt[:, :, :Lk] = v.transpose(0, 2, 1)
    o = torch.zeros(nb, Lq, heads * hd, device="cuda", dtype=torch.bfloat16)
    err = err_word()
    B.attention(dev(q, torch.bfloat16), dev(k, torch.bfloat16), dev(vt, torch.bfloat16), o, nb, heads, Lq, Lk, hd,
                Lks, kv_shared, err=err)
    got = o.float().cpu().numpy()
    torch.cuda.synchronize()
    assert int(err[0]) == 0
    return q, k, v, got


@pytest.mark.parametrize("hd,heads,nb,Lq,Lk,kv_shared,qscale", [
    (128, 2, 2, 300, 200, False, 1.0),     # ragged queries and keys, 2 key tiles
    (128, 1, 1, 257, 1000, False, 3.0),    # peaked softmax: running max changes, lazy rescale
    (128, 3, 2, 130, 512, True, 1.0),      # cross-attention: K/V shared by all batch items
    (128, 2, 2, 520, 3000, False, 2.0),    # persistent form on a longer key loop (3 items per batch item)
    (32, 4, 4, 48, 48, False, 1.0),        # tiny model shape (one partial tile)
    (32, 4, 2, 48, 16, True, 2.0),         # tiny cross-attention, 16 text tokens
    (128, 2, 1, 1, 129, False, 1.0),       # one query row; the last key tile holds one key
    (128, 2, 2, 256, 1, False, 1.0),       # a single key: one tile, one valid column
    (128, 1, 2, 300, 8300, False, 1.0),    # more than 8192 keys: one item per CTA, ragged rows and keys
])
def test_attention_matches_oracle(B, hd, heads, nb, Lq, Lk, kv_shared, qscale):
    q, k, v, got = _attn_case(B, hd, heads, nb, Lq, Lk, kv_shared, qscale, seed=hd + Lq + Lk)
    for j in range(nb):
        for h in range(heads):
            bh, bkv = j * heads + h, (h if kv_shared else j * heads + h)
            ref = O.attention(q[bh, :, :hd].astype(np.float64), k[bkv, :, :hd], v[bkv])
            np.testing.assert_allclose(got[j, :, h * hd:(h + 1) * hd], ref, rtol=0,
                                       atol=1e-2 * np.abs(ref).max() + 1e-3)


@pytest.mark.parametrize("hd,Lk,kramp", [(128, 1536, 24.0), (32, 700, 30.0)])
def test_attention_growing_row_max_rescales_match_oracle(B, hd, Lk, kramp):
    """Keys grow along the sequence, so the running max of every row rises by more than the
    lazy-rescale threshold on many key tiles: O and the row sums are rescaled repeatedly."""
    heads, nb, Lq = 2, 1, 300
    q, k, v, got = _attn_case(B, hd, heads, nb, Lq, Lk, False, 2.0, seed=17 + Lk, kramp=kramp)
    for h in range(heads):
        qq, kk = q[h, :, :hd].astype(np.float64), k[h, :, :hd].astype(np.float64)
        s = qq @ kk.T / np.sqrt(hd) * np.log2(np.e)
        tiles = s.reshape(Lq, -1)[:, :(Lk // 128) * 128].reshape(Lq, -1, 128).max(axis=2)
        rises = (np.diff(np.maximum.accumulate(tiles, axis=1), axis=1) > 8).sum(axis=1)
        assert rises.mean() > 2      # the case does exercise repeated rescales
        ref = O.attention(qq, kk, v[h])
        np.testing.assert_allclose(got[0, :, h * hd:(h + 1) * hd], ref, rtol=0, atol=1e-2 * np.abs(ref).max() + 1e-3)


# -------------------------------------------------------------- layernorm ----

def test_layernorm_modulate_matches_oracle(B):
    M, d = 333, 1536
    x = synth.normal(21, (M, d)) * 3 + 0.5
    sh, sc = synth.normal(22, (d,)), synth.normal(23, (d,)) * 0.2
    out = torch.empty(M, d, device="cuda", dtype=torch.bfloat16)
    B.layernorm_modulate(dev(x), dev(sh), dev(sc), out)
    ref = O.layer_norm(x.astype(np.float64)) * (1 + sc) + sh
    np.testing.assert_allclose(out.float().cpu().numpy(), ref, rtol=2 ** -8, atol=1e-5 * np.abs(ref).max())
    B.layernorm_modulate(dev(x), None, None, out)
    np.testing.assert_allclose(out.float().cpu().numpy(), O.layer_norm(x.astype(np.float64)), rtol=2 ** -8,
                               atol=1e-5)


# ------------------------------------------------------------- cache rule ----

def _velocity_np(x, k):
    a = synth.uniform(500 + k, x.shape[1:], -0.9, -0.2)
    b = synth.normal(600 + k, x.shape[1:]) * 0.3
    return a * x + b


@pytest.mark.parametrize("N,D,tau,K_w,K_c", [(5, 4096, 0.08, 1, 1), (3, 1001, 0.15, 0, 0), (4, 70000, 0.0, 1, 1),
                                             (4096, 24, 0.1, 1, 1)])   # the most candidates a call takes
def test_cache_rule_matches_oracle(B, N, D, tau, K_w, K_c):
    T = 8
    t = O.time_grid(T)
    x1 = synth.normal(7, (N, D))
    y = synth.normal(8, (D,))
    st = B.new_state(N, D)
    st["x"].copy_(dev(x1))
    ws = torch.zeros(B.cache_workspace_bytes(N, D) // 4 + 1, device="cuda")
    skip = torch.zeros(N, dtype=torch.uint8, device="cuda")
    idx = torch.zeros(N, dtype=torch.int32, device="cuda")
    nc = torch.zeros(1, dtype=torch.int32, device="cuda")
    v = torch.zeros(N, D, device="cuda")
    scores = torch.zeros(N, device="cuda")
    err = err_word()
    ostates = [O.CacheState() for _ in range(N)]
    xs = x1.astype(np.float64)
    for k in range(1, T + 1):
        B.cache_decide(st["x"], st["x_ref"], st["accum"], st["has_ref"], k, T, tau, K_w, K_c, skip, idx, nc, ws,
                       err=err)
        # the test's stand-in velocity field, evaluated on the GPU state with torch
        xg = st["x"]
        a = dev(synth.uniform(500 + k, (D,), -0.9, -0.2))
        b = dev(synth.normal(600 + k, (D,)) * 0.3)
        v.copy_(a * xg + b)
        B.cache_apply(st["x"], st["x_ref"], st["delta"], v, skip, float(t[k - 1]), float(t[k]), workspace=ws,
                      target=dev(y), scores=scores)
        pre = [None if O.forced_compute(k, T, K_w, K_c, s.has_ref) else s.a + O.relative_drift(xs[i], s.x_ref)
               for i, s in enumerate(ostates)]
        near = np.array([p is not None and abs(p - tau) < 1e-3 for p in pre])
        xs, skipped, _, sc = O.search_step(ostates, xs, k, T, tau, K_w, K_c, lambda z, tt: _velocity_np(z[None], k)[0],
                                           target=y)
        gskip = skip.cpu().numpy().astype(bool)
        assert np.array_equal(gskip[~near], skipped[~near]), (k, gskip, skipped)
        assert int(nc[0]) == int((~gskip).sum())
        assert idx.cpu().numpy()[:int(nc[0])].tolist() == np.flatnonzero(~gskip).tolist()
        np.testing.assert_allclose(st["accum"].cpu().numpy(), [s.a for s in ostates], rtol=1e-5, atol=1e-6)
        np.testing.assert_allclose(st["x"].cpu().numpy(), xs, rtol=1e-5, atol=1e-5)
        np.testing.assert_allclose(scores.cpu().numpy(), sc, rtol=1e-5)
    torch.cuda.synchronize()
    assert int(err[0]) == 0


def test_cache_decide_flags_nonfinite_and_bad_force(B):
    N, D = 2, 512
    st = B.new_state(N, D)
    st["x"].normal_()
    st["x_ref"].normal_()
    st["has_ref"].fill_(1)
    st["x"][1, 7] = float("nan")
    ws = torch.zeros(B.cache_workspace_bytes(N, D) // 4 + 1, device="cuda")
    skip = torch.zeros(N, dtype=torch.uint8, device="cuda")
    idx = torch.zeros(N, dtype=torch.int32, device="cuda")
    nc = torch.zeros(1, dtype=torch.int32, device="cuda")
    err = err_word()
    B.cache_decide(st["x"], st["x_ref"], st["accum"], st["has_ref"], 3, 10, 100.0, 1, 1, skip, idx, nc, ws, err=err)
    torch.cuda.synchronize()
    assert int(err[0]) == B.CS_ERR_NONFINITE
    assert skip.cpu().tolist() == [1, 0]      # the non-finite candidate is computed
    err.zero_()
    st["has_ref"][0] = 0
    force = torch.tensor([0, 1], dtype=torch.uint8, device="cuda")
    st["x"][1, 7] = 0.0
    B.cache_decide(st["x"], st["x_ref"], st["accum"], st["has_ref"], 3, 10, 100.0, 1, 1, skip, idx, nc, ws,
                   force=force, err=err)
    torch.cuda.synchronize()
    assert int(err[0]) == B.CS_ERR_ARG


# ---------------------------------------------------------- score / select ----

def test_score_topk_and_beam_refill(B):
    N, D = 16, 3000
    x = synth.normal(31, (N, D))
    y = synth.normal(32, (D,))
    ws = torch.zeros(B.cache_workspace_bytes(N, D) // 4 + 1, device="cuda")
    scores = torch.zeros(N, device="cuda")
    B.score(dev(x), dev(y), scores, ws)
    ref = np.array([O.score(x[i], y) for i in range(N)])
    np.testing.assert_allclose(scores.cpu().numpy(), ref, rtol=1e-5)
    # top-k on values with ties and a NaN
    s = np.array([3, 1, 3, 2, np.nan, 5, 5, -1, 0, 2, 3, 4, 4, 1, -2, 5], np.float32)
    idx = torch.zeros(16, dtype=torch.int32, device="cuda")
    B.select_topk(dev(s), 16, idx)
    assert idx.cpu().tolist() == O.topk(s, 16).tolist()
    B.select_topk(scores, 4, idx)
    assert idx.cpu().tolist()[:4] == O.topk(ref, 4).tolist()
    # beam refill: keep 4, 3 children each
    src = B.new_state(N, D)
    for key in ("x", "x_ref", "delta"):
        src[key].normal_()
    src["accum"].uniform_()
    src["has_ref"].fill_(1)
    dst = B.new_state(N, D)
    surv = torch.tensor([5, 0, 11, 2], dtype=torch.int32, device="cuda")
    noise = synth.beam_noise(synth.replace_model(synth.TINY, C=1, F=1, H=30, W=100), 1, 4, 3).reshape(12, D)
    B.beam_refill(src, dst, surv, 3, 0.1, dev(noise))
    ost = [O.CacheState(src["delta"][i].cpu().numpy().astype(np.float64), src["x_ref"][i].cpu().numpy().astype(np.float64),
                        float(src["accum"][i])) for i in range(N)]
    ns, nx = O.beam_refill(ost, src["x"].cpu().numpy(), [5, 0, 11, 2], 3, 0.1, noise)
    np.testing.assert_allclose(dst["x"].cpu().numpy(), nx, rtol=1e-6, atol=1e-6)
    np.testing.assert_array_equal(dst["x_ref"].cpu().numpy(), np.stack([s.x_ref for s in ns]).astype(np.float32))
    np.testing.assert_array_equal(dst["accum"].cpu().numpy(), np.array([s.a for s in ns], np.float32))


@pytest.mark.parametrize("N,D,score", [(4, 2096640, True), (7, 50000, False), (16, 8192 * 3, True),
                                     (2, 8192 + 8, False),      # one full chunk and an 8-element tail
                                     (4096, 16, True)])         # the most candidates a call takes
def test_fused_decide_skip_equals_two_pass_path(B, N, D, score):
    """cs_cache_decide_skip + cs_cache_apply_computed give the same state bits as
    cs_cache_decide + cs_cache_apply, over three steps (forced, free, scored)."""
    T = 10
    t = O.time_grid(T)
    x0 = synth.normal(41, (N, D))
    dx = synth.normal(42, (N, D)) * 0.02
    states = []
    for _ in range(2):
        st = B.new_state(N, D)
        st["x"].copy_(dev(x0))
        st["x_ref"].copy_(dev(x0 + dx))
        st["delta"].copy_(dev(synth.normal(43, (N, D))))
        st["accum"].copy_(dev(synth.uniform(44, (N,), 0.0, 0.09)))
        st["has_ref"].fill_(1)
        st["has_ref"][N - 1] = 0
        states.append(st)
    ws = [torch.zeros(B.cache_workspace_bytes(N, D) // 4 + 1, device="cuda") for _ in range(2)]
    y = dev(synth.normal(45, (D,)))
    out = []
    for which, st in enumerate(states):
        skip = torch.zeros(N, dtype=torch.uint8, device="cuda")
        idx = torch.zeros(N, dtype=torch.int32, device="cuda")
        nc = torch.zeros(1, dtype=torch.int32, device="cuda")
        sc = torch.zeros(N, device="cuda")
        err = err_word()
        rec = []
        for k in (1, 4, 5):
            v = dev(synth.normal(50 + k, (N, D)))
            tgt = y if (score and k == 5) else None
            if which == 0:
                B.cache_decide(st["x"], st["x_ref"], st["accum"], st["has_ref"], k, T, 0.1, 1, 1, skip, idx, nc, ws[0],
                               err=err)
                B.cache_apply(st["x"], st["x_ref"], st["delta"], v, skip, float(t[k - 1]), float(t[k]),
                              workspace=ws[0], target=tgt, scores=sc if tgt is not None else None)
            else:
                B.cache_decide_skip(st["x"], st["x_ref"], st["delta"], st["accum"], st["has_ref"], k, T,
                                    float(t[k - 1]), float(t[k]), 0.1, 1, 1, skip, idx, nc, ws[1], target=tgt, err=err)
                B.cache_apply_computed(st["x"], st["x_ref"], st["delta"], v, skip, float(t[k - 1]), float(t[k]),
                                       workspace=ws[1], target=tgt, scores=sc if tgt is not None else None)
            torch.cuda.synchronize()
            rec.append((skip.clone(), idx[:int(nc[0])].clone(), sc.clone()))
        assert int(err[0]) == 0
        out.append(rec)
    for (s0, i0, c0), (s1, i1, c1) in zip(*out):
        assert torch.equal(s0, s1) and torch.equal(i0, i1)
        # score partials are summed in a different element grouping by the two paths
        torch.testing.assert_close(c0, c1, rtol=1e-6, atol=0)
    assert 0 < int(out[0][1][0].sum()) < N or 0 < int(out[0][2][0].sum()) < N   # some candidates skip
    for key in ("x", "x_ref", "delta", "accum", "has_ref"):
        assert torch.equal(states[0][key], states[1][key]), key


@pytest.mark.parametrize("m,k,score", [(synth.WAN_1_3B, 20, True), (synth.WAN_1_3B, 21, False),
                                        (synth.TINY, 5, True), (synth.WAN_1_3B_SHORT, 3, True)])
def test_apply_tokens_equals_scatter_then_apply(B, m, k, score):
    """cs_cache_apply_tokens (the computed update straight from the head's token-layout
    output) gives the state bits of the velocity scatter (the oracle's unpatchify) followed
    by cs_cache_apply_computed; skipped candidates are left alone; scores agree.  Step 3
    of the short workload lies in its warm-up window: every candidate computes."""
    N, T, tau = 4, 50 if m is not synth.TINY else 10, 0.1
    K = 5 if T == 50 else 3
    D, L = m.D, m.L
    t = O.time_grid(T)
    x = synth.normal(61, (N, D))
    xr = x + synth.normal(62, (N, D)) * np.array([0.02, 0.2, 0.01, 0.3])[:, None]
    states = []
    for _ in range(2):
        st = B.new_state(N, D)
        st["x"].copy_(dev(x))
        st["x_ref"].copy_(dev(xr))
        st["delta"].copy_(dev(synth.normal(63, (N, D))))
        st["accum"].copy_(dev(np.array([0.01, 0.0, 0.02, 0.0], np.float32)))
        st["has_ref"].fill_(1)
        states.append(st)
    y = dev(synth.normal(64, (D,)))
    hout_all = synth.normal(65, (N * L, 4 * m.C))
    out = []
    for which, st in enumerate(states):
        ws = torch.zeros(B.cache_workspace_bytes(N, D) // 4 + 1, device="cuda")
        skip = torch.zeros(N, dtype=torch.uint8, device="cuda")
        idx = torch.zeros(N, dtype=torch.int32, device="cuda")
        nc = torch.zeros(1, dtype=torch.int32, device="cuda")
        sc = torch.zeros(N, device="cuda")
        err = err_word()
        tgt = y if score else None
        B.cache_decide_skip(st["x"], st["x_ref"], st["delta"], st["accum"], st["has_ref"], k, T, float(t[k - 1]),
                            float(t[k]), tau, K, K, skip, idx, nc, ws, target=tgt, err=err)
        torch.cuda.synchronize()
        n_c = int(nc[0])
        comp = idx[:n_c].cpu().numpy()
        hout = dev(hout_all[:n_c * L])
        if which == 0:
            v = torch.full((N, D), float("nan"), device="cuda")
            for j, i in enumerate(comp):
                v[i] = dev(O.unpatchify(hout_all[j * L:(j + 1) * L], m.C, m.F, m.H, m.W).reshape(-1))
            B.cache_apply_computed(st["x"], st["x_ref"], st["delta"], v, skip, float(t[k - 1]), float(t[k]),
                                   workspace=ws, target=tgt, scores=sc if score else None)
        else:
            tp = torch.zeros(N, m.F * m.H // 2, device="cuda")
            B.cache_apply_tokens(st, skip, hout, idx, n_c, m.C, m.F, m.H, m.W, float(t[k - 1]), float(t[k]),
                                 workspace=ws, target=tgt, scores=sc if score else None, tile_partials=tp, err=err)
        torch.cuda.synchronize()
        assert int(err[0]) == 0
        out.append((skip.cpu(), comp, sc.cpu()))
    (s0, c0, sc0), (s1, c1, sc1) = out
    assert torch.equal(s0, s1) and np.array_equal(c0, c1)
    if k > K and k <= T - K:
        assert s0.tolist() == [1, 0, 1, 0]           # drifts 0.02, 0.2, 0.01, 0.3 against tau 0.1
    else:
        assert not s0.any()
    for key in ("x", "x_ref", "delta", "accum", "has_ref"):
        assert torch.equal(states[0][key], states[1][key]), key
    if score:
        torch.testing.assert_close(sc0, sc1, rtol=1e-6, atol=0)
        ref = [O.score(states[0]["x"][i].double().cpu().numpy() - t[k] * (
            states[0]["x"][i].double().cpu().numpy() - x[i]) / (t[k] - t[k - 1]), y.cpu().numpy()) for i in range(N)]
        np.testing.assert_allclose(sc1.numpy(), ref, rtol=1e-4)
