"""Parity at the full 1.3B workload sizes, in the launch configurations the bench uses,
on sampled outputs the fp64 oracle computes one by one (GPU).

* the step's GEMMs at M = 4 candidates x 32760 tokens (QKV 4608 x 1536, FFN down
  1536 x 8960) on 512 sampled output elements;
* self-attention over 4 candidates x 12 heads x 32760 tokens, 24 sampled query rows;
* cross-attention of the same queries against the 512-token text K/V;
* the fused cache step (decide + skip update + computed update + score) on the full
  4 x 2 096 640 latent, every element against the oracle's wrapper step.
"""
import numpy as np
import pytest
import torch

from oracle import cachedsearch_oracle as O
from paper_2607_23159_gb300 import synth

pytestmark = pytest.mark.gpu

L, NC, H, HD = 32760, 4, 12, 128


@pytest.fixture(scope="module")
def B():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_23159_gb300 import binding
    return binding


def bf(a):
    return synth.round_to_bf16(np.asarray(a, np.float32))


def dev(a, dtype=torch.float32):
    return torch.from_numpy(np.ascontiguousarray(a)).to("cuda").to(dtype)


@pytest.mark.parametrize("N,K,epi", [(4608, 1536, 1), (1536, 8960, 3)])
def test_full_size_gemm_sampled_outputs(B, N, K, epi):
    M = NC * L
    A = bf(synth.normal(900 + K, (M, K)))
    W = bf(synth.normal(901 + N, (N, K)) * (1.0 / np.sqrt(K)))
    bias = synth.normal(902, (N,))
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    if epi == 1:
        out = torch.empty(M, N, device="cuda", dtype=torch.bfloat16)
        B.gemm(dev(A, torch.bfloat16), dev(W, torch.bfloat16), B.EPI_BF16, out, bias=dev(bias), err=err)
    else:
        res0 = synth.normal(903, (M, N))
        gate = synth.normal(904, (N,))
        out = dev(res0)
        B.gemm(dev(A, torch.bfloat16), dev(W, torch.bfloat16), B.EPI_RESID_F32, out, bias=dev(bias), gate=dev(gate),
               err=err)
    torch.cuda.synchronize()
    assert int(err[0]) == 0
    rng = np.random.default_rng(K)
    rows = np.concatenate([rng.integers(0, M, 500), [0, M - 1, L - 1, L, M - 128, M - 1]])
    cols = np.concatenate([rng.integers(0, N, 500), [0, N - 1, 255, 256, N - 256, 17]])
    got = out.float().cpu().numpy()[rows, cols]
    ref = np.einsum("ij,ij->i", A[rows].astype(np.float64), W[cols].astype(np.float64)) + bias[cols]
    if epi == 1:
        np.testing.assert_allclose(got, ref, rtol=2 ** -8, atol=1e-4 * np.abs(ref).max())
    else:
        ref = res0[rows, cols] + gate[cols] * ref
        np.testing.assert_allclose(got, ref, rtol=1e-5, atol=1e-5 * np.abs(ref).max())


@pytest.fixture(scope="module")
def qkv():
    rng = np.random.default_rng(77)
    q = bf(rng.standard_normal((NC * H, L, HD), dtype=np.float32))
    k = bf(rng.standard_normal((NC * H, L, HD), dtype=np.float32))
    v = bf(rng.standard_normal((NC * H, L, HD), dtype=np.float32))
    return q, k, v


def test_full_size_self_attention_sampled_rows(B, qkv):
    q, k, v = qkv
    vt = np.ascontiguousarray(v.transpose(0, 2, 1))
    o = torch.empty(NC, L, H * HD, device="cuda", dtype=torch.bfloat16)
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    B.attention(dev(q, torch.bfloat16), dev(k, torch.bfloat16), dev(vt, torch.bfloat16), o, NC, H, L, L, HD, L,
                False, err=err)
    torch.cuda.synchronize()
    assert int(err[0]) == 0
    got = o.float().cpu().numpy()
    rng = np.random.default_rng(5)
    for j, h in [(0, 0), (1, 7), (2, 11), (3, 4)]:
        bh = j * H + h
        rows = np.concatenate([rng.integers(0, L, 4), [0, L - 1]])   # includes the ragged last tile
        ref = O.attention(q[bh, rows].astype(np.float64), k[bh].astype(np.float64), v[bh].astype(np.float64))
        np.testing.assert_allclose(got[j, rows, h * HD:(h + 1) * HD], ref, rtol=0, atol=1e-2 * np.abs(ref).max() + 1e-3)


def test_full_size_cross_attention_sampled_rows(B, qkv):
    q, _, _ = qkv
    Lt = 512
    rng = np.random.default_rng(6)
    kt = bf(rng.standard_normal((H, Lt, HD), dtype=np.float32) * 2)
    vtt = bf(rng.standard_normal((H, Lt, HD), dtype=np.float32))
    o = torch.empty(NC, L, H * HD, device="cuda", dtype=torch.bfloat16)
    B.attention(dev(q, torch.bfloat16), dev(kt, torch.bfloat16), dev(np.ascontiguousarray(vtt.transpose(0, 2, 1)),
                torch.bfloat16), o, NC, H, L, Lt, HD, Lt, True)
    torch.cuda.synchronize()
    got = o.float().cpu().numpy()
    for j, h in [(0, 3), (3, 10)]:
        rows = np.concatenate([rng.integers(0, L, 6), [L - 1]])
        ref = O.attention(q[j * H + h, rows].astype(np.float64), kt[h].astype(np.float64), vtt[h].astype(np.float64))
        np.testing.assert_allclose(got[j, rows, h * HD:(h + 1) * HD], ref, rtol=0, atol=1e-2 * np.abs(ref).max() + 1e-3)


def test_full_size_fused_cache_step_every_element(B):
    D = synth.WAN_1_3B.D
    N, T, tau = NC, 50, 0.1
    t = O.time_grid(T)
    x = synth.normal(31, (N, D))
    xr = x + synth.normal(32, (N, D)) * np.array([0.02, 0.05, 0.002, 0.0])[:, None]
    delta = synth.normal(33, (N, D))
    v = synth.normal(34, (N, D))
    y = synth.normal(35, (D,))
    a0 = np.array([0.05, 0.07, 0.09, 0.0])
    has = np.array([1, 1, 1, 0], np.uint8)
    st = B.new_state(N, D)
    st["x"].copy_(dev(x))
    st["x_ref"].copy_(dev(xr))
    st["delta"].copy_(dev(delta))
    st["accum"].copy_(dev(a0.astype(np.float32)))
    st["has_ref"].copy_(torch.from_numpy(has))
    ws = torch.zeros(B.cache_workspace_bytes(N, D) // 4 + 1, device="cuda")
    skip = torch.zeros(N, dtype=torch.uint8, device="cuda")
    idx = torch.zeros(N, dtype=torch.int32, device="cuda")
    nc = torch.zeros(1, dtype=torch.int32, device="cuda")
    scores = torch.zeros(N, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    k = 20
    B.cache_decide_skip(st["x"], st["x_ref"], st["delta"], st["accum"], st["has_ref"], k, T, float(t[k - 1]),
                        float(t[k]), tau, 5, 5, skip, idx, nc, ws, target=dev(y), err=err)
    B.cache_apply_computed(st["x"], st["x_ref"], st["delta"], dev(v), skip, float(t[k - 1]), float(t[k]),
                           workspace=ws, target=dev(y), scores=scores)
    torch.cuda.synchronize()
    assert int(err[0]) == 0
    # oracle: the same step through the wrapper, velocity v for computed candidates
    states = [O.CacheState(delta[i].astype(np.float64) if has[i] else None,
                           xr[i].astype(np.float64) if has[i] else None, float(a0[i])) for i in range(N)]
    xo, sk, so = [], [], []
    for i in range(N):
        vi = v[i].astype(np.float64)
        vel, comp, _ = O.wrapper_call(states[i], x[i], k, T, tau, 5, 5, lambda z: vi)
        xn = O.euler(x[i].astype(np.float64), t[k - 1], t[k], vel)
        xo.append(xn)
        sk.append(not comp)
        so.append(O.score(xn - t[k] * vel, y))
    assert skip.cpu().numpy().astype(bool).tolist() == sk
    assert sk == [True, False, True, False]      # a = 0.07, 0.12, 0.092 against tau 0.1; empty cache
    np.testing.assert_allclose(st["x"].cpu().numpy(), np.stack(xo), rtol=1e-5, atol=1e-5)
    np.testing.assert_allclose(st["accum"].cpu().numpy(), [s.a for s in states], rtol=1e-5, atol=1e-7)
    np.testing.assert_allclose(scores.cpu().numpy(), so, rtol=1e-5)
    for i in (1, 3):    # computed: the reference and the transformation vector are refreshed
        np.testing.assert_array_equal(st["x_ref"][i].cpu().numpy(), x[i])
        np.testing.assert_allclose(st["delta"][i].cpu().numpy(), v[i] - x[i], rtol=1e-6, atol=1e-6)


@pytest.mark.parametrize("base", ["wan1.3b", "wan1.3b-short"])
def test_composed_block_and_head_full_length_sampled_rows(B, base):
    """The composed DiT forward (patch embed, LayerNorm + adaLN, QKV scatter, self-attention
    over all tokens -- 32760 for the best-of-4 and beam latent, 14040 for the short clips --,
    gated O projection, cross-attention to the 512 text tokens, GELU FFN, head) of one
    1.3B-width block on a compacted subset of 4 candidates (idx 0, 2, 3), against the
    oracle's one-block velocity on 40 sampled token rows x all 64 features; full-length K/V
    on both sides.  The row outside the subset stays untouched."""
    m = synth.replace_model(synth.WAN_1_3B if base == "wan1.3b" else synth.WAN_1_3B_SHORT, blocks=1)
    flat, params = synth.make_params(m)
    ctx = synth.text_context(m)
    x1 = synth.initial_noise(m, range(NC))
    model = B.Model(m, NC)
    model.load_weights(flat)
    model.set_text_context(dev(ctx))
    x = dev(x1.reshape(NC, -1))
    v = torch.full((NC, m.D), 7.0, device="cuda")
    idx = torch.tensor([0, 2, 3], dtype=torch.int32, device="cuda")
    t = 0.7
    model.dit_forward(x, idx, 3, t, v)
    torch.cuda.synchronize()
    assert model.device_error() == 0
    model.close()
    got = v.cpu().numpy()
    assert np.all(got[1] == 7.0)
    dit = O.DiT(m, params)
    kv = dit.text_kv(ctx)
    rng = np.random.default_rng(71)
    rows = np.unique(np.concatenate([rng.integers(0, m.L, 38), [0, m.L - 1]]))
    f_, hh, ww = rows // ((m.H // 2) * (m.W // 2)), (rows // (m.W // 2)) % (m.H // 2), rows % (m.W // 2)
    for i in (0, 2, 3):
        ref = dit.velocity_rows(x1[i], t, kv, rows)                      # [rows, 4C]
        g = got[i].reshape(m.C, m.F, m.H, m.W)
        # token layout of the GPU velocity at the sampled rows: feature 4c + 2 ph + pw
        gt = np.stack([g[c, f_, 2 * hh + ph, 2 * ww + pw] for c in range(m.C) for ph in (0, 1) for pw in (0, 1)],
                      axis=1)
        rel = np.abs(gt - ref).max() / np.abs(ref).max()
        assert rel < 2e-2, (i, rel)
