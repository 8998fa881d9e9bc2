"""Parity at the full sizes of the other workloads, in the launch configurations that
``bench.py --config NAME`` runs, on sampled outputs the fp64 oracle computes one by one
(GPU).

* wan14b-best-of-4 (d 5120, 40 heads, FFN 13824; M = 4 x 32760 rows): the Q/K/V^T
  projection with its per-head scatter, FFN up with GELU, FFN down with the gated
  residual, and self-attention over 4 x 40 heads x 32760 tokens;
* wan1.3b-short32 (32 candidates x 14040 tokens, so ragged query and key tiles): the
  Q/K/V^T projection, FFN down, self- and cross-attention;
* the fused cache step on the short32 latent (N 32) and the beam16 latent (N 16), every
  element.

The [M, K] activations are tiled from a seeded block of 4099 rows (a prime, so no tile
boundary lines up with the period) to bound the host's work; the kernels still run on
the full M.  Attention inputs repeat over (candidate, head) with period 7 likewise.
"""
import numpy as np
import pytest
import torch

from oracle import cachedsearch_oracle as O
from paper_2607_23159_gb300 import synth

pytestmark = pytest.mark.gpu

P_ROWS = 4099
P_BH = 7


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


def tiled(base, M, dtype):
    """[M, K] device tensor whose row m is base[m % len(base)]."""
    t = dev(base, dtype)
    return t.repeat((M + len(base) - 1) // len(base), 1)[:M].contiguous()


def sample(M, N, seed, extra_rows, extra_cols, n=400):
    """n random (row, col) pairs plus every pairing of the edge rows with the edge columns."""
    rng = np.random.default_rng(seed)
    er, ec = np.meshgrid(np.asarray(extra_rows), np.asarray(extra_cols), indexing="ij")
    rows = np.concatenate([rng.integers(0, M, n), er.ravel()]).astype(np.int64)
    cols = np.concatenate([rng.integers(0, N, n), ec.ravel()]).astype(np.int64)
    return rows, cols


def ref_dot(A_base, W, bias, rows, cols):
    a = A_base[rows % len(A_base)].astype(np.float64)
    return np.einsum("ij,ij->i", a, W[cols].astype(np.float64)) + bias[cols]


# ------------------------------------------------------------------- GEMMs ----

@pytest.mark.parametrize("m,nb", [(synth.WAN_14B, 4), (synth.WAN_1_3B_SHORT, 32)], ids=["14b", "short32"])
def test_full_size_qkv_projection_scatter(B, m, nb):
    L, d, heads, hd = m.L, m.d, m.heads, m.hd
    M, N, K = nb * L, 3 * d, d
    A_base = bf(synth.normal(1100 + d, (P_ROWS, K)))
    W = bf(synth.normal(1101 + d, (N, K)) * (1.0 / np.sqrt(K)))
    bias = synth.normal(1102, (N,))
    hds, Lv = max(hd, 64), (L + 7) // 8 * 8
    q = torch.zeros(nb * heads, L, hds, device="cuda", dtype=torch.bfloat16)
    k = torch.zeros_like(q)
    vt = torch.zeros(nb * heads, hd, Lv, device="cuda", dtype=torch.bfloat16)
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    B.gemm_qkv(tiled(A_base, M, torch.bfloat16), dev(W, torch.bfloat16), dev(bias), L, d, heads, 0, q, k, vt, Lv,
               err=err)
    torch.cuda.synchronize()
    assert int(err[0]) == 0
    rows, cols = sample(M, N, d, [0, M - 1, L - 1, L, M - 128], [0, N - 1, d - 1, d, 2 * d, hd])
    ref = ref_dot(A_base, W, bias, rows, cols)
    b, l = rows // L, rows % L
    part, head, c = cols // d, (cols % d) // hd, cols % hd
    bh = torch.from_numpy(b * heads + head).cuda()
    lt, ct = torch.from_numpy(l).cuda(), torch.from_numpy(c).cuda()
    got = torch.where(torch.from_numpy(part == 0).cuda(), q[bh, lt, ct],
                      torch.where(torch.from_numpy(part == 1).cuda(), k[bh, lt, ct], vt[bh, ct, lt]))
    np.testing.assert_allclose(got.float().cpu().numpy(), ref, rtol=2 ** -8, atol=1e-4 * np.abs(ref).max())


@pytest.mark.parametrize("m,nb,which", [(synth.WAN_14B, 4, "up"), (synth.WAN_14B, 4, "down"),
                                        (synth.WAN_1_3B_SHORT, 32, "down")], ids=["14b-up", "14b-down", "short32-down"])
def test_full_size_ffn_gemms(B, m, nb, which):
    M = nb * m.L
    N, K = (m.ffn, m.d) if which == "up" else (m.d, m.ffn)
    A_base = bf(synth.normal(1200 + K, (P_ROWS, K)))
    W = bf(synth.normal(1201 + N, (N, K)) * (1.0 / np.sqrt(K)))
    bias = synth.normal(1202, (N,))
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    rows, cols = sample(M, N, K, [0, M - 1, m.L, M - 256], [0, N - 1, 255, 256, N - 256])
    dot = ref_dot(A_base, W, bias, rows, cols)
    if which == "up":
        out = torch.empty(M, N, device="cuda", dtype=torch.bfloat16)
        B.gemm(tiled(A_base, M, torch.bfloat16), dev(W, torch.bfloat16), B.EPI_GELU_BF16, out, bias=dev(bias),
               err=err)
        ref = O.gelu_tanh(dot)
        tol = dict(rtol=2 ** -8, atol=1e-4 * np.abs(ref).max())
    else:
        res_base = synth.normal(1203, (P_ROWS, N))
        gate = synth.normal(1204, (N,))
        out = tiled(res_base, M, torch.float32)
        B.gemm(tiled(A_base, M, torch.bfloat16), dev(W, torch.bfloat16), B.EPI_RESID_F32, out, bias=dev(bias),
               gate=dev(gate), err=err)
        ref = res_base[rows % P_ROWS, cols] + gate[cols] * dot
        tol = dict(rtol=1e-5, atol=1e-5 * np.abs(ref).max())
    torch.cuda.synchronize()
    assert int(err[0]) == 0
    got = out[torch.from_numpy(rows).cuda(), torch.from_numpy(cols).cuda()].float().cpu().numpy()
    np.testing.assert_allclose(got, ref, **tol)
    del out


# --------------------------------------------------------------- attention ----

def _bh_tiled(base, BH):
    """[BH, ...] device tensor whose entry bh is base[bh % len(base)]."""
    idx = torch.arange(BH, device="cuda") % len(base)
    return dev(base, torch.bfloat16)[idx].contiguous()


@pytest.mark.parametrize("m,nb,picks", [(synth.WAN_14B, 4, [(0, 0), (1, 17), (2, 39), (3, 23)]),
                                        (synth.WAN_1_3B_SHORT, 32, [(0, 0), (13, 5), (31, 11)])],
                         ids=["14b", "short32"])
def test_full_size_self_attention_sampled_rows(B, m, nb, picks):
    L, H, hd = m.L, m.heads, m.hd
    BH = nb * H
    q_b = bf(synth.normal(1300 + L, (P_BH, L, hd)))
    k_b = bf(synth.normal(1301 + L, (P_BH, L, hd)))
    v_b = bf(synth.normal(1302 + L, (P_BH, L, hd)))
    o = torch.empty(nb, L, H * hd, device="cuda", dtype=torch.bfloat16)
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    B.attention(_bh_tiled(q_b, BH), _bh_tiled(k_b, BH), _bh_tiled(np.ascontiguousarray(v_b.transpose(0, 2, 1)), BH),
                o, nb, H, L, L, hd, L, False, err=err)
    torch.cuda.synchronize()
    assert int(err[0]) == 0
    rng = np.random.default_rng(L)
    for j, h in picks:
        s = (j * H + h) % P_BH
        rows = np.concatenate([rng.integers(0, L, 3), [0, L - 1]])   # L - 1 sits in the ragged last tile
        ref = O.attention(q_b[s, rows].astype(np.float64), k_b[s].astype(np.float64), v_b[s].astype(np.float64))
        got = o[j, torch.from_numpy(rows).cuda(), h * hd:(h + 1) * hd].float().cpu().numpy()
        np.testing.assert_allclose(got, ref, rtol=0, atol=1e-2 * np.abs(ref).max() + 1e-3)


def test_full_size_short32_cross_attention_sampled_rows(B):
    m, nb = synth.WAN_1_3B_SHORT, 32
    L, H, hd, Lt = m.L, m.heads, m.hd, m.Lt
    q_b = bf(synth.normal(1400, (P_BH, L, hd)))
    kt = bf(synth.normal(1401, (H, Lt, hd)) * 2)
    vtt = bf(synth.normal(1402, (H, Lt, hd)))
    o = torch.empty(nb, L, H * hd, device="cuda", dtype=torch.bfloat16)
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    B.attention(_bh_tiled(q_b, nb * H), dev(kt, torch.bfloat16), dev(np.ascontiguousarray(vtt.transpose(0, 2, 1)),
                torch.bfloat16), o, nb, H, L, Lt, hd, Lt, True, err=err)
    torch.cuda.synchronize()
    assert int(err[0]) == 0
    rng = np.random.default_rng(9)
    for j, h in [(0, 2), (17, 9), (31, 11)]:
        rows = np.concatenate([rng.integers(0, L, 4), [L - 1]])
        ref = O.attention(q_b[(j * H + h) % P_BH, rows].astype(np.float64), kt[h].astype(np.float64),
                          vtt[h].astype(np.float64))
        got = o[j, torch.from_numpy(rows).cuda(), h * hd:(h + 1) * hd].float().cpu().numpy()
        np.testing.assert_allclose(got, ref, rtol=0, atol=1e-2 * np.abs(ref).max() + 1e-3)


# -------------------------------------------------------------- cache step ----

@pytest.mark.parametrize("m,N", [(synth.WAN_1_3B_SHORT, 32), (synth.WAN_1_3B, 16)], ids=["short32", "beam16"])
def test_full_size_fused_cache_step_every_element(B, m, N):
    D, T, tau, K_w, K_c, k = m.D, 50, 0.1, 5, 5, 20
    t = O.time_grid(T)
    x = synth.normal(41, (N, D))
    # accumulated drift a = 0.04 + ~scale lands 5-14e-3 above (even i) or below (odd i) tau
    off = np.array([(-1) ** i * (0.005 + 0.001 * (i % 10)) for i in range(N)])
    scale = (0.06 + off).astype(np.float32)
    xr = x + synth.normal(42, (N, D)) * scale[:, None]
    delta = synth.normal(43, (N, D))
    v = synth.normal(44, (N, D))
    y = synth.normal(45, (D,))
    a0 = np.full(N, 0.04)
    has = np.ones(N, np.uint8)
    has[N // 3] = 0                                             # one empty cache: must compute
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
    B.cache_decide_skip(st["x"], st["x_ref"], st["delta"], st["accum"], st["has_ref"], k, T, float(t[k - 1]),
                        float(t[k]), tau, K_w, K_c, skip, idx, nc, ws, target=dev(y), err=err)
    B.cache_apply_computed(st["x"], st["x_ref"], st["delta"], dev(v), skip, float(t[k - 1]), float(t[k]),
                           workspace=ws, target=dev(y), scores=scores)
    torch.cuda.synchronize()
    assert int(err[0]) == 0
    states = [O.CacheState(delta[i].astype(np.float64) if has[i] else None,
                           xr[i].astype(np.float64) if has[i] else None, float(a0[i])) for i in range(N)]
    xo, sk, so, near = [], [], [], []
    for i in range(N):
        a_before = states[i].a
        vi = v[i].astype(np.float64)
        vel, comp, _ = O.wrapper_call(states[i], x[i], k, T, tau, K_w, K_c, lambda z: vi)
        xn = O.euler(x[i].astype(np.float64), t[k - 1], t[k], vel)
        xo.append(xn)
        sk.append(not comp)
        so.append(O.score(xn - t[k] * vel, y))
        near.append(bool(has[i]) and abs(a_before + O.relative_drift(x[i], xr[i]) - tau) < 1e-3)
    assert 0 < sum(sk) < N - 1                                   # both branches at full size
    got_skip = skip.cpu().numpy().astype(bool)
    assert not any(near), "a drift lands in the near-tie zone; pick other seeds"
    assert got_skip.tolist() == sk
    assert int(nc[0]) == N - sum(sk) and idx[:int(nc[0])].cpu().tolist() == [i for i in range(N) if not sk[i]]
    np.testing.assert_allclose(st["x"].cpu().numpy(), np.stack(xo), rtol=1e-5, atol=1e-5)
    np.testing.assert_allclose(st["accum"].cpu().numpy(), [s.a for s in states], rtol=1e-5, atol=1e-7)
    np.testing.assert_allclose(scores.cpu().numpy(), so, rtol=1e-5)
    comp_i = [i for i in range(N) if not sk[i]]
    for i in comp_i[:2]:
        np.testing.assert_array_equal(st["x_ref"][i].cpu().numpy(), x[i])
        np.testing.assert_allclose(st["delta"][i].cpu().numpy(), v[i] - x[i], rtol=1e-6, atol=1e-6)
