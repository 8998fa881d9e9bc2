"""Time one of the library's kernels alone at a given shape (CUDA events, warm-up first).

  python -m paper_2607_23159_gb300.kernel_bench attention --batch 1 --L 32760 --heads 12 --hd 128
  python -m paper_2607_23159_gb300.kernel_bench gemm --M 131040 --N 8960 --K 1536 --epi 2
  python -m paper_2607_23159_gb300.kernel_bench cache --N 16 --D 2096640

Inputs are random device tensors (the timing does not depend on their values).  Prints
one JSON line with the average launch time and the achieved TFLOP/s or GB/s.  The cache
step is timed launch by launch after an L2-evicting write (median), since back-to-back
launches of it measure the host's launch rate rather than the kernel.

``--torch`` times PyTorch's own kernels on the same shape instead (informal comparators,
never part of the library's path): ``scaled_dot_product_attention`` for attention,
``torch.matmul`` for the GEMMs, and the cache step written as torch elementwise ops.
"""
from __future__ import annotations

import argparse
import json


def _time(fn, reps, warmup):
    import torch
    for _ in range(warmup):
        fn()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(reps):
        fn()
    e1.record()
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / reps


def _time_cold(fn, reps, warmup):
    """Median of single launches, each after a 256 MB write that evicts the L2 (the
    way the cache step runs inside a search step, between DiT evaluations)."""
    import torch
    for _ in range(warmup):
        fn()
    flush = torch.empty(64 << 20, device="cuda")
    times = []
    for _ in range(reps):
        flush.add_(1.0)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        fn()
        e1.record()
        torch.cuda.synchronize()
        times.append(e0.elapsed_time(e1))
    times.sort()
    return times[len(times) // 2]


def cache_step(N, lat, skip_frac, reps=9, warmup=3, seed=0, carried=True):
    """One free step's cache work for N candidates on a C x F x H x W latent, as the search
    step runs it.  carried (the step's own form): cs_cache_decide_skip_carry with the drift
    the previous step left (decisions, skipped updates and their next drift in one
    launch), then cs_cache_apply_tokens_carry for the computing candidates (head output in
    token layout); 16 D bytes per skipped candidate, 20 D per computed one.  Otherwise the
    drift-pass form, cs_cache_decide_skip + cs_cache_apply_tokens (24 D per computed one).
    The round(N (1 - skip_frac)) candidates that compute are a seeded random subset.
    Returns (median ms of single calls after an L2-evicting write, algorithmic bytes,
    skipped)."""
    import torch
    from paper_2607_23159_gb300 import binding as B
    dev = "cuda"
    C_, F_, H_, W_ = lat
    D = C_ * F_ * H_ * W_
    g = torch.Generator(device=dev)
    g.manual_seed(seed)
    st = B.new_state(N, D)
    st["x"].normal_(generator=g)
    st["x_ref"].copy_(st["x"] * 0.99)
    st["delta"].normal_(generator=g)
    st["has_ref"].fill_(1)
    ws = torch.zeros(B.cache_workspace_bytes(N, D) // 4 + 1, device=dev)
    sws = torch.zeros(B.cache_step_bytes(N, C_, F_, H_, W_) // 4 + 1, device=dev)
    skip = torch.zeros(N, dtype=torch.uint8, device=dev)
    idx = torch.zeros(N, dtype=torch.int32, device=dev)
    nc = torch.zeros(1, dtype=torch.int32, device=dev)
    n_comp = int(round(N * (1.0 - skip_frac)))
    force = torch.zeros(N, dtype=torch.uint8, device=dev)
    force[torch.randperm(N, generator=g, device=dev)[:n_comp]] = 1
    hout = torch.randn(max(1, n_comp) * F_ * (H_ // 2) * (W_ // 2), 4 * C_, device=dev, generator=g)
    comp_idx = torch.nonzero(force).to(torch.int32).reshape(-1)
    if carried:
        # step 19 with the drift pass leaves every candidate's drift for step 20
        B.cache_decide_skip_carry(st, lat, 19, 50, 0.62, 0.6, 0.1, 5, 5, skip, idx, nc, sws, carried=False,
                                  force=force)
        B.cache_apply_tokens_carry(st, skip, hout, comp_idx, n_comp, lat, 19, 0.62, 0.6, sws)

    def run():
        if carried:
            B.cache_decide_skip_carry(st, lat, 20, 50, 0.6, 0.58, 0.1, 5, 5, skip, idx, nc, sws, carried=True,
                                      force=force)
            B.cache_apply_tokens_carry(st, skip, hout, comp_idx, n_comp, lat, 20, 0.6, 0.58, sws)
        else:
            B.cache_decide_skip(st["x"], st["x_ref"], st["delta"], st["accum"], st["has_ref"], 20, 50, 0.6, 0.58,
                                0.1, 5, 5, skip, idx, nc, ws, force=force)
            B.cache_apply_tokens(st, skip, hout, comp_idx, n_comp, C_, F_, H_, W_, 0.6, 0.58)
    ms = _time_cold(run, reps, warmup)
    if carried:
        assert int(nc[0]) == n_comp, "the carried decision did not run"
    n_skip = N - n_comp
    return ms, (n_skip * 16.0 + n_comp * (20.0 if carried else 24.0)) * D, n_skip


def main():
    import torch
    from paper_2607_23159_gb300 import build
    build.build()
    from paper_2607_23159_gb300 import binding as B
    ap = argparse.ArgumentParser()
    ap.add_argument("kernel", choices=["attention", "gemm", "qkv", "layernorm", "cache", "cache-fused", "cache-tokens"])
    ap.add_argument("--batch", type=int, default=1)
    ap.add_argument("--L", type=int, default=32760)
    ap.add_argument("--Lk", type=int, default=None)
    ap.add_argument("--heads", type=int, default=12)
    ap.add_argument("--hd", type=int, default=128)
    ap.add_argument("--M", type=int, default=131040)
    ap.add_argument("--N", type=int, default=1536)
    ap.add_argument("--K", type=int, default=1536)
    ap.add_argument("--epi", type=int, default=1)
    ap.add_argument("--D", type=int, default=2096640)
    ap.add_argument("--skip-frac", type=float, default=1.0)
    ap.add_argument("--latent", default="16x21x60x104", help="C x F x H x W of the latent (cache-tokens)")
    ap.add_argument("--drift-pass", action="store_true",
                    help="cache-tokens: the drift-pass form instead of the carried drift the search step uses")
    ap.add_argument("--reps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=2)
    ap.add_argument("--torch", action="store_true", help="time the PyTorch comparator instead")
    a = ap.parse_args()
    dev = "cuda"
    bf = torch.bfloat16
    out = {"kernel": a.kernel, "impl": "torch" if a.torch else "ours"}
    if a.torch and a.kernel == "attention":
        Lk = a.Lk or a.L
        q = torch.randn(a.batch, a.heads, a.L, a.hd, device=dev).to(bf)
        k = torch.randn(a.batch, a.heads, Lk, a.hd, device=dev).to(bf)
        v = torch.randn(a.batch, a.heads, Lk, a.hd, device=dev).to(bf)
        sdpa = torch.nn.functional.scaled_dot_product_attention
        ms = _time(lambda: sdpa(q, k, v), a.reps, a.warmup)
        out.update(shape=dict(batch=a.batch, L=a.L, Lk=Lk, heads=a.heads, hd=a.hd), ms=ms,
                   tflops=4.0 * a.batch * a.heads * a.L * Lk * a.hd / (ms / 1e3) / 1e12)
    elif a.torch and a.kernel in ("gemm", "qkv"):
        N = a.N if a.kernel == "gemm" else 3 * a.heads * a.hd
        M = a.M if a.kernel == "gemm" else a.batch * a.L
        A = torch.randn(M, a.K, device=dev).to(bf)
        W = (torch.randn(N, a.K, device=dev) * 0.05).to(bf)
        ms = _time(lambda: torch.matmul(A, W.t()), a.reps, a.warmup)
        out.update(shape=dict(M=M, N=N, K=a.K), ms=ms, tflops=2.0 * M * N * a.K / (ms / 1e3) / 1e12)
    elif a.torch and a.kernel in ("cache", "cache-fused"):
        N, D = a.N, a.D
        x = torch.randn(N, D, device=dev)
        xr = x * 0.99
        delta = torch.randn(N, D, device=dev)
        h = -0.02

        def run():   # every candidate skipped: drift, then x += h (x + delta)
            d = torch.linalg.vector_norm(x - xr, dim=1) / torch.linalg.vector_norm(xr, dim=1)
            x.add_(x + delta, alpha=h)
            return d
        ms = _time_cold(run, a.reps, a.warmup)
        out.update(shape=dict(N=N, D=D, skipped=N), ms=ms, gbs=16.0 * N * D / (ms / 1e3) / 1e9)
    elif a.kernel == "attention":
        Lk = a.Lk or a.L
        hds = max(a.hd, 64)
        BH = a.batch * a.heads
        q = torch.randn(BH, a.L, hds, device=dev).to(bf)
        k = torch.randn(BH, Lk, hds, device=dev).to(bf)
        if hds > a.hd:
            q[:, :, a.hd:] = 0
            k[:, :, a.hd:] = 0
        Ls = (Lk + 7) // 8 * 8
        vt = torch.randn(BH, a.hd, Ls, device=dev).to(bf)
        o = torch.empty(a.batch, a.L, a.heads * a.hd, device=dev, dtype=bf)
        ms = _time(lambda: B.attention(q, k, vt, o, a.batch, a.heads, a.L, Lk, a.hd, Ls, False), a.reps, a.warmup)
        flops = 4.0 * BH * a.L * Lk * a.hd
        out.update(shape=dict(batch=a.batch, L=a.L, Lk=Lk, heads=a.heads, hd=a.hd), ms=ms,
                   tflops=flops / (ms / 1e3) / 1e12)
    elif a.kernel == "gemm":
        A = torch.randn(a.M, a.K, device=dev).to(bf)
        W = (torch.randn(a.N, a.K, device=dev) * 0.05).to(bf)
        bias = torch.zeros(a.N, device=dev)
        if a.epi in (B.EPI_F32, B.EPI_RESID_F32):
            C = torch.zeros(a.M, a.N, device=dev)
        else:
            C = torch.empty(a.M, a.N, device=dev, dtype=bf)
        ms = _time(lambda: B.gemm(A, W, a.epi, C, bias=bias), a.reps, a.warmup)
        out.update(shape=dict(M=a.M, N=a.N, K=a.K, epi=a.epi), ms=ms,
                   tflops=2.0 * a.M * a.N * a.K / (ms / 1e3) / 1e12)
    elif a.kernel == "qkv":
        # QKV projection with the per-head Q/K and transposed V scatter; M = batch * L rows
        M, d = a.batch * a.L, a.heads * a.hd
        A = torch.randn(M, a.K, device=dev).to(bf)
        W = (torch.randn(3 * d, a.K, device=dev) * 0.05).to(bf)
        bias = torch.zeros(3 * d, device=dev)
        hds, Lv = max(a.hd, 64), (a.L + 7) // 8 * 8
        q = torch.zeros(a.batch * a.heads, a.L, hds, device=dev, dtype=bf)
        k = torch.zeros_like(q)
        vt = torch.zeros(a.batch * a.heads, a.hd, Lv, device=dev, dtype=bf)
        ms = _time(lambda: B.gemm_qkv(A, W, bias, a.L, d, a.heads, 0, q, k, vt, Lv), a.reps, a.warmup)
        out.update(shape=dict(M=M, N=3 * d, K=a.K), ms=ms, tflops=2.0 * M * 3 * d * a.K / (ms / 1e3) / 1e12)
    elif a.kernel == "layernorm":
        M, d = a.M, a.K
        x = torch.randn(M, d, device=dev)
        sh, sc = torch.randn(d, device=dev), torch.randn(d, device=dev)
        o = torch.empty(M, d, device=dev, dtype=bf)
        ms = _time(lambda: B.layernorm_modulate(x, sh, sc, o), a.reps, a.warmup)
        out.update(shape=dict(M=M, d=d), ms=ms, gbs=M * d * 6.0 / (ms / 1e3) / 1e9)
    else:
        N, D = a.N, a.D
        lat = [int(v) for v in a.latent.split("x")]
        if a.kernel == "cache-tokens":
            ms, byts, n_skip = cache_step(N, lat, a.skip_frac, a.reps, a.warmup, carried=not a.drift_pass)
            D = lat[0] * lat[1] * lat[2] * lat[3]
            out.update(shape=dict(N=N, D=D, skipped=n_skip), ms=ms, gbs=byts / (ms / 1e3) / 1e9)
            print(json.dumps(out), flush=True)
            return
        st = B.new_state(N, D)
        st["x"].normal_()
        st["x_ref"].copy_(st["x"] * 0.99)
        st["delta"].normal_()
        st["has_ref"].fill_(1)
        v = torch.randn(N, D, device=dev)
        ws = torch.zeros(B.cache_workspace_bytes(N, D) // 4 + 1, device=dev)
        skip = torch.zeros(N, dtype=torch.uint8, device=dev)
        idx = torch.zeros(N, dtype=torch.int32, device=dev)
        nc = torch.zeros(1, dtype=torch.int32, device=dev)
        force = (torch.rand(N, device=dev) >= a.skip_frac).to(torch.uint8)

        def run():
            if a.kernel == "cache-fused":
                B.cache_decide_skip(st["x"], st["x_ref"], st["delta"], st["accum"], st["has_ref"], 20, 50, 0.6, 0.58,
                                    0.1, 5, 5, skip, idx, nc, ws, force=force)
                B.cache_apply_computed(st["x"], st["x_ref"], st["delta"], v, skip, 0.6, 0.58)
            else:
                B.cache_decide(st["x"], st["x_ref"], st["accum"], st["has_ref"], 20, 50, 0.1, 5, 5, skip, idx, nc,
                               ws, force=force)
                B.cache_apply(st["x"], st["x_ref"], st["delta"], v, skip, 0.6, 0.58)
        ms = _time_cold(run, a.reps, a.warmup)
        n_skip = int((force == 0).sum())
        byts = (n_skip * 16.0 + (N - n_skip) * 24.0) * D
        out.update(shape=dict(N=N, D=D, skipped=n_skip), ms=ms, gbs=byts / (ms / 1e3) / 1e9)
    print(json.dumps(out), flush=True)


if __name__ == "__main__":
    main()
