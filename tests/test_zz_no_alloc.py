"""The allocation-free cache decision (cs_cache_decide_noalloc) against cs_cache_decide.

Callers that cannot allocate device memory (a serving runtime whose pool owns the GPU,
or code that must not let an allocation synchronise the device) use the variant whose
scratch is a fixed array inside the library.  This file runs last so that a failure
here leaves every other test already run; it passes alone or after the others.
"""
import numpy as np
import pytest
import torch

from paper_2607_23159_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def B():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_23159_gb300 import binding
    torch.cuda.init()
    return binding


def _state(B, N, D, seed):
    st = B.new_state(N, D)
    if N * D <= 1 << 24:
        x = synth.normal(seed, (N, D))
        st["x"].copy_(torch.from_numpy(x))
        st["x_ref"].copy_(torch.from_numpy(x + 0.05 * synth.normal(seed + 1, (N, D))))
    else:                                      # the limit case: seeded normals drawn on the device
        g = torch.Generator(device="cuda").manual_seed(seed)
        st["x"].normal_(generator=g)
        st["x_ref"].normal_(generator=g).mul_(0.05).add_(st["x"])
    st["accum"].copy_(torch.from_numpy(synth.uniform(seed + 2, (N,), 0.0, 0.08)))
    st["has_ref"].fill_(1)
    st["has_ref"][0] = 0                       # one empty cache: must compute
    return st


def _decide(B, fn, st, k, T, tau, ws=None):
    N = st["x"].shape[0]
    accum = st["accum"].clone()
    has_ref = st["has_ref"].clone()
    skip = torch.full((N,), 9, dtype=torch.uint8, device="cuda")
    idx = torch.full((N,), -1, dtype=torch.int32, device="cuda")
    nc = torch.zeros(1, dtype=torch.int32, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    if ws is None:
        fn(st["x"], st["x_ref"], accum, has_ref, k, T, tau, 1, 1, skip, idx, nc, err=err)
    else:
        fn(st["x"], st["x_ref"], accum, has_ref, k, T, tau, 1, 1, skip, idx, nc, ws, err=err)
    torch.cuda.synchronize()
    assert int(err[0]) == 0
    n = int(nc[0])
    return skip.cpu(), idx.cpu()[:n], n, accum.cpu(), has_ref.cpu()


# (N, D, steps): free steps 4 and 5 of 10, or a free step followed by a warm-up (k = 1) or
# cool-down (k = 10) step, where no drift is evaluated and the partials left in the fixed
# array by the call before must not be read.  (64, 512 * 8192) fills the array exactly.
@pytest.mark.parametrize("N,D,steps", [(6, 50000, (4, 5)), (3, 2096640, (4, 5)), (5, 30000, (4, 1)),
                                       (4, 40000, (5, 10)), (64, 512 * 8192, (4, 5))])
def test_noalloc_decide_matches_workspace_decide_twice_in_a_row(B, N, D, steps):
    T, tau = 10, 0.1
    ws = torch.zeros(B.cache_workspace_bytes(N, D) // 4 + 1, device="cuda")
    for call, k in enumerate(steps):           # two calls in a row, different inputs
        st = _state(B, N, D, seed=10 * N + call)
        ref = _decide(B, B.cache_decide, st, k, T, tau, ws)
        got = _decide(B, B.cache_decide_noalloc, st, k, T, tau)
        assert torch.equal(got[0], ref[0])     # skip mask
        assert torch.equal(got[1], ref[1])     # compaction list
        assert got[2] == ref[2]
        np.testing.assert_allclose(got[3].numpy(), ref[3].numpy(), rtol=1e-6, atol=1e-7)
        assert torch.equal(got[4], ref[4])
        assert 0 < ref[2] <= N
        if k in (1, T):                        # window step: every candidate computes
            assert ref[2] == N and not got[0].any()
        elif N >= 6:
            assert ref[2] < N                  # some candidates skip on a free step


def test_noalloc_rejects_sizes_beyond_the_fixed_scratch(B):
    N, D = 65, 1024
    st = B.new_state(N, D)
    skip = torch.zeros(N, dtype=torch.uint8, device="cuda")
    idx = torch.zeros(N, dtype=torch.int32, device="cuda")
    nc = torch.zeros(1, dtype=torch.int32, device="cuda")
    with pytest.raises(B.CSError) as e:
        B.cache_decide_noalloc(st["x"], st["x_ref"], st["accum"], st["has_ref"], 3, 10, 0.1, 1, 1, skip, idx, nc)
    assert e.value.status == B.CS_ERR_ARG and "limit" in str(e.value)
    big = torch.zeros(1, 512 * 8192 + 1, device="cuda")
    with pytest.raises(B.CSError) as e:
        B.cache_decide_noalloc(big, big, st["accum"][:1], st["has_ref"][:1], 3, 10, 0.1, 1, 1, skip, idx, nc)
    assert e.value.status == B.CS_ERR_ARG and "limit" in str(e.value)
