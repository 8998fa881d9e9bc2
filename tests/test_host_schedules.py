"""Host-side schedule helpers of the product (CPU): the time grid and the static
every-k-th-step schedule in search.py agree with the oracle's, and the paper-density
plan of bench.py has the paper's skip count with the warm-up and cool-down windows
computing."""
import os
import sys

import numpy as np
import pytest

from oracle import cachedsearch_oracle as O

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def S():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_23159_gb300 import search
    return search


@pytest.mark.parametrize("T", [1, 3, 10, 30, 50])
def test_time_grid_matches_oracle(S, T):
    np.testing.assert_array_equal(S.time_grid(T), O.time_grid(T))


@pytest.mark.parametrize("T,K_w,K_c,every", [(50, 5, 5, 3), (30, 3, 3, 2), (10, 1, 1, 1), (50, 5, 5, 7), (12, 0, 0, 4)])
def test_static_schedule_matches_oracle(S, T, K_w, K_c, every):
    got = [S.static_schedule(k, T, K_w, K_c, every) for k in range(1, T + 1)]
    ref = [bool(O.static_schedule(k, T, K_w, K_c, every)) for k in range(1, T + 1)]
    assert got == ref


@pytest.mark.parametrize("T,K_w,K_c", [(50, 5, 5), (30, 3, 3), (10, 1, 1)])
def test_paper_density_plan(T, K_w, K_c):
    sys.path.insert(0, ROOT)
    import bench
    plan = bench.paper_density_plan(T, K_w, K_c)
    assert len(plan) == T
    assert all(plan[k - 1] for k in range(1, T + 1) if k <= K_w or k > T - K_c)
    assert plan.count(False) == round(T * 26 / 50)     # 26 of 50 steps skipped (App. Reproducibility)
