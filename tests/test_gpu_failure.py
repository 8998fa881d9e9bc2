"""Failure detection on the GPU without a GPU fault: a bounded device-side wait that
nothing satisfies gives up, reports CS_ERR_TIMEOUT through the device error word, and
the CUDA context stays usable for the next kernel."""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def B():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_23159_gb300 import binding
    torch.cuda.init()
    return binding


def test_unsatisfied_wait_times_out_and_context_survives(B):
    err = torch.zeros(4, dtype=torch.int32, device="cuda")
    B.selftest_bounded_wait(err)
    torch.cuda.synchronize()                      # ~2 s: the wait's time limit
    assert int(err[0]) == B.CS_ERR_TIMEOUT
    # the context still runs kernels: a top-k on fresh data
    scores = torch.tensor([0.5, 2.0, -1.0, 2.0, float("nan")], device="cuda")
    idx = torch.zeros(5, dtype=torch.int32, device="cuda")
    B.select_topk(scores, 5, idx)
    torch.cuda.synchronize()
    assert idx.cpu().tolist() == [1, 3, 0, 2, 4]
