"""Failure detection without a GPU fault: a device wait that nothing satisfies gives up after
its bounded limit, reports PTD_ERR_TIMEOUT through the status word, and the context keeps
working (the next calls run and give correct results)."""
import time

import numpy as np
import pytest
import torch

import oracle
from paper_2607_10661_gb300 import ptd

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__

    __graft_entry__.build()


def test_bounded_wait_times_out_and_the_context_survives():
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    torch.cuda.synchronize()
    t0 = time.time()
    assert ptd.check_bounded_wait(status) == 1
    torch.cuda.synchronize()
    dt = time.time() - t0
    assert int(status.item()) == ptd.TIMEOUT
    assert 1.5 < dt < 30.0                      # the 2 s limit, not an endless wait
    # the context still works: a top-k call right after, checked against the oracle
    g = np.random.default_rng(3)
    x = g.normal(size=(5, 3000)).astype(np.float32)
    idx = torch.empty((5, 4), dtype=torch.int32, device="cuda")
    val = torch.empty((5, 4), dtype=torch.float32, device="cuda")
    ptd.topk_draft(torch.tensor(x, device="cuda"), 4, idx, val)
    torch.cuda.synchronize()
    assert np.array_equal(idx.cpu().numpy(), oracle.topk_rows(x, 4)[0])
