"""Device-side failure detection without a GPU fault: a bounded wait that runs
out is reported as GS_ERR_TIMEOUT through the status word, the status clears
on read, and the context keeps working (a normal call afterwards matches the
oracle).  Nothing here traps, faults or hangs."""
import time

import numpy as np
import pytest

from parity import compare_sparse

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def gs():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    import paper_1710_09854_gb300 as gs
    gs.gs_set_option(gs.GS_OPT_FORCE_EXACT_SOLVE, 0)
    assert gs.gs_sync_status() == gs.GS_OK
    return gs


@pytest.mark.parametrize("kind", [0, 1])
def test_wait_timeout_is_reported_and_the_context_survives(gs, kind):
    import torch
    t0 = time.monotonic()
    gs.gs_selftest_timeout(kind)
    assert gs.gs_sync_status() == gs.GS_ERR_TIMEOUT
    assert time.monotonic() - t0 < 60
    assert gs.gs_sync_status() == gs.GS_OK      # the status word clears on read
    d = 50003
    g = np.random.default_rng(kind).standard_t(3, d).astype(np.float32)
    idx = torch.empty(d, dtype=torch.int32, device="cuda")
    val = torch.empty(d, dtype=torch.float32, device="cuda")
    nnz = torch.empty(1, dtype=torch.int32, device="cuda")
    gs.gs_sparsify(torch.from_numpy(g).cuda(), 0.02, 2, 3, 1, 0, idx, val, nnz)
    assert gs.gs_sync_status() == gs.GS_OK
    n = int(nnz.item())
    assert compare_sparse(idx[:n].cpu().numpy(), val[:n].cpu().numpy(), g, 0.02, 2, 3, 1, 0) <= 1
