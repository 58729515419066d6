"""gs_sparsify_noalloc: the single-worker sparsify that runs on the library's
static scratch, for callers that cannot allocate device memory during a call.
Its output must equal gs_sparsify's on the same inputs bit for bit, call
after call, although each call finds the previous call's leftovers in the
scratch; one call is also checked against the oracle directly.  This file is
named to be collected last, so that it also runs after every other GPU test
in the same process."""
import numpy as np
import pytest

import workloads
from parity import compare_sparse

MAX_D = 1 << 22


@pytest.fixture(scope="module")
def gs():
    import __graft_entry__
    __graft_entry__.build()
    import paper_1710_09854_gb300 as gs
    return gs


def test_noalloc_rejects_bad_arguments(gs):
    # Host-side validation fails before any CUDA call, so this runs without a GPU.
    L = gs.lib()
    fake = 256  # never dereferenced
    rc = L.gs_sparsify_noalloc(fake, MAX_D + 1, 0.01, 2, 1, 0, 0, fake, fake, fake, None, fake, None)
    assert rc == gs.GS_ERR_INVALID_ARG
    assert b"limit" in L.gs_last_error()
    assert L.gs_sparsify_noalloc(fake, 0, 0.01, 2, 1, 0, 0, fake, fake, fake, None, fake, None) == rc
    assert L.gs_sparsify_noalloc(None, 10, 0.01, 2, 1, 0, 0, fake, fake, fake, None, fake, None) == rc
    # The status word is required: it is the only place device-side errors go.
    assert L.gs_sparsify_noalloc(fake, 10, 0.01, 2, 1, 0, 0, fake, fake, fake, None, None, None) == rc
    assert b"status" in L.gs_last_error()


def _run_pair(gs, torch, g, kappa, iters, seed, step, worker):
    d = g.numel()
    dev = g.device
    out = {}
    for name in ("pool", "static"):
        idx = torch.full((d,), -7, dtype=torch.int32, device=dev)
        val = torch.full((d,), -7.0, dtype=torch.float32, device=dev)
        nnz = torch.zeros(1, dtype=torch.int32, device=dev)
        if name == "pool":
            gs.gs_sparsify(g, kappa, iters, seed, step, worker, idx, val, nnz)
            assert gs.gs_sync_status() == gs.GS_OK
            info = None
            code = None
        else:
            info = torch.zeros(gs.INFO_BYTES, dtype=torch.uint8, device=dev)
            code = torch.full((1,), -1, dtype=torch.int32, device=dev)
            gs.gs_sparsify_noalloc(g, kappa, iters, seed, step, worker, idx, val, nnz, code, info=info)
        torch.cuda.synchronize()
        n = int(nnz.item())
        out[name] = (n, idx[:n].cpu(), val[:n].cpu(), info, code)
    return out


def _assert_same(out):
    """The static-scratch call returns gs_sparsify's idx / val / nnz bit for bit."""
    n0, i0, v0, _, _ = out["pool"]
    n1, i1, v1, info, code = out["static"]
    assert int(code.item()) == 0
    assert n1 == n0 and n0 > 0
    np.testing.assert_array_equal(i1.numpy(), i0.numpy())
    np.testing.assert_array_equal(v1.numpy().view(np.uint32), v0.numpy().view(np.uint32))
    rec = info.cpu().numpy().view(np.uint8)
    lam = rec[:8].view(np.float64)[0]
    assert np.isfinite(lam) and lam > 0


@pytest.mark.gpu
def test_noalloc_matches_pool_path_on_consecutive_calls(gs):
    import torch
    dev = torch.device("cuda:0")
    # First call: the largest vector the static scratch takes, heavy tailed,
    # also compared with the oracle directly.
    g1 = workloads.device_student_t(1, MAX_D, seed0=11, device=dev)[0]
    a = _run_pair(gs, torch, g1, 0.01, 2, seed=5, step=3, worker=1)
    _assert_same(a)
    n, i, v, _, _ = a["static"]
    flips = compare_sparse(i.numpy(), v.numpy(), g1.cpu().numpy(), 0.01, 2, 5, 3, 1)
    assert flips <= 1
    # Second call, right after: a smaller ragged vector (several chunks and a
    # partial one, d % 4 != 0, so the generic-load streaming pass) that finds
    # the first call's leftovers in the scratch.
    g2 = workloads.device_student_t(1, 3 * 16384 + 1233, seed0=12, device=dev)[0]
    b = _run_pair(gs, torch, g2, 0.05, 2, seed=5, step=4, worker=0)
    _assert_same(b)
    # Third: a vector whose start is 4 bytes past a 16-byte boundary (the
    # generic pass again), over the second call's leftovers.
    base = workloads.device_student_t(1, 200_001, seed0=13, device=dev)[0]
    g3 = base[1:]
    assert g3.data_ptr() % 16 == 4
    c = _run_pair(gs, torch, g3, 0.02, 3, seed=9, step=1, worker=2)
    _assert_same(c)


@pytest.mark.gpu
def test_noalloc_takes_no_device_memory_and_reports_status(gs):
    import torch
    dev = torch.device("cuda:0")
    d = 200003
    g = workloads.device_student_t(1, d, seed0=21, device=dev)[0]
    idx = torch.empty(d, dtype=torch.int32, device=dev)
    val = torch.empty(d, dtype=torch.float32, device=dev)
    nnz = torch.zeros(1, dtype=torch.int32, device=dev)
    code = torch.full((1,), -1, dtype=torch.int32, device=dev)
    # The first call may set up (symbol lookup, code loading); later ones
    # must leave the device's free memory exactly as they found it.
    gs.gs_sparsify_noalloc(g, 0.02, 2, 1, 0, 0, idx, val, nnz, code)
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    for step in range(3):
        gs.gs_sparsify_noalloc(g, 0.02, 2, 1, step, 0, idx, val, nnz, code)
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0
    assert int(code.item()) == 0
    # A non-finite gradient is reported through the caller's status word ...
    bad = g.clone()
    bad[d // 2] = float("nan")
    gs.gs_sparsify_noalloc(bad, 0.02, 2, 1, 0, 0, idx, val, nnz, code)
    torch.cuda.synchronize()
    assert int(code.item()) == gs.GS_ERR_NONFINITE
    # ... not through gs_sync_status (the library's allocated status word) ...
    assert gs.gs_sync_status() == gs.GS_OK
    # ... and does not carry over into the next call.
    gs.gs_sparsify_noalloc(g, 0.02, 2, 1, 0, 0, idx, val, nnz, code)
    torch.cuda.synchronize()
    assert int(code.item()) == 0
