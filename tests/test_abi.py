"""The C ABI library loads and exports every entry point include/gs.h
declares; host-side argument checks answer without touching a GPU."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "gs.h")


def declared():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(gs_[a-z_0-9]+)\s*\(", text)))


@pytest.fixture(scope="module")
def gs():
    import __graft_entry__
    __graft_entry__.build()
    import paper_1710_09854_gb300 as gs
    return gs


def test_library_exports_every_declared_symbol(gs):
    names = declared()
    assert len(names) >= 12
    L = ctypes.CDLL(gs.LIB_PATH)
    for n in names:
        assert hasattr(L, n), n
    assert set(names) == set(gs.EXPORTS)


def test_status_strings_and_version(gs):
    assert gs.status_string(0) == "GS_OK"
    assert gs.status_string(4) == "GS_ERR_NONFINITE"
    assert gs.status_string(99) == "GS_UNKNOWN_STATUS"
    assert gs.gs_version() >= 100


def test_host_argument_checks(gs):
    L = gs.lib()
    inv = gs.GS_ERR_INVALID_ARG
    fake = 256  # never dereferenced: every call below fails validation first
    # kappa outside (0, 1], negative iters, empty vector, null pointers, bad dtype
    assert L.gs_batched_sparsify(fake, 0, 2, 100, 0.0, 2, 1, 0, 0, fake, fake, fake, 100, None, None) == inv
    assert L.gs_batched_sparsify(fake, 0, 2, 100, 1.5, 2, 1, 0, 0, fake, fake, fake, 100, None, None) == inv
    assert L.gs_batched_sparsify(fake, 0, 2, 100, 0.5, -1, 1, 0, 0, fake, fake, fake, 100, None, None) == inv
    assert L.gs_batched_sparsify(fake, 0, 0, 100, 0.5, 2, 1, 0, 0, fake, fake, fake, 100, None, None) == inv
    assert L.gs_batched_sparsify(fake, 0, 2, 0, 0.5, 2, 1, 0, 0, fake, fake, fake, 100, None, None) == inv
    assert L.gs_batched_sparsify(None, 0, 2, 100, 0.5, 2, 1, 0, 0, fake, fake, fake, 100, None, None) == inv
    assert L.gs_batched_sparsify(fake, 7, 2, 100, 0.5, 2, 1, 0, 0, fake, fake, fake, 100, None, None) == inv
    assert L.gs_batched_sparsify(fake, 0, 2, 100, 0.5, 2, 1, 0, 0, fake, fake, fake, 0, None, None) == inv
    assert L.gs_batched_sparsify(fake + 1, 0, 2, 100, 0.5, 2, 1, 0, 0, fake, fake, fake, 100, None, None) == inv
    assert L.gs_probabilities(fake, 1 << 31, 0.5, 2, fake, None) == inv
    assert L.gs_sparsify(fake, 10, float("nan"), 2, 1, 0, 0, fake, fake, fake, None) == inv
    # segment offsets must start at 0, increase strictly and end at d
    import numpy as np
    for off in ([0, 5, 5, 10], [1, 5, 10], [0, 5, 9]):
        o = np.array(off, dtype=np.int64)
        assert L.gs_segmented_sparsify(fake, 0, 1, 10, o.ctypes.data, o.size - 1, 0.5, 2, 1, 0, 0, fake, fake, fake,
                                       10, None, None) == inv
    # sparse sum: M out of range, null lists
    ip = (ctypes.c_void_p * 1)(fake)
    assert L.gs_sparse_aggregate(ip, ip, fake, 0, 10, fake, None) == inv
    assert L.gs_sparse_aggregate(ip, ip, fake, 513, 10, fake, None) == inv
    nul = (ctypes.c_void_p * 1)(None)
    assert L.gs_sparse_aggregate(nul, ip, fake, 1, 10, fake, None) == inv
    assert L.gs_random_words(1, 0, 0, -1, 4, fake, None) == inv
    # options
    assert L.gs_set_option(99, 0) == inv
    assert L.gs_set_option(gs.GS_OPT_SAMPLE_SIZE, 100) == inv
    assert L.gs_set_option(gs.GS_OPT_FORCE_EXACT_SOLVE, 2) == inv
    assert L.gs_set_option(gs.GS_OPT_SAMPLE_SIZE, 16384) == 0
    assert L.gs_set_option(gs.GS_OPT_SAMPLE_SIZE, 0) == 0   # back to the automatic size


def test_eps_entry_points_reject_bad_budgets():
    # Host-side validation: these return before any CUDA call.
    import paper_1710_09854_gb300 as gs
    L = gs.lib()
    fake = 256  # never dereferenced
    for eps in (-0.5, float("nan"), float("inf")):
        assert L.gs_probabilities_eps(fake, 10, eps, fake, None, None) == gs.GS_ERR_INVALID_ARG
        assert L.gs_batched_sparsify_eps(fake, 0, 1, 10, eps, 1, 0, 0, fake, fake, fake, 10, None,
                                         None) == gs.GS_ERR_INVALID_ARG


def test_average_sparsify_rejects_bad_arguments():
    # Host-side validation: these return before any CUDA call.
    import paper_1710_09854_gb300 as gs
    L = gs.lib()
    fake = 256  # never dereferenced
    args = lambda M, kv, iv, v: (fake, 0, M, 10, 0.1, 2, 1, 0, 0, fake, fake, fake, 10, v, kv, iv, 7, fake, fake,
                                 fake, None, None)
    assert L.gs_sparsify_average_sparsify(*args(0, 0.1, 2, fake)) == gs.GS_ERR_INVALID_ARG
    assert L.gs_sparsify_average_sparsify(*args(513, 0.1, 2, fake)) == gs.GS_ERR_INVALID_ARG
    assert L.gs_sparsify_average_sparsify(*args(4, 0.0, 2, fake)) == gs.GS_ERR_INVALID_ARG
    assert L.gs_sparsify_average_sparsify(*args(4, 0.1, -1, fake)) == gs.GS_ERR_INVALID_ARG
    assert L.gs_sparsify_average_sparsify(*args(4, 0.1, 2, None)) == gs.GS_ERR_INVALID_ARG


def test_training_loop_entry_points_reject_bad_arguments():
    # Host-side validation: these return before any CUDA call.
    import paper_1710_09854_gb300 as gs
    L = gs.lib()
    fake = 256  # never dereferenced
    bad = gs.GS_ERR_INVALID_ARG
    assert L.gs_logreg_grad(fake, fake, 10, 10, fake, fake, 2, 65, 0.0, fake, fake, None) == bad   # B > 64
    assert L.gs_logreg_grad(fake, fake, 10, 10, fake, fake, 2, 0, 0.0, fake, fake, None) == bad
    assert L.gs_logreg_grad(fake, fake, 10, 10, fake, fake, 2, 8, -1.0, fake, fake, None) == bad
    assert L.gs_logreg_margins(None, fake, 10, 10, fake, fake, None) == bad
    assert L.gs_row_sq_norms(fake, fake, 0, 10, fake, None) == bad
    assert L.gs_sum_rows(fake, 2, 0, fake, None) == bad
    assert L.gs_sgd_step(fake, fake, 10, 1.0, 0.1, 0.0, 0, fake, fake, 2, None, None) == bad       # T0 = 0
    assert L.gs_sgd_step(fake, fake, 10, 1.0, 0.1, 4.0, -1, fake, fake, 2, None, None) == bad      # t < 0


def test_selftest_timeout_rejects_unknown_kind():
    import paper_1710_09854_gb300 as gs
    assert gs.lib().gs_selftest_timeout(2, None) == gs.GS_ERR_INVALID_ARG


def test_tensors_must_live_on_the_current_device(monkeypatch):
    """The binding refuses a tensor of another device before any call."""
    import types
    import torch
    import paper_1710_09854_gb300 as gs
    monkeypatch.setattr(torch.cuda, "current_device", lambda: 0)
    t = types.SimpleNamespace(is_cuda=True, device=torch.device("cuda", 1), dtype=torch.float32,
                              is_contiguous=lambda: True, data_ptr=lambda: 4096)
    with pytest.raises(ValueError, match="current CUDA device"):
        gs._ptr(t, "g")
    t.device = torch.device("cuda", 0)
    assert gs._ptr(t, "g") == 4096
    cpu = types.SimpleNamespace(is_cuda=False)
    with pytest.raises(ValueError, match="CUDA tensor"):
        gs._ptr(cpu, "g")
