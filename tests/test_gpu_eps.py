"""GPU parity of Algorithm 2 (section 3.2, the variance budget eps): the
CUDA path through the C ABI (gs_probabilities_eps, gs_batched_sparsify_eps)
against the oracle's sort-based restatement, on the same seeded inputs and
with the tolerances of tests/parity.py."""
import numpy as np
import pytest

import oracle
import workloads
from parity import P_RTOL, compare_sparse

pytestmark = pytest.mark.gpu

SIZES = [1, 2, 3, 5, 31, 1023, 4097, 16384, 16385, 50003, 200001]


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


def _dev(x):
    import torch
    return torch.from_numpy(np.ascontiguousarray(x)).cuda()


def _vector(kind, d, seed):
    rng = np.random.default_rng(seed)
    if kind == "t3":
        g = rng.standard_t(3, d)
        g[rng.random(d) < 0.01] = 0
    elif kind == "lognormal":
        g = rng.lognormal(0, 2, d) * np.where(rng.random(d) < 0.5, -1, 1)
        g[rng.random(d) < 0.001] *= 100
    elif kind == "normal":
        g = rng.standard_normal(d)
    elif kind == "ties":
        g = rng.integers(-3, 4, d).astype(np.float64)
    else:
        raise ValueError(kind)
    return g.astype(np.float32)


def _check_p(p_gpu, g, eps):
    p_ref, info = oracle.probabilities_eps(g, eps)
    p_gpu = np.asarray(p_gpu, dtype=np.float64)
    zero = p_ref == 0
    assert np.all(p_gpu[zero] == 0)
    rel = np.abs(p_gpu[~zero] - p_ref[~zero]) / p_ref[~zero]
    assert (rel.max() if rel.size else 0.0) <= P_RTOL
    return info


@pytest.mark.parametrize("d", SIZES)
def test_eps_probabilities_sizes(gs, d):
    import torch
    for kind, eps in [("t3", 0.05), ("lognormal", 1.0), ("normal", 0.3), ("ties", 2.0), ("t3", 20.0)]:
        g = _vector(kind, d, 3 * d + int(eps * 10))
        p = torch.empty(d, dtype=torch.float32, device="cuda")
        info = gs.info_tensor(1)
        gs.gs_probabilities_eps(_dev(g), eps, p, info)
        assert gs.gs_sync_status() == gs.GS_OK
        ref = _check_p(p.cpu().numpy(), g, eps)
        got = gs.decode_info(info)[0]
        assert got["flags"] == 0
        if ref["lambda"] > 0:
            assert got["lambda"] == pytest.approx(ref["lambda"], rel=1e-6)
            assert got["capped"] == ref["capped"]
            assert got["sum_p"] == pytest.approx(ref["sum_p"], rel=1e-6)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_eps_batched_parity(gs, dtype):
    import torch
    M, d, eps, seed, step, w0 = 5, 100_003, 0.5, 13, 2, 4
    g_host = np.stack([_vector(k, d, 70 + m) for m, k in enumerate(["t3", "lognormal", "normal", "t3", "ties"])])
    g = _dev(g_host)
    if dtype == "bf16":
        g_host = workloads.bf16_bits_to_f32(workloads.f32_to_bf16_bits(g_host)).reshape(M, d)
        g = _dev(workloads.f32_to_bf16_bits(g_host).reshape(M, d)).view(torch.bfloat16)
    idx = torch.full((M, d), -1, dtype=torch.int32, device="cuda")
    val = torch.zeros((M, d), dtype=torch.float32, device="cuda")
    nnz = torch.zeros(M, dtype=torch.int32, device="cuda")
    info = gs.info_tensor(M)
    gs.gs_batched_sparsify_eps(g, eps, seed, step, w0, idx, val, nnz, info=info)
    assert gs.gs_sync_status() == gs.GS_OK
    n = nnz.cpu().numpy()
    ii, vv = idx.cpu().numpy(), val.cpu().numpy()
    recs = gs.decode_info(info)
    flips = 0
    for m in range(M):
        ref = oracle.sparsify_eps(g_host[m], eps, seed, step, w0 + m)
        flips += compare_sparse(ii[m, :n[m]], vv[m, :n[m]], g_host[m], None, None, seed, step, w0 + m, ref=ref)
        assert recs[m]["lambda"] == pytest.approx(ref[2]["lambda"], rel=1e-6)
        assert recs[m]["capped"] == ref[2]["capped"]
    assert flips <= 1
    # the same call again gives the same bits
    idx2, val2, nnz2 = torch.full_like(idx, -1), torch.zeros_like(val), torch.zeros_like(nnz)
    gs.gs_batched_sparsify_eps(g, eps, seed, step, w0, idx2, val2, nnz2)
    assert gs.gs_sync_status() == gs.GS_OK
    assert torch.equal(nnz2, nnz) and torch.equal(idx2, idx) and torch.equal(val2, val)


def test_eps_take_all_matches(gs):
    # With every coordinate a candidate (the forced mode), the Newton solve runs
    # on the whole vector and must give the same answer.
    import torch
    d = 3 * 16384 + 77
    g = _vector("t3", d, 5)
    p = torch.empty(d, dtype=torch.float32, device="cuda")
    info = gs.info_tensor(1)
    gs.gs_set_option(gs.GS_OPT_FORCE_EXACT_SOLVE, 1)
    try:
        gs.gs_probabilities_eps(_dev(g), 0.2, p, info)
        assert gs.gs_sync_status() == gs.GS_OK
    finally:
        gs.gs_set_option(gs.GS_OPT_FORCE_EXACT_SOLVE, 0)
    ref = _check_p(p.cpu().numpy(), g, 0.2)
    assert gs.decode_info(info)[0]["lambda"] == pytest.approx(ref["lambda"], rel=1e-6)


def test_eps_degenerate_inputs(gs):
    import torch
    d = 40000
    # eps = 0: every non-zero coordinate kept with its own value
    g = _vector("t3", d, 9)
    idx = torch.empty((1, d), dtype=torch.int32, device="cuda")
    val = torch.empty((1, d), dtype=torch.float32, device="cuda")
    nnz = torch.empty(1, dtype=torch.int32, device="cuda")
    gs.gs_batched_sparsify_eps(_dev(g[None]), 0.0, 1, 0, 0, idx, val, nnz)
    assert gs.gs_sync_status() == gs.GS_OK
    n = int(nnz.item())
    nz = np.nonzero(g)[0]
    assert n == nz.size
    np.testing.assert_array_equal(idx[0, :n].cpu().numpy(), nz)
    np.testing.assert_allclose(val[0, :n].cpu().numpy(), g[nz], rtol=1e-6)
    # tiny budgets (every coordinate a candidate; the solve may finish by bisection)
    p = torch.empty(d, dtype=torch.float32, device="cuda")
    for e in (0.0, 1e-9, 2.0 ** -20, 2.0 ** -19):
        info = gs.info_tensor(1)
        gs.gs_probabilities_eps(_dev(g), e, p, info)
        assert gs.gs_sync_status() == gs.GS_OK
        ref = _check_p(p.cpu().numpy(), g, e)
        assert gs.decode_info(info)[0]["lambda"] == pytest.approx(ref["lambda"], rel=1e-6)
    # equal magnitudes: p = 1 / (1 + eps) everywhere
    h = (0.5 * np.where(np.arange(d) % 3 == 0, -1.0, 1.0)).astype(np.float32)
    gs.gs_probabilities_eps(_dev(h), 3.0, p)
    assert gs.gs_sync_status() == gs.GS_OK
    np.testing.assert_allclose(p.cpu().numpy(), 0.25, rtol=1e-6)
    # g = 0: nothing kept
    z = np.zeros(d, np.float32)
    gs.gs_batched_sparsify_eps(_dev(z[None]), 0.5, 1, 0, 0, idx, val, nnz)
    assert gs.gs_sync_status() == gs.GS_OK
    assert int(nnz.item()) == 0
    # a NaN is reported
    bad = g.copy()
    bad[d // 3] = np.nan
    gs.gs_batched_sparsify_eps(_dev(bad[None]), 0.5, 1, 0, 0, idx, val, nnz)
    assert gs.gs_sync_status() == gs.GS_ERR_NONFINITE


def test_eps_full_student_t_d2p24_m16(gs):
    """The headline gradients (M=16, d=2^24, Student-t) under a variance
    budget; workers 0 and 15 are checked against the oracle in full."""
    import torch
    w = workloads.C3
    g = workloads.device_student_t(w.M, w.d, seed0=w.data_seed)
    M, d = g.shape
    eps = 4.0
    idx = torch.empty((M, d), dtype=torch.int32, device="cuda")
    val = torch.empty((M, d), dtype=torch.float32, device="cuda")
    nnz = torch.empty(M, dtype=torch.int32, device="cuda")
    info = gs.info_tensor(M)
    gs.gs_batched_sparsify_eps(g, eps, w.seed, w.step, 0, idx, val, nnz, info=info)
    assert gs.gs_sync_status() == gs.GS_OK
    recs = gs.decode_info(info)
    n = nnz.cpu().numpy()
    flips = 0
    for m in (0, M - 1):
        gh = g[m].cpu().numpy()
        ref = oracle.sparsify_eps(gh, eps, w.seed, w.step, m)
        assert recs[m]["lambda"] == pytest.approx(ref[2]["lambda"], rel=1e-6)
        assert recs[m]["capped"] == ref[2]["capped"]
        flips += compare_sparse(idx[m, :n[m]].cpu().numpy(), val[m, :n[m]].cpu().numpy(), gh, None, None, w.seed,
                                w.step, m, ref=ref)
    assert flips <= 2
    for m in range(M):
        assert recs[m]["flags"] == 0 and recs[m]["iters_run"] <= 16
    del g, idx, val
    torch.cuda.empty_cache()
