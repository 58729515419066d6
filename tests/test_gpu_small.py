"""GPU parity of the cluster-resident path for short rows (d <= 2^21: one
thread-block cluster per worker runs Algorithm 3's passes, the draw and the
compaction; k_small_sum adds M > 1 workers).  Compared with the oracle on
the same seeded inputs: kept sets (flips only where |u - p| < 1e-6), values,
lambda, the capped count and the rescalings taken, and the worker-order sum;
plus the shapes where the cluster's layout changes (cluster size, shared-
memory caching of the share, ragged tiles), the path the library picks, and
the sum modes (plain, continued, averaged)."""
import numpy as np
import pytest

import oracle
import workloads
from parity import compare_sparse, compare_sum

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
    gs.gs_set_option(gs.GS_OPT_SMALL_PATH, 2)
    yield gs
    gs.gs_set_option(gs.GS_OPT_SMALL_PATH, 0)


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
    else:   # many exact ties
        g = rng.integers(-3, 4, d).astype(np.float64)
    return g.astype(np.float32)


def _run(gs, g_host, kappa, iters, seed, step, worker0, dtype="f32", out=False, g_dev=None):
    import torch
    M, d = g_host.shape
    g = g_dev if g_dev is not None else (
        _dev(workloads.f32_to_bf16_bits(g_host).reshape(M, d)).view(torch.bfloat16) if dtype == "bf16"
        else _dev(g_host))
    idx = torch.full((M, d), -1, dtype=torch.int32, device="cuda")
    val = torch.zeros((M, d), dtype=torch.float32, device="cuda")
    nnz = torch.zeros(M, dtype=torch.int32, device="cuda")
    inf = gs.info_tensor(M)
    if out:
        o = torch.full((d,), float("nan"), dtype=torch.float32, device="cuda")
        gs.gs_sparsify_aggregate(g, kappa, iters, seed, step, worker0, idx, val, nnz, o, info=inf)
    else:
        o = None
        gs.gs_batched_sparsify(g, kappa, iters, seed, step, worker0, idx, val, nnz, info=inf)
    return idx, val, nnz, gs.decode_info(inf), o


def _check(g_host, res, kappa, iters, seed, step, worker0):
    idx, val, nnz, infos, o = res
    M, d = g_host.shape
    n = nnz.cpu().numpy()
    flips = 0
    il, vl = [], []
    for m in range(M):
        ref = oracle.greedy_lambda(g_host[m], kappa, iters)
        ri, rv, _ = oracle.sparsify(g_host[m], kappa, iters, seed, step, worker0 + m)
        flips += compare_sparse(idx[m, :n[m]].cpu().numpy(), val[m, :n[m]].cpu().numpy(), g_host[m], kappa, iters,
                                seed, step, worker0 + m, ref=(ri, rv, ref))
        assert infos[m]["lambda"] == pytest.approx(ref["lambda"], rel=1e-6)
        assert infos[m]["capped"] == ref["capped"]
        if infos[m]["iters_run"] != ref["iters_run"]:
            # Only where the rescaling factor c is 1 up to the rounding of the
            # sums (fp32 pairs of four values added error-free: ~2^-24
            # relative, like the chunked path's streaming sums), so that
            # rounding decides c > 1: the extra rescalings then move lambda by
            # no more than that.
            assert infos[m]["lambda"] == pytest.approx(ref["lambda"], rel=4e-7)
        assert infos[m]["sum_p"] == pytest.approx(ref["sum_p"], rel=1e-6, abs=1e-9)
        assert infos[m]["flags"] == 0
        il.append(ri)
        vl.append(rv)
    if o is not None:
        compare_sum(o.cpu().numpy(), il, vl, d)
    return flips


# Cluster sizes 1 .. 12 (shares of ~4096 coordinates), shares cached in shared
# memory up to 40960 coordinates (d <= 655360) and re-read above, ragged tiles.
SHAPES = [1, 3, 127, 128, 129, 4095, 4096, 4097, 8193, 65536, 70_001, 655_360, 655_361, (1 << 20) + 3, 1 << 21]


@pytest.mark.parametrize("d", SHAPES)
def test_sizes_match_the_oracle(gs, d):
    kinds = ["t3", "lognormal", "normal", "ties"]
    M = 1 if d > 300_000 else 3
    g_host = np.stack([_vector(kinds[(d + m) % 4], d, d + m) for m in range(M)])
    for kappa, iters, seed, step, w0 in [(0.01, 3, 1, 0, 0), (0.2, 2, 2**33 + 5, 7, 9)]:
        res = _run(gs, g_host, kappa, iters, seed, step, w0, out=True)
        assert gs.gs_sync_status() == gs.GS_OK
        assert _check(g_host, res, kappa, iters, seed, step, w0) <= 1


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_bf16_and_unaligned_rows(gs, dtype):
    """bf16 input, and a row length that is not a multiple of 4 (every row but
    the first starts off the 16-byte grid), plus a base 4 bytes past it."""
    import torch
    M, d, kappa, iters, seed, step = 4, 50_001, 0.05, 3, 3, 2
    g_host = np.stack([_vector(k, d, 60 + m) for m, k in enumerate(["t3", "lognormal", "normal", "ties"])])
    if dtype == "bf16":
        g_host = workloads.bf16_bits_to_f32(workloads.f32_to_bf16_bits(g_host)).reshape(M, d)
    res = _run(gs, g_host, kappa, iters, seed, step, 0, dtype=dtype, out=True)
    assert gs.gs_sync_status() == gs.GS_OK
    assert _check(g_host, res, kappa, iters, seed, step, 0) <= 1
    if dtype == "f32":
        base = torch.zeros(M * d + 1, dtype=torch.float32, device="cuda")
        base[1:] = _dev(g_host.reshape(-1))
        g = base[1:].view(M, d)
        assert g.data_ptr() % 16 == 4
        res2 = _run(gs, g_host, kappa, iters, seed, step, 0, out=True, g_dev=g)
        assert gs.gs_sync_status() == gs.GS_OK
        for a, b in zip(res[:3], res2[:3]):
            assert torch.equal(a, b)
        assert torch.equal(res[4], res2[4])


def test_rows_do_not_depend_on_the_batch(gs):
    """A worker's result is a function of its own row, seed, step and id: the
    same row alone, or third of five, or with other neighbours, gives the same
    bits (every sum of the cluster path is in a fixed order)."""
    import torch
    d = 100_003
    rows = np.stack([_vector(k, d, 80 + m) for m, k in enumerate(["t3", "lognormal", "normal", "ties", "t3"])])
    a = _run(gs, rows, 0.03, 3, 4, 1, 10)
    b = _run(gs, rows[2:3], 0.03, 3, 4, 1, 12)
    c = _run(gs, rows[[4, 1, 2]], 0.03, 3, 4, 1, 10)
    k = int(a[2][2].item())
    assert int(b[2][0].item()) == k
    assert torch.equal(a[0][2, :k], b[0][0, :k]) and torch.equal(a[1][2, :k], b[1][0, :k])
    # rows[2] is the third row of c with id 12 as well
    assert torch.equal(a[0][2, :k], c[0][2, :k]) and torch.equal(a[1][2, :k], c[1][2, :k])


def test_path_choice_and_kernels(gs):
    """The automatic choice: rows of at most 2^21 coordinates in calls of at
    most 2^24 coordinates run k_small (+ k_small_sum for a sum over M > 1),
    others the chunked kernels; option 1 forces the chunked kernels."""
    import torch

    def launched(M, d, mode, out=True):
        gs.gs_set_option(gs.GS_OPT_SMALL_PATH, mode)
        g = torch.ones((M, d), dtype=torch.float32, device="cuda")
        idx = torch.empty((M, d), dtype=torch.int32, device="cuda")
        val = torch.empty((M, d), dtype=torch.float32, device="cuda")
        nnz = torch.empty(M, dtype=torch.int32, device="cuda")
        o = torch.empty(d, dtype=torch.float32, device="cuda")
        gs.gs_kernel_times()
        if out:
            gs.gs_sparsify_aggregate(g, 0.1, 2, 1, 0, 0, idx, val, nnz, o)
        else:
            gs.gs_batched_sparsify(g, 0.1, 2, 1, 0, 0, idx, val, nnz)
        torch.cuda.synchronize()
        assert gs.gs_sync_status() == gs.GS_OK
        return {k for k, (_, n) in gs.gs_kernel_times().items() if n}

    try:
        assert launched(1, 65536, 0) == {"k_small"}
        assert launched(8, 1 << 20, 0) == {"k_small", "k_small_sum"}
        assert launched(8, 1 << 20, 0, out=False) == {"k_small"}
        big = launched(17, 1 << 20, 0)        # M d above 2^24
        assert "k_small" not in big and "k_decide" in big
        assert "k_small" not in launched(1, (1 << 21) + 4, 2)   # row too long for the cluster path
        assert launched(17, 1 << 20, 2) == {"k_small", "k_small_sum"}
        assert "k_small" not in launched(1, 65536, 1)
    finally:
        gs.gs_set_option(gs.GS_OPT_SMALL_PATH, 2)


def test_sum_modes(gs):
    """Step 6 of Algorithm 1 through the cluster path: one worker (the cluster
    writes the dense vector itself) and several (k_small_sum), the average of
    gs_sparsify_average_sparsify, and the sum continued across worker groups
    by gs_pipeline_host, each against the oracle's worker-order fp32 sum."""
    import torch
    d, kappa, iters, seed, step = 30_011, 0.04, 2, 6, 3
    for M in (1, 5):
        g_host = np.stack([_vector(k, d, 120 + m) for m, k in enumerate(["lognormal", "t3", "normal", "ties", "t3"][:M])])
        res = _run(gs, g_host, kappa, iters, seed, step, 0, out=True)
        assert gs.gs_sync_status() == gs.GS_OK
        _check(g_host, res, kappa, iters, seed, step, 0)
    # the average (M = 5) and the step-7 resparsification of it
    g = _dev(g_host)
    M = g_host.shape[0]
    idx = torch.empty((M, d), dtype=torch.int32, device="cuda")
    val = torch.empty((M, d), dtype=torch.float32, device="cuda")
    nnz = torch.empty(M, dtype=torch.int32, device="cuda")
    v = torch.empty(d, dtype=torch.float32, device="cuda")
    iv = torch.empty(d, dtype=torch.int32, device="cuda")
    vv = torch.empty(d, dtype=torch.float32, device="cuda")
    nv = torch.empty(1, dtype=torch.int32, device="cuda")
    gs.gs_sparsify_average_sparsify(g, kappa, iters, seed, step, 0, idx, val, nnz, v, 0.1, 2, 99, iv, vv, nv)
    assert gs.gs_sync_status() == gs.GS_OK
    n = nnz.cpu().numpy()
    il = [idx[m, :n[m]].cpu().numpy() for m in range(M)]
    vl = [val[m, :n[m]].cpu().numpy() for m in range(M)]
    v_ref = oracle.average(il, vl, d)
    np.testing.assert_array_equal(v.cpu().numpy(), v_ref)
    k = int(nv.item())
    compare_sparse(iv[:k].cpu().numpy(), vv[:k].cpu().numpy(), v_ref, 0.1, 2, seed, step, 99)


def test_edge_cases(gs):
    import torch
    d = 9_001
    # all zero, one non-zero, kappa = 1, iters = 0
    z = np.zeros((2, d), np.float32)
    res = _run(gs, z, 0.1, 2, 1, 0, 0, out=True)
    assert gs.gs_sync_status() == gs.GS_OK and res[2].cpu().tolist() == [0, 0]
    assert bool((res[4] == 0).all())
    oh = np.zeros((1, d), np.float32)
    oh[0, 4321] = -2.5
    res = _run(gs, oh, 0.001, 3, 1, 0, 0)
    assert res[2].item() == 1 and res[0][0, 0].item() == 4321 and res[1][0, 0].item() == -2.5
    g = _vector("lognormal", d, 7)[None]
    g[0, ::5] = 0
    res = _run(gs, g, 1.0, 40, 1, 0, 0)
    k = int(res[2].item())
    np.testing.assert_array_equal(res[0][0, :k].cpu().numpy(), np.nonzero(g[0])[0])
    np.testing.assert_array_equal(res[1][0, :k].cpu().numpy(), g[0][g[0] != 0])
    g = _vector("t3", d, 8)[None]
    assert _check(g, _run(gs, g, 0.05, 0, 5, 1, 2), 0.05, 0, 5, 1, 2) <= 1
    # non-finite rows: reported, nothing kept in that row, the others unaffected
    for bad in (np.nan, np.inf, -np.inf):
        b = np.stack([_vector("normal", d, 1), _vector("normal", d, 2)])
        b[1, 777] = bad
        res = _run(gs, b, 0.1, 2, 1, 0, 0, out=True)
        assert gs.gs_sync_status() == gs.GS_ERR_NONFINITE
        assert res[2][1].item() == 0
        ri, _, _ = oracle.sparsify(b[0], 0.1, 2, 1, 0, 0)
        assert res[2][0].item() == ri.size
    # capacity: the true count is reported, the first cap entries written
    g = _vector("normal", d, 3)[None]
    idx = torch.full((1, 500 + 64), -9, dtype=torch.int32, device="cuda")
    val = torch.zeros((1, 500 + 64), dtype=torch.float32, device="cuda")
    nnz = torch.zeros(1, dtype=torch.int32, device="cuda")
    gs.gs_batched_sparsify(_dev(g), 0.5, 2, 1, 0, 0, idx[:, :500], val[:, :500], nnz)
    assert gs.gs_sync_status() == gs.GS_ERR_CAPACITY
    ri, rv, _ = oracle.sparsify(g[0], 0.5, 2, 1, 0, 0)
    assert int(nnz.item()) == ri.size > 500
    np.testing.assert_array_equal(idx[0, :500].cpu().numpy(), ri[:500])
    assert bool((idx[0, 500:] == -9).all())
    # ... and the sum holds the written entries only (one worker: the cluster
    # writes the sum itself; two: k_small_sum from the bits)
    for M in (1, 2):
        gm = np.stack([_vector("normal", d, 3 + m) for m in range(M)])
        idx = torch.empty((M, 500), dtype=torch.int32, device="cuda")
        val = torch.empty((M, 500), dtype=torch.float32, device="cuda")
        nnz = torch.zeros(M, dtype=torch.int32, device="cuda")
        o = torch.empty(d, dtype=torch.float32, device="cuda")
        gs.gs_sparsify_aggregate(_dev(gm), 0.5, 2, 1, 0, 0, idx, val, nnz, o)
        assert gs.gs_sync_status() == gs.GS_ERR_CAPACITY
        n = np.minimum(nnz.cpu().numpy(), 500)
        il = [idx[m, :n[m]].cpu().numpy() for m in range(M)]
        vl = [val[m, :n[m]].cpu().numpy() for m in range(M)]
        np.testing.assert_array_equal(o.cpu().numpy(), oracle.aggregate(il, vl, d))


def test_full_c1(gs):
    """The single-vector workload at its configured size (d = 65536,
    log-normal(0, 1.5) magnitudes, kappa 0.1, 2 rescalings), in the call and
    path bench.py times: the kept pairs and the dense reconstruction."""
    w = workloads.C1
    gs.gs_set_option(gs.GS_OPT_SMALL_PATH, 0)
    try:
        g = workloads.device_c1(w.d, seed=w.data_seed)
        g_host = g.cpu().numpy()
        res = _run(gs, g_host, w.kappa, w.iters, w.seed, w.step, 0, out=True, g_dev=g)
        assert gs.gs_sync_status() == gs.GS_OK
        assert _check(g_host, res, w.kappa, w.iters, w.seed, w.step, 0) <= 1
    finally:
        gs.gs_set_option(gs.GS_OPT_SMALL_PATH, 2)
