"""GPU parity: the CUDA path through the C ABI against the CPU oracle, on the
same seeded inputs, element by element (tolerances in tests/parity.py)."""
import numpy as np
import pytest

import oracle
import workloads
from parity import compare_probabilities, compare_sparse, compare_sum, oracle_rows

pytestmark = pytest.mark.gpu

SIZES = [1, 2, 3, 4, 5, 7, 31, 64, 1023, 4096, 4097, 16383, 16384, 16385, 50003, 65536, 200001]


@pytest.fixture(scope="module")
def gs():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    import paper_1710_09854_gb300 as gs
    gs.gs_set_option(gs.GS_OPT_FORCE_EXACT_SOLVE, 0)
    gs.gs_set_option(gs.GS_OPT_SAMPLE_SIZE, 0)
    assert gs.gs_sync_status() == gs.GS_OK
    return gs


@pytest.fixture(autouse=True)
def _path(gs, request):
    """Short rows take the chunked kernels here unless a test asks for the
    cluster-resident path (its `small` parameter); the full-size workloads
    take the path the library picks, as bench.py times them."""
    gs.gs_set_option(gs.GS_OPT_SMALL_PATH, 0 if request.node.name.startswith("test_full") else 1)
    yield
    gs.gs_set_option(gs.GS_OPT_SMALL_PATH, 0)


# 1: the chunked kernels; 2: one thread-block cluster per worker (rows of d <= 2^21).
BOTH_PATHS = pytest.mark.parametrize("small", [1, 2], ids=["chunked", "cluster"])


def _use(gs, small):
    gs.gs_set_option(gs.GS_OPT_SMALL_PATH, small)


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


def _sparsify_batched(gs, g_host, kappa, iters, seed, step, worker0=0, dtype="f32", cap=None, info=False):
    import torch
    M, d = g_host.shape
    cap = d if cap is None else cap
    g = _dev(g_host)
    if dtype == "bf16":
        g = _dev(workloads.f32_to_bf16_bits(g_host).reshape(M, d)).view(torch.bfloat16)
    idx = torch.full((M, cap), -1, dtype=torch.int32, device="cuda")
    val = torch.zeros((M, cap), dtype=torch.float32, device="cuda")
    nnz = torch.zeros(M, dtype=torch.int32, device="cuda")
    inf = gs.info_tensor(M) if info else None
    gs.gs_batched_sparsify(g, kappa, iters, seed, step, worker0, idx, val, nnz, info=inf)
    return idx, val, nnz, inf


# ---------------------------------------------------------------------------
def test_random_words_match_oracle(gs):
    import torch
    for seed, step, worker, i0, n in [(1, 0, 0, 0, 4099), (2**40 + 3, 9, 15, 2**33 + 1, 1001),
                                      (0xFFFFFFFFFFFFFFFF, 2**32 - 1, 2**32 - 1, 5, 77)]:
        out = torch.empty(n, dtype=torch.int32, device="cuda")
        gs.gs_random_words(seed, step, worker, i0, out)
        got = out.cpu().numpy().view(np.uint32)
        ref = (oracle.uniforms(seed, step, worker, i0, n) * 2.0**32).astype(np.uint64).astype(np.uint32)
        np.testing.assert_array_equal(got, ref)


@pytest.mark.parametrize("d", SIZES)
def test_probabilities_sizes(gs, d):
    import torch
    for kind, kappa, iters in [("t3", 0.01, 3), ("lognormal", 0.1, 2), ("normal", 0.5, 0), ("ties", 0.05, 10)]:
        g_host = _vector(kind, d, d * 7 + iters)
        p = torch.empty(d, dtype=torch.float32, device="cuda")
        info = gs.info_tensor(1)
        gs.gs_probabilities_ex(_dev(g_host), kappa, iters, p, info)
        assert gs.gs_sync_status() == gs.GS_OK
        ref_info, _ = compare_probabilities(p.cpu().numpy(), g_host, kappa, iters)
        got = gs.decode_info(info)[0]
        if ref_info["lambda"] > 0:
            assert got["lambda"] == pytest.approx(ref_info["lambda"], rel=1e-6)
            assert got["sum_p"] == pytest.approx(ref_info["sum_p"], rel=1e-6)


@pytest.mark.parametrize("d", SIZES)
@BOTH_PATHS
def test_sparsify_sizes(gs, d, small):
    _use(gs, small)
    import torch
    for kind, kappa, iters, seed, step, worker in [("t3", 0.01, 3, 1, 0, 0), ("lognormal", 0.1, 2, 99, 5, 3),
                                                   ("normal", 0.3, 1, 2**35 + 1, 2**31, 2**32 - 2),
                                                   ("ties", 0.5, 4, 7, 1, 1)]:
        g_host = _vector(kind, d, d + step)
        idx = torch.empty(d, dtype=torch.int32, device="cuda")
        val = torch.empty(d, dtype=torch.float32, device="cuda")
        nnz = torch.empty(1, dtype=torch.int32, device="cuda")
        gs.gs_sparsify(_dev(g_host), kappa, iters, seed, step, worker, idx, val, nnz)
        assert gs.gs_sync_status() == gs.GS_OK
        n = int(nnz.item())
        flips = compare_sparse(idx[:n].cpu().numpy(), val[:n].cpu().numpy(), g_host, kappa, iters, seed, step, worker)
        assert flips <= 1


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@BOTH_PATHS
def test_batched_parity(gs, dtype, small):
    _use(gs, small)
    M, d, kappa, iters, seed, step, w0 = 5, 100_003, 0.02, 3, 11, 7, 3
    g_host = np.stack([_vector(k, d, 50 + m) for m, k in enumerate(["t3", "lognormal", "normal", "t3", "ties"])])
    if dtype == "bf16":
        g_host = workloads.bf16_bits_to_f32(workloads.f32_to_bf16_bits(g_host)).reshape(M, d)
    idx, val, nnz, inf = _sparsify_batched(gs, g_host, kappa, iters, seed, step, w0, dtype, info=True)
    assert gs.gs_sync_status() == gs.GS_OK
    n = nnz.cpu().numpy()
    ii, vv = idx.cpu().numpy(), val.cpu().numpy()
    infos = gs.decode_info(inf)
    flips = 0
    for m in range(M):
        flips += compare_sparse(ii[m, :n[m]], vv[m, :n[m]], g_host[m], kappa, iters, seed, step, w0 + m)
        ref = oracle.greedy_lambda(g_host[m], kappa, iters)
        assert infos[m]["lambda"] == pytest.approx(ref["lambda"], rel=1e-6)
        assert infos[m]["capped"] == ref["capped"]
    assert flips <= 1


@BOTH_PATHS
def test_single_equals_batched_row(gs, small):
    _use(gs, small)
    import torch
    M, d = 3, 70_001
    g_host = np.stack([_vector("lognormal", d, 900 + m) for m in range(M)])
    idx, val, nnz, _ = _sparsify_batched(gs, g_host, 0.05, 2, 5, 3, worker0=10)
    for m in range(M):
        i1 = torch.empty(d, dtype=torch.int32, device="cuda")
        v1 = torch.empty(d, dtype=torch.float32, device="cuda")
        n1 = torch.empty(1, dtype=torch.int32, device="cuda")
        gs.gs_sparsify(_dev(g_host[m]), 0.05, 2, 5, 3, 10 + m, i1, v1, n1)
        k = int(nnz[m].item())
        assert int(n1.item()) == k
        assert torch.equal(i1[:k], idx[m, :k]) and torch.equal(v1[:k], val[m, :k])


@BOTH_PATHS
def test_deterministic(gs, small):
    _use(gs, small)
    import torch
    M, d = 4, 300_001
    g_host = np.stack([_vector("t3", d, 77 + m) for m in range(M)])
    a = _sparsify_batched(gs, g_host, 0.01, 3, 1, 0)
    b = _sparsify_batched(gs, g_host, 0.01, 3, 1, 0)
    assert torch.equal(a[2], b[2])
    for m in range(M):
        k = int(a[2][m].item())
        assert torch.equal(a[0][m, :k], b[0][m, :k]) and torch.equal(a[1][m, :k], b[1][m, :k])


def test_forced_exact_and_small_sample(gs):
    M, d, kappa, iters = 3, 120_007, 0.03, 3
    g_host = np.stack([_vector(k, d, 31 + m) for m, k in enumerate(["lognormal", "t3", "ties"])])
    for opt, val in [(gs.GS_OPT_FORCE_EXACT_SOLVE, 1), (gs.GS_OPT_SAMPLE_SIZE, 256)]:
        gs.gs_set_option(opt, val)
        try:
            idx, v, nnz, inf = _sparsify_batched(gs, g_host, kappa, iters, 3, 2, info=True)
            assert gs.gs_sync_status() == gs.GS_OK
        finally:
            gs.gs_set_option(gs.GS_OPT_FORCE_EXACT_SOLVE, 0)
            gs.gs_set_option(gs.GS_OPT_SAMPLE_SIZE, 0)
        n = nnz.cpu().numpy()
        for m in range(M):
            compare_sparse(idx[m, :n[m]].cpu().numpy(), v[m, :n[m]].cpu().numpy(), g_host[m], kappa, iters, 3, 2, m)
        if opt == gs.GS_OPT_FORCE_EXACT_SOLVE:
            assert all(r["flags"] & 1 for r in gs.decode_info(inf))


@pytest.mark.parametrize("sample", [0, 1024, 256])
def test_segmented_parity(gs, sample):
    """Layer-wise calls against the oracle, layer by layer.  The bound's
    sample size decides how its short segments (at most 1024 values) are
    taken: the default packs them a warp each, several to a CTA; a sample of
    1024 leaves one per CTA; 256 sends every segment through one CTA each."""
    gs.gs_set_option(gs.GS_OPT_SAMPLE_SIZE, sample)
    try:
        _segmented_parity(gs)
    finally:
        gs.gs_set_option(gs.GS_OPT_SAMPLE_SIZE, 0)


def _segmented_parity(gs):
    import torch
    rng = np.random.default_rng(4)
    lens = [64, 3, 1, 17000, 5, 40000, 64, 16384, 2, 1024, 1025, 700, 9]
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    M, d = 3, int(off[-1])
    g_host = np.stack([(rng.standard_normal(d) * rng.choice([1e-3, 1, 50], d)).astype(np.float32) for _ in range(M)])
    kappa, iters, seed, step = 0.05, 2, 8, 4
    g = _dev(g_host)
    idx = torch.empty((M, d), dtype=torch.int32, device="cuda")
    val = torch.empty((M, d), dtype=torch.float32, device="cuda")
    nnz = torch.empty(M, dtype=torch.int32, device="cuda")
    inf = gs.info_tensor(M * (off.size - 1))
    gs.gs_segmented_sparsify(g, off, kappa, iters, seed, step, 0, idx, val, nnz, info=inf)
    assert gs.gs_sync_status() == gs.GS_OK
    infos = gs.decode_info(inf)
    n = nnz.cpu().numpy()
    for m in range(M):
        ri, rv, lams = oracle.segmented_sparsify(g_host[m], off, kappa, iters, seed, step, m)
        got_i, got_v = idx[m, :n[m]].cpu().numpy(), val[m, :n[m]].cpu().numpy()
        # per segment comparison against the oracle's per-layer result
        for l in range(off.size - 1):
            a, b = off[l], off[l + 1]
            sel = (got_i >= a) & (got_i < b)
            r = oracle.sparsify(g_host[m, a:b], kappa, iters, seed, step, m, i0=a)
            compare_sparse(got_i[sel], got_v[sel], g_host[m, a:b], kappa, iters, seed, step, m, i0=a, ref=r)
            assert infos[m * (off.size - 1) + l]["lambda"] == pytest.approx(lams[l], rel=1e-6)
    _check_segmented_fused(gs, g, off, kappa, iters, seed, step, idx, val, nnz)


def _check_segmented_fused(gs, g, off, kappa, iters, seed, step, idx, val, nnz):
    """gs_segmented_sparsify_aggregate equals gs_segmented_sparsify followed by
    gs_sparse_aggregate, bit for bit (lists, counts and the sum)."""
    import torch
    M, d = g.shape
    out = torch.empty(d, dtype=torch.float32, device="cuda")
    gs.gs_sparse_aggregate([idx[m] for m in range(M)], [val[m] for m in range(M)], nnz, d, out)
    idx2, val2, nnz2 = torch.full_like(idx, -1), torch.zeros_like(val), torch.zeros_like(nnz)
    out2 = torch.full_like(out, float("nan"))
    gs.gs_segmented_sparsify_aggregate(g, off, kappa, iters, seed, step, 0, idx2, val2, nnz2, out2)
    assert gs.gs_sync_status() == gs.GS_OK
    assert torch.equal(nnz2, nnz)
    assert torch.equal(out2, out)
    for m in range(M):
        k = int(nnz[m].item())
        assert torch.equal(idx2[m, :k], idx[m, :k]) and torch.equal(val2[m, :k], val[m, :k])


def test_aggregate_parity_and_validation(gs):
    import torch
    rng = np.random.default_rng(3)
    for M, d in [(1, 1), (3, 8191), (16, 100_000), (7, 3 * 8192 + 5)]:
        il, vl = [], []
        for m in range(M):
            k = int(rng.integers(0, min(d, 5000) + 1))
            il.append(np.sort(rng.choice(d, size=k, replace=False)).astype(np.int32))
            vl.append((rng.standard_normal(k) * 10 ** rng.uniform(-3, 3, k)).astype(np.float32))
        nnz = torch.tensor([x.size for x in il], dtype=torch.int32, device="cuda")
        it = [_dev(x) if x.size else torch.zeros(1, dtype=torch.int32, device="cuda") for x in il]
        vt = [_dev(x) if x.size else torch.zeros(1, dtype=torch.float32, device="cuda") for x in vl]
        out = torch.full((d,), float("nan"), dtype=torch.float32, device="cuda")
        gs.gs_sparse_aggregate(it, vt, nnz, d, out)
        assert gs.gs_sync_status() == gs.GS_OK
        ref = compare_sum(out.cpu().numpy(), il, vl, d)
        np.testing.assert_array_equal(out.cpu().numpy(), ref)   # same fp32 adds in the same order
    # unsorted and out-of-range lists are reported
    for bad in (np.array([5, 3, 9], np.int32), np.array([1, 1, 2], np.int32), np.array([0, 10], np.int32)):
        out = torch.zeros(10, dtype=torch.float32, device="cuda")
        gs.gs_sparse_aggregate([_dev(bad)], [_dev(np.ones(bad.size, np.float32))],
                               torch.tensor([bad.size], dtype=torch.int32, device="cuda"), 10, out)
        assert gs.gs_sync_status() == gs.GS_ERR_INVALID_ARG


@BOTH_PATHS
def test_edge_cases(gs, small):
    _use(gs, small)
    import torch
    d = 40_000
    # all zero: nothing kept
    z = np.zeros((2, d), np.float32)
    idx, val, nnz, inf = _sparsify_batched(gs, z, 0.1, 2, 1, 0, info=True)
    assert gs.gs_sync_status() == gs.GS_OK and nnz.cpu().tolist() == [0, 0]
    # kappa = 1 with enough iterations: every non-zero coordinate capped and kept as is
    g = _vector("lognormal", d, 5)
    g[::3] = 0
    idx, val, nnz, _ = _sparsify_batched(gs, g[None], 1.0, 40, 1, 0)
    k = int(nnz.item())
    np.testing.assert_array_equal(idx[0, :k].cpu().numpy(), np.nonzero(g)[0])
    np.testing.assert_array_equal(val[0, :k].cpu().numpy(), g[g != 0])
    # equal magnitudes: p = kappa everywhere (uniform sampling)
    e = np.where(np.arange(d) % 2 == 0, 2.0, -2.0).astype(np.float32)
    p = torch.empty(d, dtype=torch.float32, device="cuda")
    gs.gs_probabilities(_dev(e), 0.25, 3, p)
    np.testing.assert_allclose(p.cpu().numpy(), 0.25, rtol=1e-6)
    # one-hot
    oh = np.zeros(d, np.float32)
    oh[12345] = -3.0
    gs.gs_probabilities(_dev(oh), 0.001, 2, p)
    want = np.zeros(d)
    want[12345] = 1
    np.testing.assert_array_equal(p.cpu().numpy(), want)
    # non-finite gradients are reported
    for bad in (np.nan, np.inf, -np.inf):
        b = _vector("normal", d, 1)
        b[777] = bad
        _sparsify_batched(gs, b[None], 0.1, 2, 1, 0)
        assert gs.gs_sync_status() == gs.GS_ERR_NONFINITE
    # capacity overflow: true count reported, writes clipped
    g = _vector("normal", d, 2)
    idx, val, nnz, _ = _sparsify_batched(gs, g[None], 0.5, 2, 1, 0, cap=100)
    assert gs.gs_sync_status() == gs.GS_ERR_CAPACITY
    assert int(nnz.item()) > 100
    ri, rv, _ = oracle.sparsify(g, 0.5, 2, 1, 0, 0)
    assert int(nnz.item()) == ri.size
    np.testing.assert_array_equal(idx[0].cpu().numpy(), ri[:100])


@BOTH_PATHS
def test_pipeline_host_matches_device_path(gs, small):
    _use(gs, small)
    import torch
    M, d, kappa, iters, seed, step = 4, 65_537, 0.05, 2, 3, 1
    g_host = np.stack([_vector("t3", d, 10 + m) for m in range(M)])
    gh = torch.from_numpy(g_host).pin_memory()
    g_dev = torch.empty((M, d), dtype=torch.float32, device="cuda")
    idx = torch.empty((M, d), dtype=torch.int32, device="cuda")
    val = torch.empty((M, d), dtype=torch.float32, device="cuda")
    nnz = torch.empty(M, dtype=torch.int32, device="cuda")
    out = torch.empty(d, dtype=torch.float32, device="cuda")
    out_h = torch.empty(d, dtype=torch.float32).pin_memory()
    nnz_h = torch.empty(M, dtype=torch.int32).pin_memory()
    gs.gs_pipeline_host(gh, kappa, iters, seed, step, 0, g_dev, idx, val, nnz, out, out_h, nnz_h)
    torch.cuda.synchronize()
    assert gs.gs_sync_status() == gs.GS_OK
    il, vl = [], []
    for m in range(M):
        ri, rv, _ = oracle.sparsify(g_host[m], kappa, iters, seed, step, m)
        il.append(ri)
        vl.append(rv)
        assert nnz_h[m].item() == ri.size
    compare_sum(out_h.numpy(), il, vl, d)


@BOTH_PATHS
def test_pipeline_host_equals_the_fused_call(gs, small):
    """gs_pipeline_host copies worker groups while earlier groups compute and
    continues the sum across groups: its outputs equal one gs_sparsify_aggregate
    call's bit for bit (bf16 input, more workers than groups, a ragged d)."""
    _use(gs, small)
    import torch
    M, d, kappa, iters, seed, step = 19, 70_001, 0.03, 3, 4, 2
    g_host = np.stack([_vector(k, d, 300 + m) for m, k in enumerate(["t3", "lognormal", "normal"] * 6 + ["ties"])])
    g_host = workloads.bf16_bits_to_f32(workloads.f32_to_bf16_bits(g_host)).reshape(M, d)
    bits = workloads.f32_to_bf16_bits(g_host).reshape(M, d)
    g = _dev(bits).view(torch.bfloat16)
    outs = []
    for pipe in (False, True):
        idx = torch.full((M, d), -1, dtype=torch.int32, device="cuda")
        val = torch.zeros((M, d), dtype=torch.float32, device="cuda")
        nnz = torch.zeros(M, dtype=torch.int32, device="cuda")
        out = torch.full((d,), float("nan"), dtype=torch.float32, device="cuda")
        if pipe:
            gh = torch.from_numpy(bits).view(torch.bfloat16).pin_memory()
            g_dev = torch.empty_like(g)
            out_h = torch.empty(d, dtype=torch.float32).pin_memory()
            nnz_h = torch.empty(M, dtype=torch.int32).pin_memory()
            gs.gs_pipeline_host(gh, kappa, iters, seed, step, 0, g_dev, idx, val, nnz, out, out_h, nnz_h)
            torch.cuda.synchronize()
            assert torch.equal(out_h, out.cpu()) and torch.equal(nnz_h, nnz.cpu())
        else:
            gs.gs_sparsify_aggregate(g, kappa, iters, seed, step, 0, idx, val, nnz, out)
        assert gs.gs_sync_status() == gs.GS_OK
        outs.append((idx, val, nnz, out))
    (i0, v0, n0, o0), (i1, v1, n1, o1) = outs
    assert torch.equal(n0, n1) and torch.equal(o0, o1)
    for m in range(M):
        k = int(n0[m].item())
        assert torch.equal(i0[m, :k], i1[m, :k]) and torch.equal(v0[m, :k], v1[m, :k])


# ---------------------------------------------------------------------------
# Full-size workloads in the launch configuration bench.py times.
# ---------------------------------------------------------------------------
def _full_check(gs, g_dev, kappa, iters, seed=1, step=0, workers=None, offsets=None, dtype="f32"):
    """The fused call bench.py times (gs_sparsify_aggregate, or the layer-wise
    gs_segmented_sparsify_aggregate) on a full-size input; the separate calls
    (sparsify, then gs_sparse_aggregate) must equal it bit for bit.  Every
    worker in `workers` (default: all) is compared with the oracle element by
    element, and the fused sum with the oracle's worker-order sum of the
    oracle's own lists over all M workers.  Returns the boundary flips."""
    import torch
    M, d = g_dev.shape
    idx = torch.empty((M, d), dtype=torch.int32, device="cuda")
    val = torch.empty((M, d), dtype=torch.float32, device="cuda")
    nnz = torch.empty(M, dtype=torch.int32, device="cuda")
    out = torch.empty(d, dtype=torch.float32, device="cuda")
    if offsets is None:
        gs.gs_sparsify_aggregate(g_dev, kappa, iters, seed, step, 0, idx, val, nnz, out)
    else:
        gs.gs_segmented_sparsify_aggregate(g_dev, offsets, kappa, iters, seed, step, 0, idx, val, nnz, out)
    assert gs.gs_sync_status() == gs.GS_OK
    # The separate calls equal the fused one bit for bit (lists, counts, sum).
    idx2, val2 = torch.full_like(idx, -1), torch.zeros_like(val)
    nnz2, out2 = torch.zeros_like(nnz), torch.full_like(out, float("nan"))
    if offsets is None:
        gs.gs_batched_sparsify(g_dev, kappa, iters, seed, step, 0, idx2, val2, nnz2)
    else:
        gs.gs_segmented_sparsify(g_dev, offsets, kappa, iters, seed, step, 0, idx2, val2, nnz2)
    gs.gs_sparse_aggregate([idx2[m] for m in range(M)], [val2[m] for m in range(M)], nnz2, d, out2)
    assert gs.gs_sync_status() == gs.GS_OK
    assert torch.equal(nnz2, nnz)
    assert torch.equal(out2, out)
    for m in range(M):
        k = int(nnz[m].item())
        assert torch.equal(idx2[m, :k], idx[m, :k]) and torch.equal(val2[m, :k], val[m, :k])
    del idx2, val2, out2
    g_host = g_dev.float().cpu().numpy() if dtype == "bf16" else g_dev.cpu().numpy()
    rows = [g_host[m] for m in range(M)]
    if offsets is None:
        refs = oracle_rows(oracle.sparsify, rows, kappa, iters, seed, step)
    else:
        refs = oracle_rows(oracle.segmented_sparsify, rows, offsets, kappa, iters, seed, step)
    n = nnz.cpu().numpy()
    workers = range(M) if workers is None else workers
    flips = 0
    for m in workers:
        gi = idx[m, :n[m]].cpu().numpy()
        gv = val[m, :n[m]].cpu().numpy()
        if offsets is None:
            flips += compare_sparse(gi, gv, rows[m], kappa, iters, seed, step, m, ref=refs[m])
        else:
            np.testing.assert_array_equal(gi, refs[m][0])
            np.testing.assert_allclose(gv, refs[m][1], rtol=1e-5)
    compare_sum(out.cpu().numpy(), [r[0] for r in refs], [r[1] for r in refs], d)
    return flips


def test_full_student_t_d2p24_m16(gs):
    """The headline workload (M=16, d=2^24, kappa=0.01, 3 iterations)."""
    import torch
    w = workloads.C3
    g = workloads.device_student_t(w.M, w.d, seed0=w.data_seed)
    flips = _full_check(gs, g, w.kappa, w.iters, w.seed, w.step)
    assert flips <= 2
    del g
    torch.cuda.empty_cache()


def test_full_resnet50_layerwise_m8(gs):
    """The layer-wise workload at its configured size: 8 workers x 161
    ResNet-50-shaped layers (25,557,032 coordinates), every worker and the sum."""
    import torch
    w = workloads.C4
    g, off = workloads.device_layerwise(w.M, seed0=w.data_seed)
    _full_check(gs, g, w.kappa, w.iters, w.seed, w.step, offsets=off)
    del g
    torch.cuda.empty_cache()


def test_full_logreg_c2(gs):
    """The logistic-regression workload at its configured size, all 8 workers."""
    import torch
    w = workloads.C2
    g = workloads.device_logreg(w.M, w.d, seed0=w.data_seed)
    _full_check(gs, g, w.kappa, w.iters, w.seed, w.step)
    del g
    torch.cuda.empty_cache()


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("kappa", [0.001, 0.01, 0.1])
def test_full_lognormal_outliers_c5(gs, kappa, dtype):
    """The large workload at its configured size: 8 workers x 2^27 log-normal
    magnitudes with 0.1% outliers, fp32 and bf16, each kappa of the sweep;
    every worker compared with the oracle and the fused sum over all 8."""
    import torch
    w = workloads.C5
    g = workloads.device_lognormal(w.M, w.d, seed0=w.data_seed)
    if dtype == "bf16":
        g = workloads.device_to_bf16(g)
        torch.cuda.empty_cache()
    flips = _full_check(gs, g, kappa, w.iters, w.seed, w.step, dtype=dtype)
    assert flips <= 2
    del g
    torch.cuda.empty_cache()


@pytest.mark.parametrize("path", [1, 2])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_stream_paths(gs, path, dtype):
    """The generic-load and the TMA streaming kernels both match the oracle,
    on full stages, partial stages and chunk starts inside a 128-byte row."""
    import torch
    gs.gs_set_option(gs.GS_OPT_STREAM_PATH, path)
    try:
        gs.gs_kernel_times()
        M, d = 3, (1 << 20) + 64 * 3 + 64       # d % 64 == 0: whole rows for both dtypes
        g_host = np.stack([_vector(k, d, 70 + m) for m, k in enumerate(["t3", "lognormal", "ties"])])
        if dtype == "bf16":
            g_host = workloads.bf16_bits_to_f32(workloads.f32_to_bf16_bits(g_host)).reshape(M, d)
        idx, val, nnz, _ = _sparsify_batched(gs, g_host, 0.02, 3, 9, 4, 2, dtype)
        assert gs.gs_sync_status() == gs.GS_OK
        n = nnz.cpu().numpy()
        for m in range(M):
            compare_sparse(idx[m, :n[m]].cpu().numpy(), val[m, :n[m]].cpu().numpy(), g_host[m], 0.02, 3, 9, 4, 2 + m)
        # layer-wise with offsets that are multiples of 4 but not of a row
        lens = [64, 1000, 4, 17004, 36, 40000, 20, 16384 * 2 + 4, 12]
        off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
        d2 = int(off[-1])
        M2 = 2                                      # M * d2 a multiple of 32 (fp32) and 64 (bf16)
        assert (M2 * d2) % (32 if dtype == "f32" else 64) == 0
        rng = np.random.default_rng(5)
        g2 = np.stack([(rng.standard_normal(d2) * rng.choice([1e-3, 1, 50], d2)).astype(np.float32)
                       for _ in range(M2)])
        if dtype == "bf16":
            g2 = workloads.bf16_bits_to_f32(workloads.f32_to_bf16_bits(g2)).reshape(M2, d2)
            gd = _dev(workloads.f32_to_bf16_bits(g2).reshape(M2, d2)).view(torch.bfloat16)
        else:
            gd = _dev(g2)
        idx = torch.empty((M2, d2), dtype=torch.int32, device="cuda")
        val = torch.empty((M2, d2), dtype=torch.float32, device="cuda")
        nnz = torch.empty(M2, dtype=torch.int32, device="cuda")
        gs.gs_segmented_sparsify(gd, off, 0.05, 2, 8, 4, 0, idx, val, nnz)
        assert gs.gs_sync_status() == gs.GS_OK
        n = nnz.cpu().numpy()
        for m in range(M2):
            ri, rv, _ = oracle.segmented_sparsify(g2[m], off, 0.05, 2, 8, 4, m)
            got_i = idx[m, :n[m]].cpu().numpy()
            got_v = val[m, :n[m]].cpu().numpy()
            for l in range(off.size - 1):
                a, b = off[l], off[l + 1]
                sel = (got_i >= a) & (got_i < b)
                r = oracle.sparsify(g2[m, a:b], 0.05, 2, 8, 4, m, i0=a)
                compare_sparse(got_i[sel], got_v[sel], g2[m, a:b], 0.05, 2, 8, 4, m, i0=a, ref=r)
        times = gs.gs_kernel_times()
        if path == 2:
            assert times["k_stream_tma"][1] == 2 and times["k_stream"][1] == 0
        else:
            assert times["k_stream"][1] == 2 and times["k_stream_tma"][1] == 0
    finally:
        gs.gs_set_option(gs.GS_OPT_STREAM_PATH, 0)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@BOTH_PATHS
def test_sparsify_aggregate_fused(gs, dtype, small):
    """gs_sparsify_aggregate equals gs_batched_sparsify + gs_sparse_aggregate
    bit for bit, and the oracle's worker-order sum."""
    _use(gs, small)
    import torch
    M, d, kappa, iters, seed, step = 6, 3 * 16384 + 1000, 0.03, 3, 21, 2
    g_host = np.stack([_vector(k, d, 400 + m) for m, k in enumerate(["t3", "lognormal", "normal"] * 2)])
    if dtype == "bf16":
        g_host = workloads.bf16_bits_to_f32(workloads.f32_to_bf16_bits(g_host)).reshape(M, d)
        g = _dev(workloads.f32_to_bf16_bits(g_host).reshape(M, d)).view(torch.bfloat16)
    else:
        g = _dev(g_host)
    for cap in (d, 700):   # 700 < kept count for some workers: the sum uses only the written entries
        idx = torch.empty((M, cap), dtype=torch.int32, device="cuda")
        val = torch.empty((M, cap), dtype=torch.float32, device="cuda")
        nnz = torch.empty(M, dtype=torch.int32, device="cuda")
        out = torch.empty(d, dtype=torch.float32, device="cuda")
        gs.gs_sparsify_aggregate(g, kappa, iters, seed, step, 0, idx, val, nnz, out)
        rc = gs.gs_sync_status()
        n = np.minimum(nnz.cpu().numpy(), cap)
        if cap == d:
            assert rc == gs.GS_OK
            out2 = torch.empty(d, dtype=torch.float32, device="cuda")
            gs.gs_sparse_aggregate([idx[m] for m in range(M)], [val[m] for m in range(M)], nnz, d, out2)
            assert gs.gs_sync_status() == gs.GS_OK
            assert torch.equal(out, out2)
            il, vl = [], []
            for m in range(M):
                ri, rv, _ = oracle.sparsify(g_host[m], kappa, iters, seed, step, m)
                compare_sparse(idx[m, :n[m]].cpu().numpy(), val[m, :n[m]].cpu().numpy(), g_host[m], kappa, iters,
                               seed, step, m, ref=(ri, rv, oracle.greedy_lambda(g_host[m], kappa, iters)))
                il.append(ri)
                vl.append(rv)
            compare_sum(out.cpu().numpy(), il, vl, d)
        else:
            assert rc == gs.GS_ERR_CAPACITY
            il = [idx[m, :n[m]].cpu().numpy() for m in range(M)]
            vl = [val[m, :n[m]].cpu().numpy() for m in range(M)]
            np.testing.assert_array_equal(out.cpu().numpy(), oracle.aggregate(il, vl, d))


@BOTH_PATHS
def test_sparsify_aggregate_fused_long_runs_many_workers(gs, small):
    """The fused sum with more than 32 workers (several worker batches per
    slice) and kappa large enough that runs exceed 32 entries per slice."""
    _use(gs, small)
    import torch
    M, d, kappa, iters, seed, step = 40, 2 * 16384 + 777, 0.2, 2, 5, 9
    kinds = ["t3", "lognormal", "normal", "ties"]
    g_host = np.stack([_vector(kinds[m % 4], d, 700 + m) for m in range(M)])
    g = _dev(g_host)
    idx = torch.empty((M, d), dtype=torch.int32, device="cuda")
    val = torch.empty((M, d), dtype=torch.float32, device="cuda")
    nnz = torch.empty(M, dtype=torch.int32, device="cuda")
    out = torch.empty(d, dtype=torch.float32, device="cuda")
    gs.gs_sparsify_aggregate(g, kappa, iters, seed, step, 0, idx, val, nnz, out)
    assert gs.gs_sync_status() == gs.GS_OK
    out2 = torch.empty(d, dtype=torch.float32, device="cuda")
    gs.gs_sparse_aggregate([idx[m] for m in range(M)], [val[m] for m in range(M)], nnz, d, out2)
    assert gs.gs_sync_status() == gs.GS_OK
    assert torch.equal(out, out2)
    n = nnz.cpu().numpy()
    assert n.max() * 1024 / d > 32   # kept entries per 1024-coordinate slice well above 32
    il, vl = [], []
    for m in range(M):
        ri, rv, _ = oracle.sparsify(g_host[m], kappa, iters, seed, step, m)
        compare_sparse(idx[m, :n[m]].cpu().numpy(), val[m, :n[m]].cpu().numpy(), g_host[m], kappa, iters, seed,
                       step, m, ref=(ri, rv, oracle.greedy_lambda(g_host[m], kappa, iters)))
        il.append(ri)
        vl.append(rv)
    compare_sum(out.cpu().numpy(), il, vl, d)


@pytest.mark.parametrize("force_exact", [0, 1])
def test_cluster_solve_large_budget(gs, force_exact):
    """Budgets above 2^20 run the solve on a cluster of CTAs per segment; with
    heavy tails at a large kappa the capped-candidate set is far too large for
    shared memory, so every pass walks the chunks (and the forced exact
    fallback runs on the cluster's first CTA)."""
    import torch
    M, d, kappa, iters = 2, (1 << 23) + 4 * 777, 0.2, 3
    g = workloads.device_lognormal(M, d, seed0=31)
    gs.gs_set_option(gs.GS_OPT_FORCE_EXACT_SOLVE, force_exact)
    try:
        flips = _full_check(gs, g, kappa, iters, seed=4, step=6)
    finally:
        gs.gs_set_option(gs.GS_OPT_FORCE_EXACT_SOLVE, 0)
    assert flips <= 2
    del g
    torch.cuda.empty_cache()


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("kind,kappa,d", [("t3", 0.02, 3 * 16384 + 1000), ("lognormal", 0.2, 2 * 16384 + 4),
                                          ("normal", 0.05, 40_001)])
def test_hybrid_code(gs, dtype, kind, kappa, d):
    """gs_batched_sparsify_hybrid (section 3.3, eqs. 9-10): its Q_A / Q_B equal
    the oracle's split of the plain lists bit for bit, decode to exactly the
    plain output, and match the oracle's Q(g)."""
    import torch
    M, iters, seed, step = 4, 3, 13, 5
    g_host = np.stack([_vector(kind, d, 900 + m) for m in range(M)])
    if dtype == "bf16":
        g_host = workloads.bf16_bits_to_f32(workloads.f32_to_bf16_bits(g_host)).reshape(M, d)
        g = _dev(workloads.f32_to_bf16_bits(g_host).reshape(M, d)).view(torch.bfloat16)
    else:
        g = _dev(g_host)
    idx, val, nnz, inf = _sparsify_batched(gs, g_host, kappa, iters, seed, step, 0, dtype, info=True)
    assert gs.gs_sync_status() == gs.GS_OK
    qa_i = torch.empty((M, d), dtype=torch.int32, device="cuda")
    qa_v = torch.empty((M, d), dtype=torch.float32, device="cuda")
    qb = torch.empty((M, d), dtype=torch.int32, device="cuda")
    na = torch.empty(M, dtype=torch.int32, device="cuda")
    nb = torch.empty(M, dtype=torch.int32, device="cuda")
    il = torch.empty(M, dtype=torch.float32, device="cuda")
    info = torch.zeros(M * gs.INFO_BYTES, dtype=torch.uint8, device="cuda")
    gs.gs_batched_sparsify_hybrid(g, kappa, iters, seed, step, 0, qa_i, qa_v, qb, na, nb, il, info=info)
    assert gs.gs_sync_status() == gs.GS_OK
    rec = gs.decode_info(info)
    n = nnz.cpu().numpy()
    na_h, nb_h, il_h = na.cpu().numpy(), nb.cpu().numpy(), il.cpu().numpy()
    for m in range(M):
        lam = rec[m]["lambda"]
        gi = idx[m, :n[m]].cpu().numpy()
        gv = val[m, :n[m]].cpu().numpy()
        ea, ev, eb, einv = oracle.hybrid_encode(g_host[m], lam, gi, gv)
        got_a = qa_i[m, :na_h[m]].cpu().numpy()
        got_v = qa_v[m, :na_h[m]].cpu().numpy()
        got_b = qb[m, :nb_h[m]].cpu().numpy().view(np.uint32)
        np.testing.assert_array_equal(got_a, ea)
        np.testing.assert_array_equal(got_v, ev)
        np.testing.assert_array_equal(got_b, eb)
        assert il_h[m] == np.float32(einv)
        assert na_h[m] == rec[m]["capped"]
        di, dv = oracle.hybrid_decode(got_a, got_v, got_b, float(il_h[m]))
        np.testing.assert_array_equal(di, gi)
        np.testing.assert_array_equal(dv, gv)
        compare_sparse(di, dv, g_host[m], kappa, iters, seed, step, m)


@BOTH_PATHS
def test_outputs_stay_inside_their_buffers(gs, small):
    """Guard bands: every output sits inside a larger sentinel-filled buffer;
    after each call the band past the buffer and, within each row, the slots
    past the written count still hold the sentinel."""
    _use(gs, small)
    import torch
    G = 4096
    SI, SV = -123456789, -7.5e33
    M, d = 5, 50003
    g_host = np.stack([_vector(k, d, 90 + m) for m, k in enumerate(["t3", "lognormal", "normal", "t3", "ties"])])
    g = _dev(g_host)

    def bands(shape, dtype, fill):
        n = int(np.prod(shape))
        full = torch.full((n + G,), fill, dtype=dtype, device="cuda")
        return full, full[:n].view(*shape)

    def check_tail(full, n, fill):
        assert bool((full[n:] == fill).all()), "write past the end of an output buffer"

    def check_rows(view, counts, fill):
        for m, k in enumerate(counts):
            assert bool((view[m, min(int(k), view.shape[1]):] == fill).all()), "write past a row's count"

    for cap in (d, 1000):
        fi, idx = bands((M, cap), torch.int32, SI)
        fv, val = bands((M, cap), torch.float32, SV)
        fn, nnz = bands((M,), torch.int32, SI)
        fo, out = bands((d,), torch.float32, SV)
        gs.gs_sparsify_aggregate(g, 0.02, 3, 5, 1, 0, idx, val, nnz, out)
        rc = gs.gs_sync_status()
        assert rc == (gs.GS_OK if cap == d else gs.GS_ERR_CAPACITY)
        counts = nnz.cpu().numpy()
        check_tail(fi, M * cap, SI)
        check_tail(fv, M * cap, SV)
        check_tail(fn, M, SI)
        check_tail(fo, d, SV)
        check_rows(idx, counts, SI)
        check_rows(val, counts, SV)
    # the hybrid code
    fa, qa_i = bands((M, d), torch.int32, SI)
    fav, qa_v = bands((M, d), torch.float32, SV)
    fb, qb = bands((M, d), torch.int32, SI)
    fna, n_a = bands((M,), torch.int32, SI)
    fnb, n_b = bands((M,), torch.int32, SI)
    fl, il = bands((M,), torch.float32, SV)
    gs.gs_batched_sparsify_hybrid(g, 0.05, 2, 5, 2, 0, qa_i, qa_v, qb, n_a, n_b, il)
    assert gs.gs_sync_status() == gs.GS_OK
    for full, n, fill in ((fa, M * d, SI), (fav, M * d, SV), (fb, M * d, SI), (fna, M, SI), (fnb, M, SI), (fl, M, SV)):
        check_tail(full, n, fill)
    check_rows(qa_i, n_a.cpu().numpy(), SI)
    check_rows(qb, n_b.cpu().numpy(), SI)
    # Algorithm 2 and the probabilities
    fi, idx = bands((M, d), torch.int32, SI)
    fv, val = bands((M, d), torch.float32, SV)
    fn, nnz = bands((M,), torch.int32, SI)
    gs.gs_batched_sparsify_eps(g, 0.5, 5, 3, 0, idx, val, nnz)
    assert gs.gs_sync_status() == gs.GS_OK
    check_tail(fi, M * d, SI)
    check_tail(fv, M * d, SV)
    check_rows(idx, nnz.cpu().numpy(), SI)
    fp, p = bands((d,), torch.float32, SV)
    gs.gs_probabilities(g[0].contiguous(), 0.02, 3, p)
    assert gs.gs_sync_status() == gs.GS_OK
    check_tail(fp, d, SV)
