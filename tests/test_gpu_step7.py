"""GPU parity of Algorithm 1 steps 6-7 (gs_sparsify_average_sparsify): the
workers' Q(g^m), their average v (bit-equal to the fused sum divided by M in
fp32) and the re-sparsified Q(v), against the oracle on the same bytes."""
import numpy as np
import pytest

import oracle
import workloads
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


def _run(gs, g, kappa, iters, seed, step, kappa_v, iters_v, worker_v):
    import torch
    M, d = g.shape
    idx = torch.empty((M, d), dtype=torch.int32, device="cuda")
    val = torch.empty((M, d), dtype=torch.float32, device="cuda")
    nnz = torch.empty(M, dtype=torch.int32, device="cuda")
    v = torch.empty(d, dtype=torch.float32, device="cuda")
    idx_v = torch.empty(d, dtype=torch.int32, device="cuda")
    val_v = torch.empty(d, dtype=torch.float32, device="cuda")
    nnz_v = torch.empty(1, dtype=torch.int32, device="cuda")
    info = gs.info_tensor(M + 1)
    gs.gs_sparsify_average_sparsify(g, kappa, iters, seed, step, 0, idx, val, nnz, v, kappa_v, iters_v, worker_v,
                                    idx_v, val_v, nnz_v, info=info)
    assert gs.gs_sync_status() == gs.GS_OK
    # the same first stage through the fused sum: v is that sum / M, bit for bit
    out = torch.empty(d, dtype=torch.float32, device="cuda")
    idx2, val2, nnz2 = torch.empty_like(idx), torch.empty_like(val), torch.empty_like(nnz)
    gs.gs_sparsify_aggregate(g, kappa, iters, seed, step, 0, idx2, val2, nnz2, out)
    assert gs.gs_sync_status() == gs.GS_OK
    assert torch.equal(nnz2, nnz)
    want = (out.cpu().numpy() / np.float32(M)).astype(np.float32)
    np.testing.assert_array_equal(v.cpu().numpy(), want)
    return idx, val, nnz, v, idx_v, val_v, nnz_v, gs.decode_info(info)


def _check(gs, g, kappa, iters, seed, step, kappa_v, iters_v, worker_v, workers=None):
    M, d = g.shape
    idx, val, nnz, v, idx_v, val_v, nnz_v, recs = _run(gs, g, kappa, iters, seed, step, kappa_v, iters_v, worker_v)
    gh = g.float().cpu().numpy()
    n = nnz.cpu().numpy()
    flips = 0
    il, vl = [], []
    for m in range(M):
        ref = oracle.sparsify(gh[m], kappa, iters, seed, step, m)
        il.append(ref[0])
        vl.append(ref[1])
        if workers is None or m in workers:
            flips += compare_sparse(idx[m, :n[m]].cpu().numpy(), val[m, :n[m]].cpu().numpy(), gh[m], kappa, iters,
                                    seed, step, m, ref=ref)
    # v against the oracle's average of the oracle's lists
    v_ref = oracle.average(il, vl, d).astype(np.float64)
    mag = np.zeros(d)
    for i, vv in zip(il, vl):
        np.add.at(mag, i.astype(np.int64), np.abs(vv.astype(np.float64)))
    vh = v.cpu().numpy()
    assert np.all(np.abs(vh.astype(np.float64) - v_ref) <= 1e-5 * mag / M)
    # step 7 on the same bytes of v
    k = int(nnz_v.item())
    ref_v = oracle.sparsify(vh, kappa_v, iters_v, seed, step, worker_v)
    flips += compare_sparse(idx_v[:k].cpu().numpy(), val_v[:k].cpu().numpy(), vh, kappa_v, iters_v, seed, step,
                            worker_v, ref=ref_v)
    assert recs[M]["lambda"] == pytest.approx(ref_v[2]["lambda"], rel=1e-6)
    assert recs[M]["capped"] == ref_v[2]["capped"]
    assert set(idx_v[:k].cpu().numpy().tolist()) <= set(np.nonzero(vh)[0].tolist())
    return flips


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_average_sparsify_parity(gs, dtype):
    import torch
    rng = np.random.default_rng(4)
    M, d = 5, 100_003
    gh = (rng.standard_t(3, (M, d)) * rng.uniform(0.5, 2, (M, 1))).astype(np.float32)
    g = torch.from_numpy(gh).cuda()
    if dtype == "bf16":
        g = torch.from_numpy(workloads.f32_to_bf16_bits(gh).reshape(M, d)).cuda().view(torch.bfloat16)
    for kappa_v, iters_v in [(0.01, 2), (0.3, 3), (1.0, 0)]:
        assert _check(gs, g, 0.05, 2, 9, 3, kappa_v, iters_v, M) <= 2


def test_average_sparsify_full_student_t(gs):
    """The headline gradients (16 x 2^24): steps 4-7, workers 0 and 15 and the
    re-sparsified average checked in full."""
    import torch
    w = workloads.C3
    g = workloads.device_student_t(w.M, w.d, seed0=w.data_seed)
    assert _check(gs, g, w.kappa, w.iters, w.seed, w.step, w.kappa, w.iters, 2 ** 32 - 1, workers=[0, 15]) <= 3
    del g
    torch.cuda.empty_cache()
