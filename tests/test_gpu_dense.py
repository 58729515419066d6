"""GPU parity of the dense code of Q(g) (section 3.3, last paragraph): the
CUDA encoder's words must equal the oracle encoder's bit for bit on the same
q~ (and chunk size), the CUDA decoder must give q~ back from either side's
code, and malformed codes and short capacities are reported."""
import numpy as np
import pytest

import oracle
import workloads
from parity import oracle_rows

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def gs():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    import paper_1710_09854_gb300 as gs
    return gs


def _dev(x):
    import torch
    return torch.from_numpy(np.ascontiguousarray(x)).cuda()


def _hybrid_from_q(qs, cap):
    """The hybrid lists (Q_A indices, Q_B codes 2 i + [negative]) of dense q~ rows."""
    M = len(qs)
    qa = np.full((M, cap), -1, np.int32)
    qb = np.zeros((M, cap), np.uint32)
    na = np.zeros(M, np.int32)
    nb = np.zeros(M, np.int32)
    for m, q in enumerate(qs):
        a = np.nonzero(q == 2)[0]
        b = np.nonzero((q == 1) | (q == -1))[0]
        qa[m, :a.size] = a
        qb[m, :b.size] = 2 * b.astype(np.uint32) + (q[b] == -1)
        na[m], nb[m] = a.size, b.size
    return qa, qb, na, nb


def _encode(gs, qa, qb, na, nb, d, log2_k, word_cap):
    import torch
    M = qa.shape[0]
    words = torch.full((M, word_cap), -1, dtype=torch.int16, device="cuda")
    n_words = torch.zeros(M, dtype=torch.int64, device="cuda")
    gs.gs_dense_encode(_dev(qa), _dev(qb.view(np.int32)), _dev(na), _dev(nb), d, log2_k, words, n_words)
    return words, n_words


def _random_q(rng, d, density, p_cap):
    q = np.zeros(d, np.int8)
    hit = rng.random(d) < density
    q[hit] = rng.choice(np.array([1, -1, 2], np.int8), int(hit.sum()), p=[(1 - p_cap) / 2, (1 - p_cap) / 2, p_cap])
    return q


@pytest.mark.parametrize("d,densities,log2_k", [(1, (1.0, 0.0), 4), (1000, (0.01, 0.5, 0.0), 4),
                                                (65_537, (0.1, 0.002, 0.9), 9), (300_003, (0.03, 0.3), 10),
                                                (1 << 20, (0.01, 0.0005, 0.2, 0.05), 6)])
def test_words_equal_the_oracle_and_round_trip(gs, d, densities, log2_k):
    import torch
    rng = np.random.default_rng(d + log2_k)
    qs = [_random_q(rng, d, p, 0.02 if i % 2 else 0.3) for i, p in enumerate(densities)]
    ref = [oracle.dense_encode(q, log2_k) for q in qs]
    word_cap = max(r.size for r in ref) + 7
    qa, qb, na, nb = _hybrid_from_q(qs, d)
    words, n_words = _encode(gs, qa, qb, na, nb, d, log2_k, word_cap)
    assert gs.gs_sync_status() == gs.GS_OK
    nw = n_words.cpu().numpy()
    got = words.cpu().numpy().view(np.uint16)
    for m, r in enumerate(ref):
        assert nw[m] == r.size
        np.testing.assert_array_equal(got[m, :r.size], r)
    # the GPU decoder on the GPU's code and on the oracle's code
    qt = torch.full((len(qs), d), 99, dtype=torch.int8, device="cuda")
    gs.gs_dense_decode(words, n_words, d, qt)
    assert gs.gs_sync_status() == gs.GS_OK
    np.testing.assert_array_equal(qt.cpu().numpy(), np.stack(qs))
    ow = np.zeros((len(qs), word_cap), np.uint16)
    for m, r in enumerate(ref):
        ow[m, :r.size] = r
    qt2 = torch.zeros((len(qs), d), dtype=torch.int8, device="cuda")
    gs.gs_dense_decode(_dev(ow.view(np.int16)), _dev(np.array([r.size for r in ref], np.int64)), d, qt2)
    assert gs.gs_sync_status() == gs.GS_OK
    np.testing.assert_array_equal(qt2.cpu().numpy(), np.stack(qs))


def test_capacity_and_malformed_codes(gs):
    import torch
    rng = np.random.default_rng(3)
    d = 50_000
    qs = [_random_q(rng, d, 0.05, 0.1), _random_q(rng, d, 0.001, 0.1)]
    ref = [oracle.dense_encode(q, 8) for q in qs]
    qa, qb, na, nb = _hybrid_from_q(qs, d)
    # capacity between the two codes' lengths: the short one is written, the long one reported
    cap = (ref[0].size + ref[1].size) // 2
    assert ref[1].size <= cap < ref[0].size
    words, n_words = _encode(gs, qa, qb, na, nb, d, 8, cap)
    assert gs.gs_sync_status() == gs.GS_ERR_CAPACITY
    nw = n_words.cpu().numpy()
    assert nw[0] == ref[0].size and nw[1] == ref[1].size
    np.testing.assert_array_equal(words.cpu().numpy().view(np.uint16)[1, :ref[1].size], ref[1])
    # a flipped payload bit, a wrong length, a wrong d
    good = np.zeros((1, ref[0].size), np.uint16)
    good[0] = ref[0]
    for bad, n, dd in [(None, ref[0].size - 1, d), (None, ref[0].size, d + 1), (5, ref[0].size, d)]:
        w = good.copy()
        if bad is not None:
            w[0, 9 + 3 * ((int(np.count_nonzero(qs[0])) + 255) // 256) + bad] ^= 0x0100
        qt = torch.zeros((1, dd), dtype=torch.int8, device="cuda")
        gs.gs_dense_decode(_dev(w.view(np.int16)), _dev(np.array([n], np.int64)), dd, qt)
        rc = gs.gs_sync_status()
        assert rc == gs.GS_ERR_INVALID_ARG or not np.array_equal(qt.cpu().numpy()[0, :d], qs[0])


def test_dense_code_of_the_sparsifier_full_c3(gs):
    """The 16 x 2^24 Student-t workload: the GPU's hybrid code coded on the GPU
    equals, word for word, the oracle's code of q~ built from the oracle's own
    sparsification (workers 0, 7 and 15 compared; every worker round-trips)."""
    import torch
    w = workloads.C3
    g = workloads.device_student_t(w.M, w.d, seed0=w.data_seed)
    M, d = g.shape
    qa_i = torch.empty((M, d), dtype=torch.int32, device="cuda")
    qa_v = torch.empty((M, d), dtype=torch.float32, device="cuda")
    qb = torch.empty((M, d), dtype=torch.int32, device="cuda")
    na = torch.empty(M, dtype=torch.int32, device="cuda")
    nb = torch.empty(M, dtype=torch.int32, device="cuda")
    il = torch.empty(M, dtype=torch.float32, device="cuda")
    gs.gs_batched_sparsify_hybrid(g, w.kappa, w.iters, w.seed, w.step, 0, qa_i, qa_v, qb, na, nb, il)
    word_cap = d // 8
    words = torch.empty((M, word_cap), dtype=torch.int16, device="cuda")
    n_words = torch.zeros(M, dtype=torch.int64, device="cuda")
    gs.gs_dense_encode(qa_i, qb, na, nb, d, 9, words, n_words)
    assert gs.gs_sync_status() == gs.GS_OK
    qt = torch.empty((M, d), dtype=torch.int8, device="cuda")
    gs.gs_dense_decode(words, n_words, d, qt)
    assert gs.gs_sync_status() == gs.GS_OK
    # round trip against the GPU's own hybrid lists, every worker
    qt_h = qt.cpu().numpy()
    na_h, nb_h = na.cpu().numpy(), nb.cpu().numpy()
    for m in range(M):
        q = np.zeros(d, np.int8)
        q[qa_i[m, :na_h[m]].cpu().numpy()] = 2
        c = qb[m, :nb_h[m]].cpu().numpy().view(np.uint32)
        q[(c >> 1).astype(np.int64)] = np.where(c & 1, -1, 1)
        np.testing.assert_array_equal(qt_h[m], q)
    # word-for-word against the oracle's code of the oracle's own q~
    g_host = g.cpu().numpy()
    sel = [0, 7, 15]
    refs = oracle_rows(oracle.sparsify, [g_host[m] for m in sel], w.kappa, w.iters, w.seed, w.step, workers=sel)
    got = words.cpu().numpy().view(np.uint16)
    nw = n_words.cpu().numpy()
    for m, (ri, rv, info) in zip(sel, refs):
        # q~ from the oracle's Q(g): 2 where p = 1 (value g itself), else the sign
        a_i, _, b_c, _ = oracle.hybrid_encode(g_host[m], info["lambda"], ri, rv)
        q = np.zeros(d, np.int8)
        q[a_i] = 2
        q[(b_c >> 1).astype(np.int64)] = np.where(b_c & 1, -1, 1)
        ref = oracle.dense_encode(q, 9)
        assert nw[m] == ref.size
        np.testing.assert_array_equal(got[m, :ref.size], ref)
    del g
    torch.cuda.empty_cache()
