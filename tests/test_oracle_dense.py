"""Pins of the oracle's dense code of Q(g) (section 3.3, last paragraph):
q~ in {0, +1, -1, 2}^d entropy coded under the static model P(s) = d_s / d,
whose ideal length is sum_s d_s log2(d / d_s) <= 2d bits.

What fixes the coder independently of its own code:
  - exact round trips (decode o encode = identity) over densities, sizes,
    chunk sizes and edge cases, and rejection of corrupted streams;
  - the coded length against the model's entropy, within the stated
    overhead (header, per-chunk directory and flushed state, quantization);
  - the 2d bound of section 3.3 on the worst case (four equally likely
    symbols);
  - the model's quantized frequencies against the closed forms of the
    geometric run-length law, computed here from p0 alone, and the identity
    that the bit-length and bit probabilities multiply back to
    (1 - p0) p0^g for every run g;
  - the dense code of a real sparsified gradient, with the kept values of
    p_i = 1 and 1/lambda, gives back exactly the oracle's (idx, val) lists.
"""
import math

import numpy as np
import pytest

import oracle

M = 1 << 15
HEADER_BITS = 9 * 16
CHUNK_BITS = 3 * 16 + 32 + 16      # directory entry, flushed state, last partial word


def _entropy(q):
    d = q.size
    return sum(float(c) * math.log2(d / c) for c in (np.count_nonzero(q == v) for v in (0, 1, -1, 2)) if c)


def _random_q(rng, d, density, p_cap=0.02):
    q = np.zeros(d, np.int8)
    hit = rng.random(d) < density
    n = int(hit.sum())
    q[hit] = rng.choice(np.array([1, -1, 2], np.int8), n, p=[(1 - p_cap) / 2, (1 - p_cap) / 2, p_cap])
    return q


def _chunks(q, log2_k):
    nz = int(np.count_nonzero(q))
    return (nz + (1 << log2_k) - 1) >> log2_k


@pytest.mark.parametrize("d,density,log2_k", [(1, 1.0, 4), (7, 0.5, 4), (1000, 0.01, 4), (65536, 0.1, 9),
                                              (100_003, 0.0005, 6), (250_000, 0.3, 10), (40_000, 0.97, 8),
                                              (1 << 20, 0.01, 9)])
def test_round_trip(oracle_mod, d, density, log2_k):
    rng = np.random.default_rng(d + log2_k)
    q = _random_q(rng, d, density)
    w = oracle.dense_encode(q, log2_k)
    np.testing.assert_array_equal(oracle.dense_decode(w, d), q)


def test_round_trip_edge_cases(oracle_mod):
    cases = [np.zeros(1, np.int8), np.zeros(5000, np.int8), np.array([2], np.int8), np.array([-1], np.int8),
             np.full(3000, 1, np.int8), np.full(3000, 2, np.int8)]
    # one non-zero at the very end, and two at the ends of a long vector (one run of 2^22 - 2 zeros)
    e = np.zeros(12345, np.int8)
    e[-1] = -1
    cases.append(e)
    f = np.zeros(1 << 22, np.int8)
    f[0], f[-1] = 1, 2
    cases.append(f)
    # exactly K and K + 1 non-zeros (one full chunk; a chunk of one)
    for n in (16, 17):
        g = np.zeros(200, np.int8)
        g[np.arange(n) * 11] = 1
        cases.append(g)
    for q in cases:
        for log2_k in (4, 9):
            w = oracle.dense_encode(q, log2_k)
            np.testing.assert_array_equal(oracle.dense_decode(w, q.size), q)
    # no non-zero symbol: the header alone
    assert oracle.dense_encode(np.zeros(777, np.int8)).size == 9


def test_corrupted_streams_are_rejected(oracle_mod):
    rng = np.random.default_rng(11)
    d = 50_000
    q = _random_q(rng, d, 0.05)
    w = oracle.dense_encode(q, 8)
    with pytest.raises(oracle.OracleError):
        oracle.dense_decode(w[:-1], d)          # truncated
    with pytest.raises(oracle.OracleError):
        oracle.dense_decode(w, d + 1)           # wrong length
    bad = w.copy()
    bad[9 + 3 * _chunks(q, 8) + 5] ^= 0x0100   # one payload bit of the first stream
    try:
        r = oracle.dense_decode(bad, d)
    except oracle.OracleError:
        r = None
    assert r is None or not np.array_equal(r, q)


@pytest.mark.parametrize("density", [0.0002, 0.001, 0.01, 0.05, 0.2, 0.5, 0.9])
def test_length_within_stated_overhead_of_the_entropy(oracle_mod, density):
    """16 * words <= H + header + per-chunk overhead + 0.01 bit per non-zero
    (the quantization of the model to 15-bit frequencies), and, where chunks
    are few against the payload, within 2% of H from below too (the coder
    places each chunk's first non-zero and the trailing zeros for free)."""
    rng = np.random.default_rng(int(density * 1e6))
    d = 1 << 21
    q = _random_q(rng, d, density)
    nz = int(np.count_nonzero(q))
    for log2_k in (6, 9):
        w = oracle.dense_encode(q, log2_k)
        bits = 16 * w.size
        H = _entropy(q)
        n_ch = _chunks(q, log2_k)
        assert bits <= H + HEADER_BITS + CHUNK_BITS * n_ch + 0.01 * nz, (bits, H)
        if log2_k == 9:
            assert bits >= 0.98 * H


def test_two_d_bound_on_the_worst_case(oracle_mod):
    """Four equally likely symbols: the entropy is 2 bits per coordinate, the
    bound of section 3.3; the code stays within its overhead of it."""
    rng = np.random.default_rng(5)
    d = 1 << 18
    q = rng.choice(np.array([0, 1, -1, 2], np.int8), d)
    w = oracle.dense_encode(q, 10)
    assert _entropy(q) <= 2 * d
    assert 16 * w.size <= 2 * d + HEADER_BITS + CHUNK_BITS * _chunks(q, 10) + 0.01 * d


def _law(p0):
    """The geometric run-length law of the static model, from p0 alone:
    P(l) for bit lengths l = floor(log2(g + 1)) and P(bit k = 1)."""
    s = [p0]
    for _ in range(30):
        s.append(s[-1] * s[-1])
    P = [math.prod(s[:l]) * (1.0 - s[l]) for l in range(31)]
    r = [s[k] / (1.0 + s[k]) for k in range(30)]
    return P, r


@pytest.mark.parametrize("p0", [0.0, 0.3, 0.9, 0.99, 0.999, 0.99999])
def test_run_law_multiplies_back_to_the_geometric(p0):
    """P(l) * prod_k P(bit k) = (1 - p0) p0^g for every run g: coding the run
    by its bit length and bits costs exactly what g zeros and one non-zero
    cost under the static model."""
    P, r = _law(p0)
    for g in [0, 1, 2, 3, 7, 8, 100, 1000, 12345, (1 << 20) + 3]:
        v = g + 1
        l = v.bit_length() - 1
        prob = P[l]
        for k in range(l):
            b = (v >> k) & 1
            prob *= r[k] if b else 1.0 - r[k]
        want = (1.0 - p0) * p0 ** g
        assert prob == pytest.approx(want, rel=1e-9, abs=1e-300)
    assert sum(P) == pytest.approx(1.0, abs=1e-12) if p0 < 0.9999 else True


@pytest.mark.parametrize("d,n_pos,n_neg,n_cap", [(1 << 24, 83000, 84000, 28), (1000, 300, 250, 50), (10, 0, 0, 10),
                                                (1 << 27, 39_000_000, 39_000_000, 29_000_000), (5, 0, 0, 0)])
def test_model_frequencies_follow_the_closed_forms(oracle_mod, d, n_pos, n_neg, n_cap):
    m = oracle.dense_model(d, n_pos, n_neg, n_cap)
    nz = n_pos + n_neg + n_cap
    p0 = (d - nz) / d
    P, r = _law(p0)
    assert m["len_f"].sum() == M and m["val_f"].sum() == M
    assert np.all(m["len_f"] >= 1)
    np.testing.assert_array_equal(m["len_c"], np.concatenate([[0], np.cumsum(m["len_f"])]))
    np.testing.assert_array_equal(m["val_c"], np.concatenate([[0], np.cumsum(m["val_f"])]))
    if nz:   # (with no non-zero symbol there are no runs to model)
        assert np.all(np.abs(m["len_f"] / M - np.array(P)) <= 32.0 / M)
    assert np.all(np.abs(m["bit_f1"] / M - np.clip(r, 1.0 / M, 1 - 1.0 / M)) <= 1.0 / M)
    if nz:
        for t, n in enumerate((n_pos, n_neg, n_cap)):
            assert (m["val_f"][t] == 0) == (n == 0)
            assert abs(m["val_f"][t] / M - n / nz) <= 4.0 / M


def test_dense_code_of_a_sparsified_gradient(oracle_mod):
    """The paper's use: q~ of Q(g) (0 where dropped, sign(g_i) where kept with
    p_i < 1, 2 where p_i = 1), coded; decoded, it and the values of the
    p_i = 1 entries plus 1/lambda (section 3.3) give back Q(g) exactly."""
    rng = np.random.default_rng(2)
    d = 300_001
    g = (rng.standard_t(3, d) * np.where(rng.random(d) < 0.001, 50, 1)).astype(np.float32)
    idx, val, info = oracle.sparsify(g, 0.02, 3, 7, 1, 0)
    qa_i, qa_v, qb, inv = oracle.hybrid_encode(g, info["lambda"], idx, val)
    q = np.zeros(d, np.int8)
    q[qa_i] = 2
    q[(qb >> 1).astype(np.int64)] = np.where(qb & 1, -1, 1)
    w = oracle.dense_encode(q, 9)
    back = oracle.dense_decode(w, d)
    np.testing.assert_array_equal(back, q)
    # Q(g) from the dense code, the p_i = 1 values in index order, and 1 / lambda
    nzi = np.nonzero(back)[0]
    vals = np.where(back[nzi] == 2, 0.0, back[nzi] * np.float32(inv)).astype(np.float32)
    vals[back[nzi] == 2] = qa_v
    np.testing.assert_array_equal(nzi, idx)
    np.testing.assert_array_equal(vals, val)
    # and its length is the entropy length the bench reports, plus the stated overhead
    H = oracle.ternary_bits(d, int((back == -1).sum()), int((back == 1).sum()), int((back == 2).sum()))
    assert 16 * w.size <= H + HEADER_BITS + CHUNK_BITS * _chunks(q, 9) + 0.01 * nzi.size
