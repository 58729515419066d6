"""Pins for the oracle's hybrid coding of Q(g) (section 3.3, eqs. 9-10), the
entropy length of the dense {0, -1, +1, 2} code (section 3.3) and the
per-step communication cost H(T, M) of section 5.  CPU only."""
import math

import numpy as np
import pytest

import oracle


def test_worked_example_split():
    # Section 3.2 worked example (g = (100, 1 x 9), kappa = 0.3): lambda ends at
    # 2/9, coordinate 0 is capped (lambda * 100 >= 1), the others have
    # p = 2/9 and keep the value sign(g_i) * 9/2.  For the kept set {0, 3, 7}
    # with g_3 < 0, eqs. (9)-(10) give Q_A = [(0, 100)], Q_B = [(3, -), (7, +)],
    # 1 / lambda = 4.5.
    g = np.array([100.0] + [1.0] * 9, np.float32)
    g[3] = -1.0
    qa_i, qa_v, qb, inv = oracle.hybrid_encode(g, 2.0 / 9.0, [0, 3, 7], [100.0, -4.5, 4.5])
    np.testing.assert_array_equal(qa_i, [0])
    np.testing.assert_array_equal(qa_v, [100.0])
    np.testing.assert_array_equal(qb, [3 * 2 + 1, 7 * 2 + 0])
    assert inv == pytest.approx(4.5, rel=1e-15)
    i, v = oracle.hybrid_decode(qa_i, qa_v, qb, inv)
    np.testing.assert_array_equal(i, [0, 3, 7])
    np.testing.assert_array_equal(v, [100.0, -4.5, 4.5])


def test_boundary_lambda_g_equal_one_is_capped():
    # p_i = min(lambda |g_i|, 1) = 1 exactly when lambda |g_i| = 1: such a
    # coordinate is in S_k and travels in Q_A with its own value.
    g = np.array([2.0, -2.0, 1.0], np.float32)
    qa_i, qa_v, qb, inv = oracle.hybrid_encode(g, 0.5, [0, 1, 2], [2.0, -2.0, 2.0])
    np.testing.assert_array_equal(qa_i, [0, 1])
    np.testing.assert_array_equal(qa_v, [2.0, -2.0])
    np.testing.assert_array_equal(qb, [2 * 2])
    assert inv == 2.0


@pytest.mark.parametrize("kind,kappa,iters", [("t3", 0.05, 3), ("lognormal", 0.2, 2), ("normal", 0.5, 0)])
def test_round_trip_and_capped_count(kind, kappa, iters):
    rng = np.random.default_rng(17)
    d = 20000
    g = {"t3": rng.standard_t(3, d), "lognormal": rng.lognormal(0, 2, d) * rng.choice([-1, 1], d),
         "normal": rng.standard_normal(d)}[kind].astype(np.float32)
    idx, val, info = oracle.sparsify(g, kappa, iters, 9, 2, 1)
    qa_i, qa_v, qb, inv = oracle.hybrid_encode(g, info["lambda"], idx, val)
    # every capped coordinate (p = 1) is kept, so Q_A holds exactly them
    assert qa_i.size == info["capped"]
    assert qa_i.size + qb.size == idx.size
    assert np.all(np.diff(qa_i) > 0) and np.all(np.diff(qb >> 1) > 0)
    # Q_B signs are the signs of g
    np.testing.assert_array_equal(qb & 1, (g[(qb >> 1).astype(np.int64)] < 0).astype(np.uint32))
    i, v = oracle.hybrid_decode(qa_i, qa_v, qb, inv)
    np.testing.assert_array_equal(i, idx)
    # capped values are carried exactly; the others become +-fl32(1/lambda),
    # within one rounding of fl32(g / (lambda |g|))
    np.testing.assert_allclose(v, val, rtol=2.0 ** -22, atol=0)


def test_ternary_bits_bound_and_closed_forms():
    assert oracle.ternary_bits(1000, 0, 0, 0) == 0.0
    assert oracle.ternary_bits(1000, 0, 0, 1000) == 0.0
    # four equally frequent symbols: exactly 2 bits each, the 2d bound
    assert oracle.ternary_bits(4000, 1000, 1000, 1000) == pytest.approx(8000.0, rel=1e-12)
    # two equally frequent symbols: one bit each
    assert oracle.ternary_bits(1000, 0, 500, 0) == pytest.approx(1000.0, rel=1e-12)
    # a binary entropy: d * H(q) with q = 1/8
    q = 1.0 / 8.0
    h = -(q * math.log2(q) + (1 - q) * math.log2(1 - q))
    assert oracle.ternary_bits(8000, 0, 1000, 0) == pytest.approx(8000 * h, rel=1e-12)
    rng = np.random.default_rng(3)
    for _ in range(200):
        d = int(rng.integers(1, 10 ** 6))
        c = rng.multinomial(d, rng.dirichlet(np.ones(4)))
        bits = oracle.ternary_bits(d, c[1], c[2], c[3])
        assert 0.0 <= bits <= 2.0 * d * (1 + 1e-12)
    assert oracle.ternary_bits(10, 6, 6, 0) < 0   # counts that exceed d are refused


def test_comm_bits_formula():
    # 3 capped entries at (32 + 10) bits, 10 * 10.5 bits of indices, one float
    assert oracle.comm_bits(1024, 3, 10.5, 32) == pytest.approx(3 * 42 + 105 + 32)
    # the index term is clamped at 2d
    assert oracle.comm_bits(16, 0, 100.0, 32) == pytest.approx(32 + 32)
    assert oracle.comm_bits(16, 2, 0.0, 16) == pytest.approx(2 * 20 + 16)
