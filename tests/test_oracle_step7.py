"""Pins for the oracle's Algorithm 1 steps 6-7: the average
v = (1/M) sum_m Q(g^m) and its re-sparsification Q(v).  CPU only."""
import numpy as np
import pytest

import oracle


def _workers(M, d, seed):
    rng = np.random.default_rng(seed)
    return (rng.standard_t(3, (M, d)) * rng.uniform(0.5, 2.0, (M, 1))).astype(np.float32)


def test_average_of_identical_workers_is_the_worker():
    # Two identical sparse vectors: (v + v) / 2 = v exactly in fp32.
    g = _workers(1, 3000, 1)[0]
    i, v, _ = oracle.sparsify(g, 0.05, 2, 3, 0, 0)
    avg = oracle.average([i, i], [v, v], g.size)
    dense = np.zeros(g.size, np.float32)
    dense[i] = v
    np.testing.assert_array_equal(avg, dense)
    # One worker: the average is the vector itself.
    np.testing.assert_array_equal(oracle.average([i], [v], g.size), dense)


def test_average_is_within_rounding_of_the_exact_mean():
    M, d = 5, 4000
    G = _workers(M, d, 2)
    il, vl = [], []
    exact = np.zeros(d)
    for m in range(M):
        i, v, _ = oracle.sparsify(G[m], 0.1, 2, 7, 1, m)
        il.append(i)
        vl.append(v)
        np.add.at(exact, i.astype(np.int64), v.astype(np.float64))
    exact /= M
    avg = oracle.average(il, vl, d).astype(np.float64)
    mag = np.zeros(d)
    for i, v in zip(il, vl):
        np.add.at(mag, i.astype(np.int64), np.abs(v.astype(np.float64)))
    # M - 1 fp32 additions and one division: a few ulps of the summed magnitudes
    assert np.all(np.abs(avg - exact) <= 2.0 ** -21 * (mag / M) + 1e-45)


def test_two_stage_estimator_is_unbiased():
    # Algorithm 1 with step 7: E[Q(v_t)] = (1/M) sum_m g^m when each stage's
    # draws are independent (the second stage uses its own worker id).
    M, d, n = 3, 24, 6000
    G = _workers(M, d, 3)
    target = G.astype(np.float64).mean(axis=0)
    acc = np.zeros(d)
    acc2 = np.zeros(d)
    for t in range(n):
        il, vl = [], []
        for m in range(M):
            i, v, _ = oracle.sparsify(G[m], 0.3, 2, 11, t, m)
            il.append(i)
            vl.append(v)
        v = oracle.average(il, vl, d)
        i2, v2, _ = oracle.sparsify(v, 0.3, 2, 11, t, M)
        q = np.zeros(d)
        q[i2] = v2
        acc += q
        acc2 += q * q
    mean = acc / n
    sd = np.sqrt(np.maximum(acc2 / n - mean ** 2, 0.0) / n)
    assert np.all(np.abs(mean - target) <= 5 * sd + 1e-6)
    # and the second stage only keeps coordinates the average holds
    assert set(i2.tolist()) <= set(np.nonzero(v)[0].tolist())
