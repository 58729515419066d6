"""Pins for the CPU oracle against what the paper and mathematics fix.

Nothing here re-derives the oracle's numbers through the oracle's own
formulas: each check comes from a different route --
  * hand-derived worked examples of Algorithm 3 (tests/golden),
  * the sort-based closed form of the fixed point of Algorithm 3
    (Proposition 1 / Eq. 5: the capped set is the top-k by magnitude), in
    exact rational arithmetic on tiny inputs,
  * closed-form special cases (uniform sampling, one-hot, full budget,
    scale invariance, permutation equivariance),
  * the statistics the paper proves in section 3 / 3.1 (unbiasedness,
    second moment sum g^2/p, expected sparsity sum p),
  * a third-party Philox4x32-10 (Triton's, run by its CPU interpreter).
"""
import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "worked_examples.json")


def _cases():
    with open(GOLDEN) as f:
        return json.load(f)["cases"]


# ---------------------------------------------------------------------------
# Worked examples of Algorithm 3 (hand-derived)
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("case", _cases(), ids=lambda c: c["name"])
def test_worked_examples(oracle_mod, case):
    g = np.array(case["g"], dtype=np.float32)
    for iters_s, lam_s in case["lambda_by_iters"].items():
        iters = int(iters_s)
        info = oracle_mod.greedy_lambda(g, case["kappa"], iters)
        lam = float(Fraction(lam_s))
        assert info["lambda"] == pytest.approx(lam, rel=1e-14), (iters, info)
        assert info["capped"] == case["capped_by_iters"][iters_s]
        assert info["sum_p"] == pytest.approx(float(Fraction(case["sum_p_by_iters"][iters_s])), rel=1e-14)
    p, info = oracle_mod.probabilities(g, case["kappa"], 5)
    want = np.array([float(Fraction(x)) for x in case["p_final"]])
    np.testing.assert_allclose(p, want, rtol=1e-14, atol=0)
    # A rescale by c within rounding of 1 may follow the exact stop; nothing else may.
    info1 = oracle_mod.greedy_lambda(g, case["kappa"], case["iters_run_exact"])
    assert info1["lambda"] == pytest.approx(info["lambda"], rel=1e-14)
    assert info["iters_run"] >= case["iters_run_exact"]


# ---------------------------------------------------------------------------
# Brute force: the fixed point of Algorithm 3 from sorted magnitudes
# ---------------------------------------------------------------------------
def fixed_point_lambda(g, kappa):
    """Exact lambda* with sum_i min(lambda* |g_i|, 1) = kappa d, found from the
    top-k structure of Proposition 1 (Eq. 5); None when kappa d >= nnz(g), in
    which case every non-zero coordinate is capped."""
    a = sorted((abs(Fraction(float(x))) for x in g), reverse=True)
    d = len(a)
    budget = Fraction(float(kappa)) * d
    nnz = sum(1 for x in a if x != 0)
    if budget >= nnz:
        return None
    for k in range(0, d):
        rest = sum(a[k:], Fraction(0))
        if rest == 0:
            break
        lam = (budget - k) / rest
        if lam <= 0:
            break
        top_ok = (k == 0) or (lam * a[k - 1] >= 1)
        next_ok = lam * a[k] < 1
        if top_ok and next_ok:
            return lam
    raise AssertionError("no fixed point found")


def _tiny_inputs():
    rng = np.random.default_rng(1234)
    out = []
    for d in range(1, 13):
        for _ in range(12):
            kind = rng.integers(0, 4)
            if kind == 0:
                g = rng.standard_normal(d)
            elif kind == 1:
                g = rng.lognormal(0, 2.0, d) * np.sign(rng.standard_normal(d))
            elif kind == 2:
                g = rng.integers(-3, 4, d).astype(np.float64)
            else:
                g = rng.standard_cauchy(d)
            g = g.astype(np.float32)
            kappa = float(np.float64(rng.choice([0.05, 0.1, 0.2, 0.3, 0.5, 0.75, 0.9, 1.0])))
            out.append((g, kappa))
    return out


def test_bruteforce_fixed_point(oracle_mod):
    checked = 0
    for g, kappa in _tiny_inputs():
        d = g.size
        lam_star = fixed_point_lambda(g, kappa)
        info = oracle_mod.greedy_lambda(g, kappa, d + 5)
        p, _ = oracle_mod.probabilities(g, kappa, d + 5)
        if lam_star is None:
            # Budget covers every non-zero coordinate: all of them end capped.
            np.testing.assert_array_equal(p, (g != 0).astype(np.float64))
            continue
        assert info["lambda"] == pytest.approx(float(lam_star), rel=1e-12), (g, kappa)
        assert info["sum_p"] == pytest.approx(kappa * d, rel=1e-12)
        # Fewer iterations never overshoot the fixed point (lambda_j increases to lambda*).
        for it in range(0, 3):
            assert oracle_mod.greedy_lambda(g, kappa, it)["lambda"] <= float(lam_star) * (1 + 1e-12)
        checked += 1
    assert checked > 50


def test_bruteforce_exhaustive_grid(oracle_mod):
    vals = [0.0, 0.5, 1.0, 2.0, 3.0]
    import itertools
    n = 0
    for combo in itertools.product(vals, repeat=4):
        g = np.array(combo, dtype=np.float32)
        if not g.any():
            continue
        for kappa in (0.25, 0.5, 0.75):
            lam_star = fixed_point_lambda(g, kappa)
            p, info = oracle_mod.probabilities(g, kappa, 10)
            if lam_star is None:
                np.testing.assert_array_equal(p, (g != 0).astype(np.float64))
            else:
                want = np.array([float(min(lam_star * Fraction(float(x)), 1)) for x in g])
                np.testing.assert_allclose(p, want, rtol=1e-12, atol=0)
            n += 1
    assert n > 1000


# ---------------------------------------------------------------------------
# Algorithm 3 as printed (p-vector) == lambda form
# ---------------------------------------------------------------------------
def test_literal_pvector_matches_lambda_form(oracle_mod):
    rng = np.random.default_rng(7)
    for trial in range(60):
        d = int(rng.integers(1, 3000))
        g = (rng.standard_t(2.5, d) * (rng.random(d) > 0.05)).astype(np.float32)
        kappa = float(rng.choice([0.01, 0.05, 0.1, 0.3, 0.7]))
        iters = int(rng.integers(0, 6))
        p_lit, it_lit = oracle_mod.greedy_pvector(g, kappa, iters)
        p_lam, info = oracle_mod.probabilities(g, kappa, iters)
        # Iteration counts may differ by rescalings whose c is 1 up to rounding
        # (at the fixed point c = 1 exactly); the probabilities may not.
        np.testing.assert_allclose(p_lam, p_lit, rtol=1e-12, atol=1e-300)


# ---------------------------------------------------------------------------
# Invariants of Algorithm 3 and Proposition 1
# ---------------------------------------------------------------------------
def test_invariants(oracle_mod):
    rng = np.random.default_rng(11)
    for trial in range(40):
        d = int(rng.integers(2, 5000))
        g = (rng.lognormal(0, 2, d) * np.sign(rng.standard_normal(d))).astype(np.float32)
        g[rng.random(d) < 0.1] = 0
        kappa = float(rng.choice([0.001, 0.01, 0.1, 0.5]))
        lams, caps = [], []
        for it in range(0, 6):
            info = oracle_mod.greedy_lambda(g, kappa, it)
            # sum p^j <= kappa d at every iteration
            assert info["sum_p"] <= kappa * d * (1 + 1e-12)
            lams.append(info["lambda"])
            caps.append(info["capped"])
        # lambda_j non-decreasing and the capped sets nested (counts non-decreasing)
        assert all(b >= a for a, b in zip(lams, lams[1:]))
        assert all(b >= a for a, b in zip(caps, caps[1:]))
        p, _ = oracle_mod.probabilities(g, kappa, 3)
        a = np.abs(g.astype(np.float64))
        # p in [0, 1]; p = 0 exactly on zeros; monotone in |g|
        assert np.all((p >= 0) & (p <= 1))
        assert np.all((p == 0) == (a == 0))
        order = np.argsort(a, kind="stable")
        assert np.all(np.diff(p[order]) >= 0)


def test_scale_invariance_and_permutation(oracle_mod):
    rng = np.random.default_rng(5)
    d = 4097
    g = rng.standard_t(3, d).astype(np.float32)
    kappa, iters = 0.05, 3
    p, info = oracle_mod.probabilities(g, kappa, iters)
    # Power-of-two scaling is exact in floating point: identical p, Q scales.
    p2, info2 = oracle_mod.probabilities(g * np.float32(4.0), kappa, iters)
    np.testing.assert_array_equal(p, p2)
    i1, v1, _ = oracle_mod.sparsify(g, kappa, iters, 9, 3, 2)
    i2, v2, _ = oracle_mod.sparsify(g * np.float32(0.25), kappa, iters, 9, 3, 2)
    np.testing.assert_array_equal(i1, i2)
    np.testing.assert_array_equal(v1 * np.float32(0.25), v2)
    # Other positive scalings: p agrees to rounding.
    p3, _ = oracle_mod.probabilities((g * np.float32(3.7)).astype(np.float32), kappa, iters)
    np.testing.assert_allclose(p3, p, rtol=1e-6)
    # Permutation equivariance.
    perm = rng.permutation(d)
    pp, _ = oracle_mod.probabilities(g[perm], kappa, iters)
    np.testing.assert_allclose(pp, p[perm], rtol=1e-12)


def test_full_budget_caps_support(oracle_mod):
    g = np.array([0, 3, -1e-3, 0, 7, 1e-6, 0, 2], dtype=np.float32)
    p, info = oracle_mod.probabilities(g, 1.0, 20)
    np.testing.assert_array_equal(p, (g != 0).astype(np.float64))
    idx, val, _ = oracle_mod.sparsify(g, 1.0, 20, 1, 0, 0)
    np.testing.assert_array_equal(idx, np.nonzero(g)[0])
    np.testing.assert_array_equal(val, g[g != 0])


def test_zero_vector_and_errors(oracle_mod):
    z = np.zeros(17, dtype=np.float32)
    info = oracle_mod.greedy_lambda(z, 0.3, 2)
    assert info["lambda"] == 0 and info["sum_p"] == 0
    idx, val, _ = oracle_mod.sparsify(z, 0.3, 2, 1, 0, 0)
    assert idx.size == 0
    bad = np.array([1, np.nan, 2], dtype=np.float32)
    with pytest.raises(oracle_mod.OracleError) as e:
        oracle_mod.greedy_lambda(bad, 0.3, 2)
    assert e.value.code == 4
    inf = np.array([1, np.inf, 2], dtype=np.float32)
    with pytest.raises(oracle_mod.OracleError):
        oracle_mod.sparsify(inf, 0.3, 2, 1, 0, 0)
    for kappa in (0.0, -0.1, 1.5):
        with pytest.raises(oracle_mod.OracleError) as e:
            oracle_mod.greedy_lambda(np.ones(4, np.float32), kappa, 2)
        assert e.value.code == 1
    with pytest.raises(oracle_mod.OracleError):
        oracle_mod.greedy_lambda(np.ones(4, np.float32), 0.5, -1)


# ---------------------------------------------------------------------------
# Section 3 / 3.1 statistics of Q(g)
# ---------------------------------------------------------------------------
def test_unbiased_variance_sparsity(oracle_mod):
    g = np.array([5.0, -3.0, 2.0, 1.0, -1.0, 0.5, 0.5, -0.25, 0.125, 0.0, 4.0, -0.75], dtype=np.float32)
    d = g.size
    kappa, iters, seed, worker = 0.3, 2, 77, 5
    p, _ = oracle_mod.probabilities(g, kappa, iters)
    n = 100_000
    s1 = np.zeros(d)
    s2 = np.zeros(d)
    hits = np.zeros(d)
    nnz_tot = 0.0
    for step in range(n):
        idx, val, _ = oracle_mod.sparsify(g, kappa, iters, seed, step, worker)
        s1[idx] += val
        s2[idx] += val.astype(np.float64) ** 2
        hits[idx] += 1
        nnz_tot += idx.size
    gd = g.astype(np.float64)
    mean = s1 / n
    live = p > 0
    # E[Q_i] = g_i  (section 3): z-scores of the Monte-Carlo mean
    sigma = np.sqrt(gd[live] ** 2 * (1 / p[live] - 1) / n)
    exact = sigma == 0
    assert np.all(mean[live][exact] == gd[live][exact])
    z = np.abs(mean[live][~exact] - gd[live][~exact]) / sigma[~exact]
    assert z.max() < 5.0, z
    # P(Z_i = 1) = p_i: binomial z-scores
    zb = np.abs(hits[live] / n - p[live]) / np.sqrt(np.maximum(p[live] * (1 - p[live]), 1e-300) / n)
    zb[p[live] == 1] = 0
    assert zb.max() < 5.0
    assert np.all(hits[~live] == 0)
    # E sum Q_i^2 = sum g_i^2 / p_i  (section 3.1)
    m2 = s2.sum() / n
    want_m2 = float(np.sum(gd[live] ** 2 / p[live]))
    per_step_var = np.sum(gd[live] ** 4 / p[live] ** 3 * (1 - p[live]))
    assert abs(m2 - want_m2) < 5 * math.sqrt(per_step_var / n)
    # E ||Q||_0 = sum p_i  (section 3.1)
    assert abs(nnz_tot / n - p.sum()) < 5 * math.sqrt(np.sum(p * (1 - p)) / n)


def test_kept_set_is_u_below_p(oracle_mod):
    rng = np.random.default_rng(3)
    d = 20000
    g = rng.standard_t(3, d).astype(np.float32)
    kappa, iters, seed, step, worker = 0.02, 3, 12345678901, 7, 3
    p, info = oracle_mod.probabilities(g, kappa, iters)
    u = oracle_mod.uniforms(seed, step, worker, 0, d)
    idx, val, _ = oracle_mod.sparsify(g, kappa, iters, seed, step, worker)
    want = np.nonzero((u < p) & (p > 0))[0]
    np.testing.assert_array_equal(idx, want)
    # Amplification Q_i = g_i / p_i; uncapped coordinates carry sign(g_i)/lambda.
    np.testing.assert_allclose(val, (g[idx] / p[idx]).astype(np.float32), rtol=0)
    unc = p[idx] < 1
    np.testing.assert_allclose(np.abs(val[unc]), 1.0 / info["lambda"], rtol=1e-7)
    # nnz within 5 sigma of sum p
    assert abs(idx.size - p.sum()) < 5 * math.sqrt(np.sum(p * (1 - p)))


def test_segmented_is_per_layer(oracle_mod):
    rng = np.random.default_rng(9)
    off = np.array([0, 64, 64 + 1000, 64 + 1000 + 7, 64 + 1000 + 7 + 5000])
    g = rng.standard_normal(off[-1]).astype(np.float32)
    idx, val, lams = oracle_mod.segmented_sparsify(g, off, 0.05, 2, 4, 1, 6)
    pieces_i, pieces_v = [], []
    for l in range(off.size - 1):
        i, v, info = oracle_mod.sparsify(g[off[l]:off[l + 1]], 0.05, 2, 4, 1, 6, i0=off[l])
        assert info["lambda"] == lams[l]
        pieces_i.append(i)
        pieces_v.append(v)
    np.testing.assert_array_equal(idx, np.concatenate(pieces_i))
    np.testing.assert_array_equal(val, np.concatenate(pieces_v))
    assert np.all(np.diff(idx) > 0)


# ---------------------------------------------------------------------------
# Aggregate (Algorithm 1, step 6, as a sum in worker order)
# ---------------------------------------------------------------------------
def test_aggregate_matches_dense_fp32_sum(oracle_mod):
    rng = np.random.default_rng(21)
    d, M = 3001, 6
    idxs, vals = [], []
    dense = np.zeros(d, dtype=np.float32)
    for m in range(M):
        k = int(rng.integers(0, 800))
        idx = np.sort(rng.choice(d, size=k, replace=False)).astype(np.int32)
        val = (rng.standard_normal(k) * 10 ** rng.uniform(-3, 3, k)).astype(np.float32)
        idxs.append(idx)
        vals.append(val)
        q = np.zeros(d, dtype=np.float32)
        q[idx] = val
        dense = (dense + q).astype(np.float32)     # numpy fp32 add, worker order
    out = oracle_mod.aggregate(idxs, vals, d)
    np.testing.assert_array_equal(out, dense)


# ---------------------------------------------------------------------------
# Philox4x32-10 against a third-party implementation (Triton's tl.philox,
# run on the CPU by the Triton interpreter)
# ---------------------------------------------------------------------------
def _triton_philox(seeds, c):
    os.environ["TRITON_INTERPRET"] = "1"
    triton = pytest.importorskip("triton")
    import torch
    import triton.language as tl

    @triton.jit
    def _k(o0, o1, o2, o3, c0p, c1p, c2p, c3p, seed, N: tl.constexpr):
        offs = tl.arange(0, N)
        a, b, cc, dd = tl.philox(seed, tl.load(c0p + offs), tl.load(c1p + offs), tl.load(c2p + offs),
                                 tl.load(c3p + offs))
        tl.store(o0 + offs, a)
        tl.store(o1 + offs, b)
        tl.store(o2 + offs, cc)
        tl.store(o3 + offs, dd)

    outs = []
    for seed, ctr in zip(seeds, c):
        n = ctr.shape[1]
        N = 1 << max(0, (n - 1).bit_length())          # tl.arange wants a power of two
        pad = np.zeros((4, N), dtype=np.uint32)
        pad[:, :n] = ctr
        cin = [torch.from_numpy(np.ascontiguousarray(pad[j]).view(np.int32)) for j in range(4)]
        o = [torch.zeros(N, dtype=torch.int32) for _ in range(4)]
        _k[(1,)](*o, *cin, seed, N=N)
        outs.append(np.stack([x.numpy().view(np.uint32)[:n] for x in o]))
    return outs


def test_philox_matches_third_party(oracle_mod):
    rng = np.random.default_rng(99)
    seeds = [1, 12345, 0x9E3779B97F4A7C15 & 0x7FFFFFFFFFFFFFFF, 2**40 + 17]
    ctrs = [rng.integers(0, 2**32, size=(4, 16), dtype=np.uint64).astype(np.uint32) for _ in seeds]
    ref = _triton_philox(seeds, ctrs)
    for seed, ctr, r in zip(seeds, ctrs, ref):
        key = (seed & 0xFFFFFFFF, seed >> 32)
        for j in range(ctr.shape[1]):
            got = oracle_mod.philox4x32_10(ctr[:, j], key)
            assert got == list(r[:, j]), (seed, j)


def test_word_mapping_matches_third_party(oracle_mod):
    # Word for coordinate i of (worker, step): counter (q lo, q hi, worker, step), q = i // 4, word i % 4.
    seed, step, worker = 2**33 + 5, 11, 6
    ii = np.array([0, 1, 2, 3, 4, 5, 1023, 2**24 - 1, 2**27 + 2, 2**34 + 3], dtype=np.int64)
    q = ii // 4
    ctr = np.stack([q & 0xFFFFFFFF, q >> 32, np.full_like(q, worker), np.full_like(q, step)]).astype(np.uint32)
    (ref,) = _triton_philox([seed], [ctr])
    for j, i in enumerate(ii):
        assert oracle_mod.word(seed, step, worker, int(i)) == ref[i % 4, j]


def test_uniforms_are_uniform(oracle_mod):
    u = oracle_mod.uniforms(1, 0, 0, 0, 200_000)
    assert u.min() >= 0 and u.max() < 1
    hist, _ = np.histogram(u, bins=100, range=(0, 1))
    e = u.size / 100
    chi2 = float(((hist - e) ** 2 / e).sum())
    # 99 dof: mean 99, sd 14; 200 is > 7 sd out.
    assert chi2 < 200
    assert abs(u.mean() - 0.5) < 5 * math.sqrt(1 / 12 / u.size)
