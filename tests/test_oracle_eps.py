"""Pins for the oracle's Algorithm 2 (section 3.2): the closed-form solution
of the variance-budget problem (4).  Each test checks it against something
the paper or the mathematics fixes independently of (6)-(7): the problem's
own constraint and objective, a generic solver, a bisection on Proposition
1's form, symmetry, Lemma 3's bound and Algorithm 3's fixed point.  CPU only."""
import numpy as np
import pytest

import oracle


def _g(kind, d, seed):
    rng = np.random.default_rng(seed)
    x = {"t3": lambda: rng.standard_t(3, d), "lognormal": lambda: rng.lognormal(0, 2, d) * rng.choice([-1, 1], d),
         "normal": lambda: rng.standard_normal(d)}[kind]()
    return x.astype(np.float32)


def _variance_ratio(g, p):
    g = g.astype(np.float64)
    nz = g != 0
    return float(np.sum(g[nz] ** 2 / p[nz]) / np.sum(g ** 2))


def test_two_level_vector_by_hand():
    # g = (100, 1 x 9): sum g^2 = 10009.  For eps = 0.05 the variance budget
    # eps * 10009 = 500.45 cannot absorb sampling the large entry
    # (its term 100 * 109 = 10900 exceeds 500.45 + 10009), so k = 1: the
    # large entry is kept and lambda = 9 / (500.45 + 9).  For eps = 0.5 the
    # budget 5004.5 does (10900 <= 15013.5): k = 0, lambda = 109 / 15013.5.
    g = np.array([100.0] + [1.0] * 9, np.float32)
    i = oracle.closed_form_lambda(g, 0.05)
    assert i["capped"] == 1
    assert i["lambda"] == pytest.approx(9.0 / 509.45, rel=1e-13)
    i = oracle.closed_form_lambda(g, 0.5)
    assert i["capped"] == 0
    assert i["lambda"] == pytest.approx(109.0 / 15013.5, rel=1e-13)


@pytest.mark.parametrize("eps", [0.01, 0.3, 4.0])
def test_equal_magnitudes_give_uniform_p(eps):
    # Problem (4) is symmetric when every |g_i| = c: the optimum is uniform,
    # and the active constraint d c^2 / p = (1 + eps) d c^2 gives p = 1 / (1 + eps).
    rng = np.random.default_rng(5)
    g = (0.75 * rng.choice([-1.0, 1.0], 1000)).astype(np.float32)
    p, info = oracle.probabilities_eps(g, eps)
    np.testing.assert_allclose(p, 1.0 / (1.0 + eps), rtol=1e-13)
    assert info["capped"] == 0


@pytest.mark.parametrize("kind", ["t3", "lognormal", "normal"])
@pytest.mark.parametrize("eps", [0.0, 0.02, 0.5, 10.0])
def test_constraint_tight_and_p_valid(kind, eps):
    g = _g(kind, 5000, 11)
    g[::97] = 0.0
    p, info = oracle.probabilities_eps(g, eps)
    nz = g != 0
    assert np.all(p[~nz] == 0)
    assert np.all(p[nz] > 0) and np.all(p <= 1.0)
    # the variance budget of (4) is used exactly (lambda > 0 makes it active)
    assert _variance_ratio(g, p) == pytest.approx(1.0 + eps, rel=1e-11)
    # Proposition 1: p is min(lambda |g|, 1), with the k largest capped
    a = np.abs(g.astype(np.float64))
    np.testing.assert_allclose(p, np.minimum(info["lambda"] * a, 1.0), rtol=1e-14)
    assert int(np.sum(p == 1.0)) >= info["capped"]
    assert info["sum_p"] == pytest.approx(float(p.sum()), rel=1e-12)


@pytest.mark.parametrize("kind", ["t3", "lognormal", "normal"])
@pytest.mark.parametrize("eps", [0.05, 1.0])
def test_bisection_on_the_active_constraint(kind, eps):
    # An independent solve of (4) in Proposition 1's form: V(lambda) =
    # sum g^2 / min(lambda |g|, 1) falls as lambda grows, so bisect lambda to
    # V = (1 + eps) sum g^2.
    g = _g(kind, 3000, 23).astype(np.float64)
    a = np.abs(g)
    a = a[a > 0]
    target = (1.0 + eps) * np.sum(a * a)
    lo, hi = 0.0, 1.0
    while np.sum(a * a / np.minimum(hi * a, 1.0)) > target:
        hi *= 2.0
    for _ in range(200):
        mid = 0.5 * (lo + hi)
        if mid <= lo or mid >= hi:
            break
        if np.sum(a * a / np.minimum(mid * a, 1.0)) > target:
            lo = mid
        else:
            hi = mid
    info = oracle.closed_form_lambda(g.astype(np.float32), eps)
    assert info["lambda"] == pytest.approx(hi, rel=1e-10)


@pytest.mark.parametrize("seed", [1, 2, 3])
def test_optimal_against_a_generic_solver(seed):
    optimize = pytest.importorskip("scipy.optimize")
    rng = np.random.default_rng(seed)
    g = (rng.standard_t(2, 6) * 3).astype(np.float32).astype(np.float64)
    eps = 0.2
    S = float(np.sum(g * g))
    cons = [{"type": "ineq", "fun": lambda p: (1 + eps) * S - np.sum(g * g / p)}]
    best = None
    for start in (np.full(6, 0.999), np.full(6, 0.9), rng.uniform(0.7, 1.0, 6)):
        r = optimize.minimize(lambda p: np.sum(p), start, method="SLSQP", bounds=[(1e-6, 1.0)] * 6,
                              constraints=cons, options={"ftol": 1e-14, "maxiter": 1000})
        if r.success and np.sum(g * g / r.x) <= (1 + eps) * S * (1 + 1e-9):
            best = r.fun if best is None else min(best, r.fun)
    assert best is not None
    p, info = oracle.probabilities_eps(g.astype(np.float32), eps)
    assert float(p.sum()) == pytest.approx(best, rel=1e-6)
    # and no random feasible point does better
    for _ in range(2000):
        q = rng.uniform(0.01, 1.0, 6)
        if np.sum(g * g / q) <= (1 + eps) * S:
            assert q.sum() >= p.sum() - 1e-12


@pytest.mark.parametrize("kind", ["t3", "lognormal"])
def test_lemma3_sparsity_bound(kind):
    # Lemma 3: if ||g_{S^c}||_1 <= rho ||g_S||_1 for some |S| = s, then with
    # eps = rho the expected sparsity sum p is at most (1 + rho) s.
    g = _g(kind, 4000, 31)
    a = np.sort(np.abs(g.astype(np.float64)))[::-1]
    for s in (1, 10, 100, 1000, 3000):
        rho = float(a[s:].sum() / a[:s].sum())
        info = oracle.closed_form_lambda(g, rho)
        assert info["sum_p"] <= (1.0 + rho) * s * (1 + 1e-12)


@pytest.mark.parametrize("kind", ["t3", "normal"])
def test_same_lambda_as_algorithm3_fixed_point(kind):
    # Both algorithms produce p = min(lambda |g|, 1); with the density budget
    # kappa d set to Algorithm 2's sum p, Algorithm 3 run to its fixed point
    # must land on the same lambda.
    g = _g(kind, 6000, 41)
    info = oracle.closed_form_lambda(g, 0.3)
    kappa = info["sum_p"] / g.size
    greedy = oracle.greedy_lambda(g, kappa, 10000)
    assert greedy["lambda"] == pytest.approx(info["lambda"], rel=1e-10)
    assert greedy["capped"] == info["capped"]


def test_degenerate_inputs():
    # eps = 0 leaves no room for extra variance: every non-zero entry is kept
    g = _g("t3", 500, 3)
    g[7] = 0.0
    p, info = oracle.probabilities_eps(g, 0.0)
    assert np.all(p[g != 0] == 1.0) and p[7] == 0.0
    # a single non-zero entry: the active constraint g^2 / p = (1 + eps) g^2
    h = np.zeros(50, np.float32)
    h[9] = -2.5
    p, info = oracle.probabilities_eps(h, 3.0)
    assert p[9] == pytest.approx(0.25, rel=1e-15) and np.count_nonzero(p) == 1
    # g = 0: nothing to keep
    info = oracle.closed_form_lambda(np.zeros(10, np.float32), 1.0)
    assert info["lambda"] == 0.0 and info["capped"] == 0
    with pytest.raises(oracle.OracleError):
        oracle.closed_form_lambda(g, -0.1)
    bad = g.copy()
    bad[3] = np.inf
    with pytest.raises(oracle.OracleError):
        oracle.closed_form_lambda(bad, 0.1)


def test_sparsify_eps_draws_and_values():
    g = _g("t3", 20000, 51)
    idx, val, info = oracle.sparsify_eps(g, 0.5, 9, 4, 2)
    p, _ = oracle.probabilities_eps(g, 0.5)
    u = oracle.uniforms(9, 4, 2, 0, g.size)
    keep = np.nonzero(u < p)[0]
    np.testing.assert_array_equal(idx, keep)
    np.testing.assert_allclose(val, (g[keep].astype(np.float64) / p[keep]).astype(np.float32), rtol=0)
    # unbiased: the mean of Q(g) over many draws approaches g
    h = _g("t3", 64, 52)
    acc = np.zeros(64)
    n = 4000
    for step in range(n):
        i, v, _ = oracle.sparsify_eps(h, 0.5, 1, step, 0)
        acc[i] += v
    p_h, _ = oracle.probabilities_eps(h, 0.5)
    sd = np.abs(h) * np.sqrt((1 - p_h) / np.maximum(p_h, 1e-300)) / np.sqrt(n)
    assert np.all(np.abs(acc / n - h) <= 6 * sd + 1e-6)
