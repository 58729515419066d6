"""Section 5's observation on Algorithm 3, checked on every input family.

The paper reports that the greedy rescaling of Algorithm 3 is good enough
after two iterations (j = 2, p <- p^j): the next update p^{j+1} - p^j is
more than an order of magnitude below p^j.  The paper fixes no norm; here it
is the l1 ratio r_j = ||p^{j+1} - p^j||_1 / ||p^j||_1, computed by the
oracle (p^j = its probabilities after j rescalings) on reduced-size copies of
the workloads' inputs.  For the uncapped coordinates p^{j+1} / p^j is the
rescaling factor c_j, so r_j is roughly (c_j - 1) times their share of the
mass.
"""
import numpy as np
import pytest

import oracle
import workloads as W


def _ratios(g, kappa, J=4):
    ps = [oracle.probabilities(g, kappa, j)[0] for j in range(J + 1)]
    return [float(np.abs(ps[j + 1] - ps[j]).sum() / ps[j].sum()) for j in range(J)]


CASES = [
    ("c1 log-normal(1.5)", lambda: W.gen_c1(65536), 0.1),
    ("c2 logistic-regression gradient", lambda: W.gen_logreg(1, 1 << 16)[0], 0.05),
    ("c3 Student-t(3)", lambda: W.gen_student_t(1, 1 << 20)[0], 0.01),
    ("c5 log-normal(2) + outliers", lambda: W.gen_c5(1, 1 << 18)[0], 0.001),
    ("c5 log-normal(2) + outliers", lambda: W.gen_c5(1, 1 << 18)[0], 0.01),
    ("c5 log-normal(2) + outliers", lambda: W.gen_c5(1, 1 << 18)[0], 0.1),
]


@pytest.mark.parametrize("name,make,kappa", CASES, ids=[f"{c[0]} k={c[2]}" for c in CASES])
def test_two_rescalings_suffice(name, make, kappa):
    g = np.asarray(make(), dtype=np.float32)
    r = _ratios(g, kappa)
    print(name, kappa, ["%.2e" % x for x in r])
    # After j = 2 the update is more than one order of magnitude below p^j.
    assert r[2] < 0.1
    # And the updates keep shrinking from there.
    assert r[3] <= r[2] + 1e-12


def test_two_rescalings_suffice_per_layer():
    """c4: every ResNet-50-shaped layer with its own budget (section 5.2)."""
    g, off = W.gen_layerwise(1)
    g = g[0]
    worst = 0.0
    for l in range(len(off) - 1):
        r = _ratios(g[off[l]:off[l + 1]], 0.02, J=3)
        worst = max(worst, r[2])
    assert worst < 0.1
