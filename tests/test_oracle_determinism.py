"""Pins of the oracle's target-block early determinism (App. B).

D_b is checked against its definition by exhaustive enumeration of the
target block (the expectation itself, and the collision sums over V^j that
the product form factorises), against closed forms (one-hot and uniform rows, b = 1), and the
M-sample estimator against D_b (unbiasedness, 4 sigma) and against the
target law of its own draws (chi-square).  CPU only.
"""
import itertools
import math

import numpy as np
import pytest
import scipy.special

from oracle import dblast_oracle as orc


def _rows(b, V, seed, scale=1.5):
    rng = np.random.default_rng(seed)
    return scipy.special.softmax(rng.normal(0, scale, size=(b, V)), axis=-1)


@pytest.mark.parametrize("b,V", [(1, 5), (3, 3), (4, 2)])
def test_exact_form_equals_definition_by_enumeration(b, V):
    """D_b = sum_x prod_i p_i(x_i) (1/b) sum_j prod_{i<=j} p_i(x_i) over V^b."""
    p = _rows(b, V, 10 * b + V)
    want = 0.0
    for x in itertools.product(range(V), repeat=b):
        px = [p[i, x[i]] for i in range(b)]
        want += np.prod(px) * np.mean(np.cumprod(px))
    assert abs(orc.early_determinism_exact(p) - want) < 1e-14


def test_collision_sum_factorises_for_prefix_independent_targets():
    """App. B: the j-th term of D_b is sum_{u in V^j} p(u)^2; with
    prefix-independent rows it factorises into prod_{i<=j} sum_v p_i(v)^2
    (enumerated over V^j)."""
    V, b = 3, 3
    p = _rows(b, V, 6)
    for j in range(1, b + 1):
        lhs = sum(np.prod([p[i, u[i]] for i in range(j)]) ** 2
                  for u in itertools.product(range(V), repeat=j))
        assert abs(lhs - np.prod(orc.collision_probability(p[:j]))) < 1e-15
        brute = sum(p[i, v] ** 2 for v in range(V) for i in [j - 1])
        assert abs(orc.collision_probability(p[j - 1:j])[0] - brute) < 1e-16


def test_closed_forms():
    V, b = 7, 5
    onehot = np.zeros((b, V))
    onehot[np.arange(b), [0, 3, 6, 2, 2]] = 1.0
    assert orc.early_determinism_exact(onehot) == 1.0
    uni = np.full((b, V), 1.0 / V)
    want = sum(V ** -j for j in range(1, b + 1)) / b
    assert abs(orc.early_determinism_exact(uni) - want) < 1e-15
    p = _rows(1, V, 3)
    assert abs(orc.early_determinism_exact(p) - np.sum(p[0] ** 2)) < 1e-16


def test_target_probs_is_tempered_softmax():
    rng = np.random.default_rng(1)
    t = rng.normal(size=(3, 11))
    np.testing.assert_allclose(orc.target_probs(t, 0.7),
                               scipy.special.softmax(t / 0.7, axis=-1), rtol=1e-14)


def test_estimator_is_unbiased_and_draws_follow_the_target():
    from scipy import stats
    b, V = 4, 6
    p = _rows(b, V, 21, scale=1.0)
    d = orc.early_determinism_exact(p)
    ests, first = [], np.zeros(V)
    for n in range(3000):
        e, smp, _ = orc.early_determinism_estimate(p, 1, 99, n)
        ests.append(e)
        first[smp[0, 0]] += 1
    ests = np.array(ests)
    assert abs(ests.mean() - d) < 4 * ests.std() / math.sqrt(len(ests))
    assert stats.chisquare(first, len(ests) * p[0]).pvalue > 1e-3
    # M samples in one call average the same terms as M calls with M = 1
    e20, smp20, _ = orc.early_determinism_estimate(p, 20, 7, 3)
    per = [np.mean(np.cumprod(p[np.arange(b), smp20[m]])) for m in range(20)]
    assert abs(e20 - np.mean(per)) < 1e-15
