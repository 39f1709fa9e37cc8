"""Pins of the oracle's training-side objectives, forward only (Sec. 3.2):
the block NLL against the brute-force joint proposal (Eq. 5) and the chain
rule, the prefix importance ratio r_l against the joint, the accepted-length
identity of Eq. acceptance-length-objective by exhaustive enumeration, and
hand-computed S_l, l_tau and J_AL.  CPU only."""
import itertools
import math

import numpy as np
import pytest
import scipy.special

from oracle import dblast_oracle as orc
from tests.test_oracle_pins import _exact_expected_length, _joint, branch_probs, rand_head


def _tiny(K, seed, V=4, H=3, r=2, b=3):
    head = rand_head(V, H, K, r, seed, e=True, vbias=True)
    rng = np.random.default_rng(seed + 1)
    h = rng.normal(size=(b, H))
    t = rng.normal(0, 1.5, size=(b + 1, V))
    return head, h, t


@pytest.mark.parametrize("K", [1, 3])
def test_block_nll_and_ratio_against_the_joint(K):
    head, h, t = _tiny(K, 100 + K)
    b, V = h.shape[0], head["W"].shape[0]
    q = branch_probs(head, h, 0.9)
    _, pi = orc.category_prior(head["Wp"], head["bp"], h[0], 1.0)
    p = scipy.special.softmax(t / 0.9, axis=-1)
    for x in itertools.product(range(V), repeat=b):
        o = orc.al_objective_sequence(head, h, None, t, list(x), 0.9, 1.0, 0.1)
        assert abs(o["nll"] + math.log(_joint(pi, q, x))) < 1e-12
        assert abs(o["nll"] + np.sum(np.log(o["q_cond"]))) < 1e-12       # chain rule
        for l in range(1, b + 1):
            want = _joint(pi, q, x[:l]) / np.prod([p[j, x[j]] for j in range(l)])
            assert abs(o["r"][l - 1] - want) < 1e-12 * max(1.0, want)
        if K == 1:
            assert abs(o["nll"] + sum(math.log(q[i, 0, x[i]]) for i in range(b))) < 1e-12


@pytest.mark.parametrize("K", [1, 2])
def test_accepted_length_identity_eq_acceptance_length_objective(K):
    """E_{x~q}[AL_b] = sum_l E_{x~p}[r_l prod_{j<=l} A_j] (exact enumeration)."""
    head, h, t = _tiny(K, 200 + K, V=4, b=3)
    e_cond, path, q, pi, p = _exact_expected_length(head, h, t, 1.0)
    rhs = 0.0
    for x in itertools.product(range(4), repeat=3):
        o = orc.al_objective_sequence(head, h, None, t, list(x), 1.0, 1.0, 0.0)
        px = np.prod([p[j, x[j]] for j in range(3)])
        rhs += px * sum(o["r"][l] * np.prod(o["A"][:l + 1]) for l in range(3))
    assert abs(rhs - e_cond) < 1e-12


def test_surrogate_hand_example():
    q = [0.5, 0.2, 0.1]
    p = [0.5, 0.5, 0.5]
    o = orc.al_surrogate(q, p, 0.1)
    np.testing.assert_allclose(o["A"], [1.0, 1.0, 1.0], rtol=1e-15)     # p / q = 1, 2.5, 5
    np.testing.assert_allclose(o["r"], [1.0, 0.4, 0.08], rtol=1e-15)
    np.testing.assert_allclose(o["S"], [1.0, 2.0, 3.0], rtol=1e-15)
    assert o["l_tau"] == 3
    want = math.log(0.4) + math.log(2.0) + math.log(0.08) + math.log(3.0)
    assert abs(o["J"] - want) < 1e-14
    o = orc.al_surrogate(q, p, 0.5)
    assert o["l_tau"] == 2
    assert abs(o["J"] - (math.log(0.4) + math.log(2.0))) < 1e-14
    assert orc.al_surrogate(q, p, 0.0)["l_tau"] == 3
    # rejections: q = (0.5, 0.8), p = (0.5, 0.4): A = (1, 0.5), r = (1, 2), S = (1, 1.5)
    o = orc.al_surrogate([0.5, 0.8], [0.5, 0.4], 0.1)
    np.testing.assert_allclose(o["A"], [1.0, 0.5], rtol=1e-15)
    np.testing.assert_allclose(o["r"], [1.0, 2.0], rtol=1e-15)
    np.testing.assert_allclose(o["S"], [1.0, 1.5], rtol=1e-15)
    assert o["l_tau"] == 2 and abs(o["J"] - (math.log(2.0) + math.log(1.5))) < 1e-14
    # the first position below tau is kept, later ones are not
    o = orc.al_surrogate([0.01, 0.5, 0.5], [0.5, 0.5, 0.5], 0.1)
    assert o["l_tau"] == 1 and abs(o["J"] - math.log(0.02)) < 1e-14
