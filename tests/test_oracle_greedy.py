"""Pins of the oracle's greedy-branch mode (Sec. 3.1, "Drafter sampling
during inference"; App. A: greedy-branch proposal, prefix-marginalized
conditional, distributional correctness).

The conditional q_greedy is checked against hand-worked examples and against
the prefix marginal of the joint proposal (Eq. greedy-branch-proposal)
enumerated by brute force; the greedy tokens against explicit loops; the
verifier against the distribution-preservation theorem (exact enumeration and
the oracle's own seeded sampler, chi-square); K = 1 and Z_T = 0 against their
closed forms.  CPU only.
"""
import itertools
import math

import numpy as np
import pytest
import scipy.special

from oracle import dblast_oracle as orc
from tests.test_oracle_pins import rand_head


# ------------------------------------------------------------ hand examples
def test_greedy_conditional_hand_example_shared_prefix():
    """Three branches, pi = (0.5, 0.3, 0.2); branches 0 and 1 share their first
    token, branch 2 leaves at position 0 and matches again at position 1."""
    xhat = np.array([[1, 1, 2],
                     [3, 4, 3],
                     [7, 8, 9]])
    pi = np.array([0.5, 0.3, 0.2])
    tokens = xhat[:, 0]                                   # z-hat = 0: (1, 3, 7)
    C = orc.consistent_branches(xhat, tokens)
    assert C.tolist() == [[True, True, True], [True, True, False],
                          [True, False, False]]
    q, pit = orc.greedy_conditional(pi, xhat, C, 10)
    want = np.zeros((3, 10))
    want[0, 1], want[0, 2] = 0.8, 0.2                     # 0.5 + 0.3, 0.2
    want[1, 3], want[1, 4] = 0.625, 0.375                 # 0.5 / 0.8, 0.3 / 0.8
    want[2, 7] = 1.0
    np.testing.assert_allclose(q, want, rtol=0, atol=1e-15)
    np.testing.assert_allclose(pit[1], [0.625, 0.375, 0.0], rtol=0, atol=1e-15)
    # z-hat = 2: the block (2, 3, 9) leaves the other branches at once
    C2 = orc.consistent_branches(xhat, xhat[:, 2])
    q2, _ = orc.greedy_conditional(pi, xhat, C2, 10)
    assert q2[1, 3] == 1.0 and q2[2, 9] == 1.0 and q2[0, 2] == pytest.approx(0.2)


def test_greedy_branch_tokens_brute_force_with_planted_ties():
    rng = np.random.default_rng(3)
    B, K, V = 4, 3, 11
    logits = rng.normal(size=(B, K, V)).round(1)          # rounding makes ties
    logits[1, 2, [3, 8]] = 9.0                            # exact tie at the top
    xhat, gap = orc.greedy_branch_tokens(logits)
    for i in range(B):
        for z in range(K):
            best, second = 0, -math.inf
            for v in range(1, V):
                if logits[i, z, v] > logits[i, z, best]:
                    best = v
            for v in range(V):
                if v != best and logits[i, z, v] > second:
                    second = logits[i, z, v]
            assert xhat[i, z] == best
            assert gap[i, z] == pytest.approx(logits[i, z, best] - second, abs=0)
    assert xhat[1, 2] == 3 and gap[1, 2] == 0.0


# ------------------------------------------------ prefix marginal of the joint
def _greedy_joint(pi, xhat, x):
    """q_greedy(x_{1:i}) = sum_z pi_z prod_{j<=i} 1{x_j = xhat_{j,z}}."""
    return sum(pi[z] for z in range(len(pi))
               if all(xhat[j, z] == x[j] for j in range(len(x))))


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_greedy_conditional_equals_prefix_marginal(seed):
    """Eq. appendix-greedy-conditional == joint(x_<i, v) / joint(x_<i) for every
    prefix with positive proposal mass (Eq. 1 / dep-conditional)."""
    rng = np.random.default_rng(seed)
    B, K, V = 3, 4, 3
    xhat = rng.integers(0, 2, size=(B, K))                # few values: shared prefixes
    pi = rng.dirichlet(np.ones(K))
    checked = 0
    for i in range(B):
        for prefix in itertools.product(range(V), repeat=i):
            den = _greedy_joint(pi, xhat, prefix)
            if den == 0.0:
                continue
            tokens = np.array(list(prefix) + [0] * (B - i))
            q, pit = orc.greedy_conditional(pi, xhat, orc.consistent_branches(xhat, tokens), V)
            assert abs(pit[i].sum() - 1.0) < 1e-15
            for v in range(V):
                want = _greedy_joint(pi, xhat, list(prefix) + [v]) / den
                assert abs(q[i, v] - want) < 1e-15
            checked += 1
    assert checked >= B


# -------------------------------------------------- verification theorems
def _tiny_greedy(K, seed, V=4, H=3, r=2, B=3):
    head = rand_head(V, H, K, r, seed, e=True, vbias=True, wscale=0.4)
    rng = np.random.default_rng(seed + 100)
    h = rng.normal(size=(B, H))
    t = rng.normal(0, 1.5, size=(B + 1, V))
    logits = orc.component_logits(head["W"], orc.branch_hidden(
        h, head["U"], head["Vf"], head["e"]), head["vbias"])
    xhat, _ = orc.greedy_branch_tokens(logits)
    _, pi = orc.category_prior(head["Wp"], head["bp"], h[0], 1.0)
    return head, h, t, xhat, pi


@pytest.mark.parametrize("K", [1, 3, 5])
def test_greedy_emitted_token_is_distributed_as_target_exact(K):
    """App. A (distributional correctness): at every reachable prefix, the
    accepted mass min(p, q_greedy) plus the residual equals p."""
    _, _, t, xhat, pi = _tiny_greedy(K, 10 + K)
    B, V = xhat.shape[0], t.shape[1]
    p = scipy.special.softmax(t, axis=-1)
    for z in range(K):
        tokens = xhat[:, z]
        C = orc.consistent_branches(xhat, tokens)
        q, _ = orc.greedy_conditional(pi, xhat, C, V)
        for i in range(B):
            res = np.maximum(p[i] - q[i], 0)
            res = res / res.sum()
            emit = np.zeros(V)
            for x in range(V):
                if q[i, x] == 0:
                    continue
                acc = min(1.0, p[i, x] / q[i, x])
                emit[x] += q[i, x] * acc
                emit += q[i, x] * (1 - acc) * res
            np.testing.assert_allclose(emit, p[i], rtol=0, atol=1e-14)


@pytest.mark.parametrize("K", [1, 3])
def test_greedy_expected_length_identities(K):
    """Eq. 3 under the greedy proposal: sum_z pi_z sum_i prod_{j<=i} A_j(z)
    equals the path sum of prod min(p, q_greedy) over all prefixes."""
    _, _, t, xhat, pi = _tiny_greedy(K, 30 + K)
    B, V = xhat.shape[0], t.shape[1]
    p = scipy.special.softmax(t, axis=-1)
    e_cond = 0.0
    for z in range(K):
        tokens = xhat[:, z]
        q, _ = orc.greedy_conditional(pi, xhat, orc.consistent_branches(xhat, tokens), V)
        A = [min(1.0, p[i, tokens[i]] / q[i, tokens[i]]) for i in range(B)]
        e_cond += pi[z] * sum(np.prod(A[:i + 1]) for i in range(B))
    path = 0.0
    for i in range(B):
        for x in itertools.product(range(V), repeat=i + 1):
            xx = np.array(list(x) + [0] * (B - i - 1))
            q, _ = orc.greedy_conditional(pi, xhat, orc.consistent_branches(xhat, xx), V)
            path += np.prod([min(p[j, x[j]], q[j, x[j]]) for j in range(i + 1)])
    assert abs(e_cond - path) < 1e-13


def test_greedy_oracle_monte_carlo_matches_exact_laws():
    """The oracle's greedy step (seeded uniforms -> decisions) emits its first
    token from p_0 and drafts x_0 from sum_z pi_z 1{xhat_{0,z}} (chi-square);
    the accepted length averages to the exact E[L] (4 sigma)."""
    from scipy import stats
    K, T = 4, 1.0
    head, h, t, xhat, pi = _tiny_greedy(K, 77, V=5, B=3)
    V = 5
    p = scipy.special.softmax(t / T, axis=-1)
    e_len = 0.0
    for z in range(K):
        tok = xhat[:, z]
        q, _ = orc.greedy_conditional(pi, xhat, orc.consistent_branches(xhat, tok), V)
        A = [min(1.0, p[i, tok[i]] / q[i, tok[i]]) for i in range(3)]
        e_len += pi[z] * sum(np.prod(A[:i + 1]) for i in range(3))
    drafted_law = np.zeros(V)
    for z in range(K):
        drafted_law[xhat[0, z]] += pi[z]
    n = 6000
    first, drafted, Ls = np.zeros(V), np.zeros(V), []
    for seed in range(n):
        out = orc.greedy_draft_and_verify_sequence(head, h, None, t, True, T, 1.0,
                                                   seed, 0, 3, 0)
        first[out["emitted"][0]] += 1
        drafted[out["tokens"][0]] += 1
        Ls.append(out["accepted"])
        if seed < 50:
            assert np.array_equal(out["xhat"], xhat)
            np.testing.assert_allclose(np.exp(out["logw"]).sum(-1), 1.0, atol=1e-14)
            A = out["accept_prob"]
            assert abs(out["exp_len"] - sum(np.prod(A[:i + 1]) for i in range(3))) < 1e-13
    assert stats.chisquare(first, n * p[0]).pvalue > 1e-3
    mask = drafted_law > 0
    assert drafted[~mask].sum() == 0
    assert stats.chisquare(drafted[mask], n * drafted_law[mask]).pvalue > 1e-3
    Ls = np.array(Ls, dtype=float)
    assert abs(Ls.mean() - e_len) < 4 * Ls.std() / math.sqrt(n)


# ------------------------------------------------------------ closed forms
def _run(head, h, t, T, Z_T, seed, B):
    return orc.greedy_draft_and_verify_sequence(head, h, None, t, True, T, Z_T, seed, 0, 7, 2)


@pytest.mark.parametrize("K,Z_T", [(1, 1.0), (4, 0.0)])
def test_greedy_point_mass_cases(K, Z_T):
    """K = 1, or Z_T = 0 with K > 1: q_greedy is a point mass on the drafted
    token, so q = 1, A_i = alpha_i = p_i(x_i), and the residual is p with the
    rejected token removed."""
    B, V = 4, 9
    head, h, t, _, _ = _tiny_greedy(K, 50 + K, V=V, H=5, r=3, B=B)
    ell, _ = orc.category_prior(head["Wp"], head["bp"], h[0], Z_T)
    logits = orc.component_logits(head["W"], orc.branch_hidden(
        h, head["U"], head["Vf"], head["e"]), head["vbias"])
    z_top = int(np.argmax(ell)) if Z_T == 0 else 0
    p = scipy.special.softmax(t, axis=-1)
    rejected = 0
    for seed in range(40):
        o = _run(head, h, t, 1.0, Z_T, seed, B)
        assert o["zhat"] == z_top
        assert o["tokens"].tolist() == [int(np.argmax(logits[i, z_top])) for i in range(B)]
        np.testing.assert_allclose(o["q_tok"], 1.0, rtol=0, atol=0)
        np.testing.assert_allclose(o["accept_prob"], p[np.arange(B), o["tokens"]], rtol=1e-14)
        np.testing.assert_allclose(o["alpha"], o["accept_prob"], rtol=1e-14)
        L = o["accepted"]
        if L < B:
            rejected += 1
            from oracle.philox import STREAM_RESIDUAL, decision_uniform
            res = p[L].copy()
            res[o["tokens"][L]] = 0.0
            u3 = decision_uniform(seed, STREAM_RESIDUAL, 2, 0, 7 + L)
            want, _ = orc.inverse_cdf(res, u3)
            assert o["emitted"][-1] == want
    assert rejected > 5


def test_greedy_tokens_do_not_depend_on_temperature():
    head, h, t, _, _ = _tiny_greedy(3, 91, V=7, H=4, r=2, B=4)
    a = _run(head, h, t, 0.4, 1.0, 5, 4)
    b = _run(head, h, t, 2.5, 1.0, 5, 4)
    assert a["zhat"] == b["zhat"]
    assert np.array_equal(a["xhat"], b["xhat"])
    assert np.array_equal(a["q_tok"], b["q_tok"])


def test_identical_branches_give_a_point_mass_with_all_branches_consistent():
    """U = 0 and no expander bias: every branch is the base head, so all K
    branches are consistent at every position and q = 1 on the shared token."""
    head, h, t, _, _ = _tiny_greedy(4, 95, V=6, H=4, r=2, B=3)
    head = dict(head, U=np.zeros_like(head["U"]), e=None)
    o = _run(head, h, t, 1.0, 1.0, 0, 3)
    assert o["consistent"].all()
    assert (o["xhat"] == o["xhat"][:, :1]).all()
    np.testing.assert_allclose(o["q_tok"], 1.0, rtol=0, atol=1e-15)
