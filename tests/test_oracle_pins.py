"""Pins of the fp64 oracle against what the paper and the mathematics fix.

Each check ties the oracle to something other than itself: the printed
Table 1, brute-force loops over explicit indices, library routines (scipy,
torch fp64 matmul), exact enumeration of the joint proposal (Eq. 1 vs the
posterior form), the distribution-preservation theorem of speculative
sampling (Appendix A), and closed forms of the expected accepted length
(Eq. 3).  CPU only.
"""
import itertools
import math
import os

import numpy as np
import pytest
import scipy.special
import torch

from oracle import dblast_oracle as orc
from oracle.philox import STREAM_PRIOR, decision_uniform

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def rand_head(V, H, K, r, seed, e=False, vbias=False, wscale=0.5):
    rng = np.random.default_rng(seed)
    head = {
        "W": rng.normal(0, wscale, (V, H)),
        "U": rng.normal(0, 1 / math.sqrt(r), (K, H, r)),
        "Vf": rng.normal(0, 1 / math.sqrt(r), (K, H, r)),
        "e": rng.normal(0, 0.5, (K, H)) if e else None,
        "Wp": rng.normal(0, 1.0, (K, H)),
        "bp": rng.normal(0, 0.3, K),
        "vbias": rng.normal(0, 0.5, V) if vbias else None,
    }
    return head


def branch_probs(head, h, T):
    """q_i(.|z) for all i, z via the oracle's head functions."""
    s = orc.component_logits(head["W"], orc.branch_hidden(
        h, head["U"], head["Vf"], head["e"]), head["vbias"]) / T
    return np.exp(s - orc.logsumexp(s)[..., None])           # [B, K, V]


# ----------------------------------------------------------------- Table 1
def test_table1_parameter_overhead():
    rows = []
    with open(os.path.join(GOLDEN, "table1_parameter_overhead.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                H, K, m = line.split()
                rows.append((int(H), int(K), float(m)))
    assert len(rows) == 2
    for H, K, m in rows:
        assert round(orc.expander_parameter_count(H, K) / 1e6, 1) == m
    assert orc.expander_parameter_count(2560, 4) == 26234884
    assert orc.expander_parameter_count(4096, 4, rank=16) == \
        2 * 4 * 4096 * 16 + 2 * 4 * 4096 + 4


# ---------------------------------------------------------- inverse CDF
def test_inverse_cdf_hand_cases():
    w = [0.2, 0.3, 0.5]
    assert orc.inverse_cdf(w, 0.1)[0] == 0
    assert orc.inverse_cdf(w, 0.2)[0] == 1          # strict: C(0)=0.2 is not > 0.2
    assert orc.inverse_cdf(w, 0.49)[0] == 1
    assert orc.inverse_cdf(w, 0.5)[0] == 2
    assert orc.inverse_cdf([2, 3, 5], 0.49)[0] == 1  # unnormalised weights
    assert orc.inverse_cdf([0, 1, 0, 1], 0.25)[0] == 1
    assert orc.inverse_cdf([0, 1, 0, 1], 0.75)[0] == 3
    idx, margin = orc.inverse_cdf(w, 0.3)
    assert idx == 1 and abs(margin - 0.1) < 1e-15


def test_inverse_cdf_stratified_frequencies_are_exact():
    rng = np.random.default_rng(3)
    w = rng.random(13) ** 3
    w[[2, 7]] = 0.0
    n = 100000
    counts = np.zeros(13)
    for k in range(n):
        counts[orc.inverse_cdf(w, (k + 0.5) / n)[0]] += 1
    assert np.all(np.abs(counts - n * w / w.sum()) <= 1.0 + 1e-9)
    assert counts[2] == 0 and counts[7] == 0


# ------------------------------------------------------------------ prior
def test_category_prior_is_softmax_and_zt0_is_argmax():
    rng = np.random.default_rng(5)
    Wp, bp, a = rng.normal(size=(6, 9)), rng.normal(size=6), rng.normal(size=9)
    ell, pi = orc.category_prior(Wp, bp, a, 0.7)
    np.testing.assert_allclose(ell, Wp @ a + bp, rtol=0, atol=1e-13)
    np.testing.assert_allclose(pi, scipy.special.softmax(ell / 0.7),
                               rtol=1e-13, atol=0)
    assert abs(pi.sum() - 1) < 1e-14
    _, pi0 = orc.category_prior(Wp, bp, a, 0.0)
    assert pi0[np.argmax(ell)] == 1.0 and pi0.sum() == 1.0
    _, pi_small = orc.category_prior(Wp, bp, a, 1e-4)
    assert abs(pi_small[np.argmax(ell)] - 1.0) < 1e-12


def test_zt0_always_selects_highest_prior_category():
    head = rand_head(7, 5, 4, 2, 11)
    rng = np.random.default_rng(0)
    h = rng.normal(size=(2, 5))
    t = rng.normal(size=(3, 7))
    ell = head["Wp"] @ h[0] + head["bp"]
    for seed in range(20):
        out = orc.draft_and_verify_sequence(head, h, None, t, True, 1.0, 0.0,
                                            seed, 0, 10, 0)
        assert out["zhat"] == int(np.argmax(ell))


# ------------------------------------------------------- component logits
def test_component_logits_brute_force_loops():
    """l[i,z,v] = sum_c W[v,c] (h[i,c] + sum_k U[z,c,k] sum_d V[z,d,k] h[i,d] + e[z,c]) + b[v]."""
    V, H, K, r, B = 5, 3, 2, 2, 2
    head = rand_head(V, H, K, r, 1, e=True, vbias=True)
    h = np.random.default_rng(2).normal(size=(B, H))
    got = orc.component_logits(head["W"], orc.branch_hidden(
        h, head["U"], head["Vf"], head["e"]), head["vbias"])
    W, U, Vf, e, b = (head[k] for k in ("W", "U", "Vf", "e", "vbias"))
    for i in range(B):
        for z in range(K):
            for v in range(V):
                acc = 0.0
                for c in range(H):
                    hz = h[i, c] + e[z, c]
                    for k in range(r):
                        code = sum(Vf[z, d, k] * h[i, d] for d in range(H))
                        hz += U[z, c, k] * code
                    acc += W[v, c] * hz
                assert abs(got[i, z, v] - (acc + b[v])) < 1e-12


def test_component_logits_reduce_to_lm_head_when_expander_is_zero():
    V, H, K, r, B = 40, 12, 3, 4, 5
    head = rand_head(V, H, K, r, 4, vbias=True)
    head["U"] = np.zeros_like(head["U"])
    h = np.random.default_rng(9).normal(size=(B, H))
    got = orc.component_logits(head["W"], orc.branch_hidden(
        h, head["U"], head["Vf"], None), head["vbias"])
    ref = (torch.tensor(h) @ torch.tensor(head["W"]).T).numpy() + head["vbias"]
    for z in range(K):
        np.testing.assert_allclose(got[:, z, :], ref, rtol=0, atol=1e-12)
    lse = orc.logsumexp(got / 0.8)
    np.testing.assert_allclose(lse, scipy.special.logsumexp(got / 0.8, axis=-1),
                               rtol=1e-14)


def test_component_logits_accept_bf16_head_in_chunks():
    V, H = 50, 16
    W = torch.randn(V, H, generator=torch.Generator().manual_seed(0)).to(
        torch.bfloat16)
    hz = np.random.default_rng(1).normal(size=(2, 3, H))
    got = orc.component_logits(W, hz, None, chunk=7)
    ref = hz.reshape(6, H) @ W.double().numpy().T
    np.testing.assert_allclose(got.reshape(6, V), ref, rtol=0, atol=1e-12)


# ------------------------------------------------------------- posterior
def _joint(pi, q, x):
    """q(x_{1:i}) = sum_z pi_z prod_j q_j(x_j|z) (Eq. 5), by brute force."""
    tot = 0.0
    for z in range(len(pi)):
        prod = pi[z]
        for j, xj in enumerate(x):
            prod *= q[j, z, xj]
        tot += prod
    return tot


@pytest.mark.parametrize("K", [1, 2, 3])
def test_posterior_mixture_equals_prefix_marginal_eq1(K):
    """Eq. category-posterior + Eq. dep-next-token == Eq. 1 / dep-conditional."""
    V, H, r, B = 4, 3, 2, 3
    head = rand_head(V, H, K, r, 20 + K, e=True, vbias=True)
    h = np.random.default_rng(K).normal(size=(B, H))
    q = branch_probs(head, h, 0.9)
    _, pi = orc.category_prior(head["Wp"], head["bp"], h[0], 1.0)
    for i in range(B):
        for prefix in itertools.product(range(V), repeat=i):
            x = list(prefix) + [0] * (B - i)
            logq_at_x = np.log(q[np.arange(B), :, x])
            w = np.exp(orc.posterior(np.log(pi), logq_at_x)[i])
            assert abs(w.sum() - 1) < 1e-13
            mix = w @ q[i]                                  # [V]
            den = _joint(pi, q, prefix)
            for v in range(V):
                eq1 = _joint(pi, q, list(prefix) + [v]) / den
                assert abs(mix[v] - eq1) < 1e-12
            if K == 1:
                np.testing.assert_allclose(mix, q[i, 0], rtol=0, atol=1e-15)


# -------------------------------------------------- verification theorems
def _tiny_case(K, seed, V=4, H=3, r=2, B=2):
    head = rand_head(V, H, K, r, seed, e=True, vbias=True)
    rng = np.random.default_rng(seed + 100)
    h = rng.normal(size=(B, H))
    t = rng.normal(0, 1.5, size=(B + 1, V))
    return head, h, t


@pytest.mark.parametrize("K", [1, 3])
def test_emitted_token_is_distributed_as_target_exact(K):
    """Appendix A: accepted mass min(p, q) plus residual mass = p, at every
    position and after every accepted prefix (exact enumeration)."""
    head, h, t = _tiny_case(K, 40 + K)
    T = 1.0
    B, V = h.shape[0], head["W"].shape[0]
    q = branch_probs(head, h, T)
    _, pi = orc.category_prior(head["Wp"], head["bp"], h[0], 1.0)
    p = scipy.special.softmax(t / T, axis=-1)
    for i in range(B):
        for prefix in itertools.product(range(V), repeat=i):
            x = list(prefix) + [0] * (B - i)
            w = np.exp(orc.posterior(np.log(pi), np.log(
                q[np.arange(B), :, x]))[i])
            qm = w @ q[i]
            res = np.maximum(p[i] - qm, 0)
            res = res / res.sum()
            emit = np.zeros(V)
            for xi in range(V):
                acc = min(1.0, p[i, xi] / qm[xi])
                emit[xi] += qm[xi] * acc
                emit += qm[xi] * (1 - acc) * res
            np.testing.assert_allclose(emit, p[i], rtol=0, atol=1e-13)


def _exact_expected_length(head, h, t, T):
    B, V = h.shape[0], head["W"].shape[0]
    q = branch_probs(head, h, T)
    _, pi = orc.category_prior(head["Wp"], head["bp"], h[0], 1.0)
    p = scipy.special.softmax(t / T, axis=-1)
    e_cond, path = 0.0, 0.0
    for x in itertools.product(range(V), repeat=B):
        qx = _joint(pi, q, x)
        logw = orc.posterior(np.log(pi), np.log(q[np.arange(B), :, list(x)]))
        qcond = [np.exp(logw[i]) @ q[i, :, x[i]] for i in range(B)]
        A = [min(1.0, p[i, x[i]] / qcond[i]) for i in range(B)]
        e_cond += qx * sum(np.prod(A[:i + 1]) for i in range(B))
    # path form: sum_i sum_{x_<=i} prod_{j<=i} min(p_j(x_j), q(x_j|x_<j))
    for i in range(B):
        for x in itertools.product(range(V), repeat=i + 1):
            xx = list(x) + [0] * (B - i - 1)
            logw = orc.posterior(np.log(pi), np.log(q[np.arange(B), :, xx]))
            prod = 1.0
            for j in range(i + 1):
                prod *= min(p[j, x[j]], np.exp(logw[j]) @ q[j, :, x[j]])
            path += prod
    return e_cond, path, q, pi, p


@pytest.mark.parametrize("K", [1, 2])
def test_expected_length_identities(K):
    """Eq. 3: E_q[sum_i prod_{j<=i} A_j] equals the path sum of prod min(p, q);
    for K = 1 it also equals sum_i prod_{j<=i} alpha_j."""
    head, h, t = _tiny_case(K, 60 + K, V=5, B=3)
    e_cond, path, q, pi, p = _exact_expected_length(head, h, t, 1.0)
    assert abs(e_cond - path) < 1e-12
    if K == 1:
        alphas = [np.minimum(p[i], q[i, 0]).sum() for i in range(3)]
        assert abs(e_cond - sum(np.prod(alphas[:i + 1]) for i in range(3))) \
            < 1e-12


def test_oracle_step_monte_carlo_matches_exact_laws():
    """The oracle's own sampler (uniforms -> decisions) reproduces p_0 for the
    first emitted token (chi-square) and the exact E[L] (4 sigma)."""
    from scipy import stats
    head, h, t = _tiny_case(2, 77, V=5, B=3)
    T = 0.7
    e_len, _, q, pi, p = _exact_expected_length(head, h, t, T)
    n = 60000
    first = np.zeros(5)
    drafted = np.zeros(5)
    Ls = []
    for seed in range(n):
        out = orc.draft_and_verify_sequence(head, h, None, t, True, T, 1.0,
                                            seed, 0, 3, 0)
        first[out["emitted"][0]] += 1
        drafted[out["tokens"][0]] += 1
        Ls.append(out["accepted"])
        if seed < 50:
            lw = out["logw"]
            np.testing.assert_allclose(np.exp(lw).sum(-1), 1.0, atol=1e-13)
            A = out["accept_prob"]
            assert abs(out["exp_len"] - sum(np.prod(A[:i + 1])
                                            for i in range(3))) < 1e-13
    assert stats.chisquare(first, n * p[0]).pvalue > 1e-3
    assert stats.chisquare(drafted, n * (pi @ q[0])).pvalue > 1e-3
    Ls = np.array(Ls, dtype=float)
    assert abs(Ls.mean() - e_len) < 4 * Ls.std() / math.sqrt(n)


def test_target_equal_to_drafter_accepts_everything():
    """K = 1 and p = q: alpha = 1, A = 1, every token accepted, E[L|x] = B."""
    V, H, B = 9, 4, 3
    head = rand_head(V, H, 1, 2, 90, vbias=True)
    h = np.random.default_rng(1).normal(size=(B, H))
    l = orc.component_logits(head["W"], orc.branch_hidden(
        h, head["U"], head["Vf"], None), head["vbias"])[:, 0, :]
    t = np.concatenate([l, l[:1]], axis=0)
    for seed in range(30):
        out = orc.draft_and_verify_sequence(head, h, None, t, True, 0.8, 1.0,
                                            seed, 0, 0, 0)
        assert out["accepted"] == B and out["n_emitted"] == B + 1
        np.testing.assert_allclose(out["alpha"], 1.0, atol=1e-13)
        assert abs(out["exp_len"] - B) < 1e-12
        assert abs(out["alpha_len"] - B) < 1e-12


def test_disjoint_target_rejects_and_resamples_from_residual():
    V, H, B = 12, 4, 3
    head = rand_head(V, H, 2, 2, 91, wscale=3.0)
    h = np.random.default_rng(2).normal(size=(B, H))
    q = branch_probs(head, h, 1.0)
    # target puts its mass where the mixture has least
    t = -50.0 * q.max(axis=1)
    t = np.concatenate([t, t[:1]], axis=0)
    n_rej = 0
    for seed in range(40):
        out = orc.draft_and_verify_sequence(head, h, None, t, False, 1.0, 1.0,
                                            seed, 0, 0, 0)
        if out["accepted"] == 0:
            n_rej += 1
            y = out["emitted"][0]
            p0 = scipy.special.softmax(t[0])
            w0 = out["logw"][0]
            assert p0[y] > np.exp(w0) @ q[0, :, y]
    assert n_rej >= 30


def test_prior_draw_uses_stream_zero_uniform():
    head, h, t = _tiny_case(3, 5)
    _, pi = orc.category_prior(head["Wp"], head["bp"], h[0], 1.3)
    for seed in range(10):
        out = orc.draft_and_verify_sequence(head, h, None, t, True, 1.0, 1.3,
                                            seed, 4, 21, 2)
        u0 = decision_uniform(seed, STREAM_PRIOR, 2, 4, 21)
        assert out["zhat"] == int(np.searchsorted(np.cumsum(pi), u0,
                                                  side="right"))
