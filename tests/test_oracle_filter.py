"""Pins of the oracle's target filter (temperature, top-k, top-p; Sec. 3.2 and
Sec. 4) and of verification against the filtered target.

The filter is checked against a hand example and a brute-force ranking with
planted ties; the verifier against the distribution-preservation theorem with
the filtered target (exact enumeration), the paper's remark that a draft
leaving the filtered support is rejected (A = 0), and the top-k = 1 case.
CPU only.
"""
import itertools

import numpy as np
import pytest
import scipy.special

from oracle import dblast_oracle as orc
from tests.test_oracle_pins import branch_probs, rand_head


def test_top_p_hand_example():
    p = np.array([0.05, 0.5, 0.15, 0.3])
    t = np.log(p)
    # order 1, 3, 2, 0; preceding mass 0, 0.5, 0.8, 0.95
    out, keep, margin = orc.filter_target(t, 1.0, 0, 0.8)
    assert sorted(keep.tolist()) == [1, 3]
    np.testing.assert_allclose(out, [0, 0.625, 0, 0.375], atol=1e-15)
    assert margin == pytest.approx(0.0, abs=1e-15)       # 0.8 sits exactly on an edge
    out, keep, _ = orc.filter_target(t, 1.0, 0, 0.81)
    assert sorted(keep.tolist()) == [1, 2, 3]
    np.testing.assert_allclose(out, np.array([0, 0.5, 0.15, 0.3]) / 0.95, atol=1e-15)
    # top-k = 2 first, then top-p over the renormalised pair (0.625, 0.375)
    out, keep, _ = orc.filter_target(t, 1.0, 2, 0.6)
    assert keep.tolist() == [1]
    np.testing.assert_allclose(out, [0, 1, 0, 0], atol=0)


def test_top_k_brute_force_with_ties_to_the_lower_index():
    rng = np.random.default_rng(2)
    for trial in range(20):
        V = 30
        t = rng.integers(-3, 4, size=V).astype(np.float64)   # many exact ties
        k = int(rng.integers(1, V))
        _, keep, _ = orc.filter_target(t, 0.9, k, 0.0)
        ranked = sorted(range(V), key=lambda v: (-t[v], v))
        assert sorted(keep.tolist()) == sorted(ranked[:k])
        out, _, _ = orc.filter_target(t, 0.9, k, 0.0)
        w = np.exp(t[ranked[:k]] / 0.9)
        np.testing.assert_allclose(out[ranked[:k]], w / w.sum(), rtol=1e-14)
        assert np.count_nonzero(out) == k


def test_filter_off_is_the_tempered_softmax():
    rng = np.random.default_rng(3)
    t = rng.normal(size=50)
    for k, tp in [(0, 0.0), (50, 1.0), (80, 0.0)]:
        out, keep, margin = orc.filter_target(t, 1.3, k, tp)
        np.testing.assert_allclose(out, scipy.special.softmax(t / 1.3), rtol=1e-14)
        assert len(keep) == 50 and margin == np.inf


@pytest.mark.parametrize("K", [1, 3])
@pytest.mark.parametrize("top_k,top_p", [(2, 0.0), (3, 0.7), (0, 0.5)])
def test_emitted_token_is_distributed_as_the_filtered_target(K, top_k, top_p):
    """App. A with p replaced by the filtered target: accepted mass plus the
    residual equals p' at every position and prefix (exact enumeration), and
    drafts outside the kept set have A = 0."""
    V, H, r, B = 5, 3, 2, 2
    head = rand_head(V, H, K, r, 70 + K, e=True, vbias=True)
    rng = np.random.default_rng(80 + K)
    h = rng.normal(size=(B, H))
    t = rng.normal(0, 1.5, size=(B + 1, V))
    q = branch_probs(head, h, 1.0)
    _, pi = orc.category_prior(head["Wp"], head["bp"], h[0], 1.0)
    ties = []
    p, _ = orc.target_distributions(t, 1.0, top_k, top_p, ties)
    assert not ties
    for i in range(B):
        assert np.count_nonzero(p[i]) < V
        for prefix in itertools.product(range(V), repeat=i):
            x = list(prefix) + [0] * (B - i)
            w = np.exp(orc.posterior(np.log(pi), np.log(q[np.arange(B), :, x]))[i])
            qm = w @ q[i]
            res = np.maximum(p[i] - qm, 0)
            res = res / res.sum()
            emit = np.zeros(V)
            for xi in range(V):
                acc = min(1.0, p[i, xi] / qm[xi])
                if p[i, xi] == 0:
                    assert acc == 0.0
                emit[xi] += qm[xi] * acc
                emit += qm[xi] * (1 - acc) * res
            np.testing.assert_allclose(emit, p[i], rtol=0, atol=1e-13)


def test_step_with_top_k_one_accepts_exactly_the_target_argmax():
    """top-k = 1 makes p' one-hot on the target argmax: a draft is accepted
    iff it equals that token (A = min(1, 1/q) = 1), and the residual after a
    rejection is the argmax itself."""
    V, H, K, r, B = 6, 4, 2, 2, 4
    head = rand_head(V, H, K, r, 5, e=False, vbias=True, wscale=0.3)
    rng = np.random.default_rng(6)
    h = rng.normal(size=(B, H))
    t = rng.normal(0, 1.0, size=(B + 1, V))
    top = np.argmax(t, axis=1)
    for mode in ("soft", "greedy"):
        fn = (orc.draft_and_verify_sequence if mode == "soft"
              else orc.greedy_draft_and_verify_sequence)
        for seed in range(30):
            o = fn(head, h, None, t, True, 1.0, 1.0, seed, 0, 0, 0, top_k=1)
            L = o["accepted"]
            assert all(o["tokens"][j] == top[j] for j in range(L))
            if L < B:
                assert o["tokens"][L] != top[L] and o["accept_prob"][L] == 0.0
            assert o["emitted"][-1] == top[len(o["emitted"]) - 1]
            np.testing.assert_allclose(o["collision"], 1.0)
