"""CPU checks of the parity harness itself (tests/parity.py): a GPU result
built from the oracle's own outputs must pass, and each kind of planted
mistake in it (a wrong accepted length, a tie bit missing where the oracle
sees a tie, a tie bit set on a clean sequence, a skipped comparison) must
fail.  No GPU: the "GPU" outputs here are the oracle's, re-packed."""
import copy

import numpy as np
import pytest
import torch

import synth
from oracle import dblast_oracle as orc
from tests import parity


def _oracle_run(mode="soft", N=8):
    cfg = synth.config("tiny", N=N)
    head = synth.make_head(cfg, "cpu")
    blk = synth.make_block(cfg, head, 0, "cpu")
    pos, rnd = synth.initial_state(cfg, "cpu")
    seqs = list(range(cfg["N"]))
    return parity.run_oracle(head, blk, 1.0, 1.0, 3, pos, rnd, seqs, mode=mode), cfg


def _flags_from_ties(o):
    """Tie bits of the oracle's own ties, each with its near bit."""
    f = 0
    for kind, _, _ in o["ties"]:
        f |= parity.TIE_BITS[kind] | (parity.TIE_BITS[kind] << parity.NEAR_SHIFT)
    return f


def _near(bit):
    return bit | (bit << parity.NEAR_SHIFT)


def _as_gpu(orcs, cfg, mode="soft"):
    """The oracle's outputs in the layout the binding returns."""
    N, B, K = cfg["N"], cfg["B"], cfg["K"]
    g = {}
    f32 = lambda key, shape: torch.tensor(np.array([o[key] for o in orcs]),  # noqa: E731
                                          dtype=torch.float32).reshape(shape)
    g["z_hat"] = torch.tensor([o["zhat"] for o in orcs], dtype=torch.int32)
    g["pi"] = f32("pi", (N, K))
    g["tokens"] = torch.tensor(np.array([o["tokens"] for o in orcs]), dtype=torch.int32)
    g["logw"] = f32("logw", (N, B, K))
    for key in ("q_tok", "p_tok", "accept_prob", "alpha"):
        g[key] = f32(key, (N, B))
    g["lse_target"] = f32("lse_target", (N, -1))
    g["exp_len"] = f32("exp_len", (N,))
    g["alpha_len"] = f32("alpha_len", (N,))
    g["collision"] = f32("collision", (N, B))
    g["determinism"] = f32("determinism", (N,))
    g["accepted"] = torch.tensor([o["accepted"] for o in orcs], dtype=torch.int32)
    g["n_emitted"] = torch.tensor([o["n_emitted"] for o in orcs], dtype=torch.int32)
    em = torch.full((N, B + 1), -1, dtype=torch.int32)
    for n, o in enumerate(orcs):
        em[n, :o["n_emitted"]] = torch.tensor(o["emitted"], dtype=torch.int32)
    g["emitted"] = em
    g["tie_flags"] = torch.tensor([_flags_from_ties(o) for o in orcs], dtype=torch.int32)
    if mode == "soft":
        g["lse"] = f32("lse", (N, B, K))
    else:
        g["branch_tokens"] = torch.tensor(np.array([o["xhat"] for o in orcs]), dtype=torch.int32)
    return g


@pytest.mark.parametrize("mode", ["soft", "greedy"])
def test_oracle_outputs_pass_the_harness(mode):
    orcs, cfg = _oracle_run(mode)
    g = _as_gpu(orcs, cfg, mode)
    cmp = parity.compare if mode == "soft" else parity.compare_greedy
    st = cmp(g, orcs, list(range(cfg["N"])))
    assert st["emitted_checked"] >= 6


def test_wrong_accepted_length_fails():
    orcs, cfg = _oracle_run()
    g = _as_gpu(orcs, cfg)
    n = next(i for i, o in enumerate(orcs) if not o["ties"])
    g["accepted"][n] += 1
    with pytest.raises(AssertionError):
        parity.compare(g, orcs, list(range(cfg["N"])))


def test_missing_tie_flag_fails():
    orcs, cfg = _oracle_run()
    orcs = copy.deepcopy(orcs)
    g = _as_gpu(orcs, cfg)
    # plant a draft decision 1e-9 from its threshold in a clean sequence
    n = next(i for i, o in enumerate(orcs) if not o["ties"])
    o = orcs[n]
    for k, d in enumerate(o["decisions"]):
        if d[0] == "draft":
            o["decisions"][k] = ("draft", d[1], 1e-9)
            o["ties"].append(("draft", d[1], 1e-9))
            break
    with pytest.raises(AssertionError, match="tie flag not set"):
        parity.check_tie_flags(g["tie_flags"][n], o, n)
    # a tie bit alone (without its near bit) is malformed
    with pytest.raises(AssertionError, match="without its near bit"):
        parity.check_tie_flags(int(g["tie_flags"][n]) | 2, o, n)
    # with the near bit the sequence passes, with or without the tie bit
    parity.check_tie_flags(int(g["tie_flags"][n]) | (2 << parity.NEAR_SHIFT), o, n)
    parity.check_tie_flags(int(g["tie_flags"][n]) | _near(2), o, n)


def test_spurious_tie_flag_fails():
    orcs, cfg = _oracle_run()
    n = next(i for i, o in enumerate(orcs) if all(d[2] >= 2e-3 for d in o["decisions"]))
    for bit in (1, 2, 4, 8, 16, 32):
        with pytest.raises(AssertionError, match="without a near decision"):
            parity.check_tie_flags(bit << parity.NEAR_SHIFT, orcs[n], n)
        with pytest.raises(AssertionError, match="without a near decision"):
            parity.check_tie_flags(_near(bit), orcs[n], n)


def test_a_tie_in_the_band_may_go_either_way():
    orcs, cfg = _oracle_run()
    orcs = copy.deepcopy(orcs)
    n = next(i for i, o in enumerate(orcs) if not o["ties"])
    o = orcs[n]
    k = next(k for k, d in enumerate(o["decisions"]) if d[0] == "accept")
    o["decisions"][k] = ("accept", o["decisions"][k][1], 3e-6)
    parity.check_tie_flags(0, o, n)
    parity.check_tie_flags(4 << parity.NEAR_SHIFT, o, n)
    parity.check_tie_flags(_near(4), o, n)


def test_vacuous_comparison_fails():
    """Every sequence excluded (z-hat drawn differently at a tie in each) is
    not a pass."""
    orcs, cfg = _oracle_run()
    orcs = copy.deepcopy(orcs)
    for o in orcs:
        o["decisions"] = [d for d in o["decisions"] if d[0] != "zhat"] + [("zhat", -1, 0.0)]
        o["ties"].append(("zhat", -1, 0.0))
    g = _as_gpu(orcs, cfg)
    g["z_hat"] = (g["z_hat"] + 1) % cfg["K"]
    g["tie_flags"] |= _near(1)
    with pytest.raises(AssertionError, match="too few sequences"):
        parity.compare(g, orcs, list(range(cfg["N"])))


def test_dependencies_of_decisions():
    zh = ("zhat", -1, 1.0)
    d3 = ("draft", 3, 1.0)
    a2 = ("accept", 2, 1.0)
    a3 = ("accept", 3, 1.0)
    r3 = ("residual", 3, 1.0)
    rm3 = ("residual_mass", 3, 1.0)
    g1 = ("greedy", 1, 1.0)
    g2 = ("greedy", 2, 1.0)
    tp4 = ("top_p", 4, 1.0)
    assert parity._prereq(zh, d3) and not parity._prereq(a2, d3)
    assert parity._prereq(d3, a3) and parity._prereq(a2, a3) and not parity._prereq(a3, a2)
    assert parity._prereq(rm3, r3) and parity._prereq(a3, r3)
    assert parity._prereq(g1, g2) and not parity._prereq(g2, g1)
    assert not parity._prereq(tp4, a3) and parity._prereq(tp4, ("accept", 4, 1.0))
    assert not parity._prereq(zh, tp4)


def test_a_token_changed_at_a_tie_is_excused_elsewhere_it_fails():
    orcs, cfg = _oracle_run()
    orcs = copy.deepcopy(orcs)
    g = _as_gpu(orcs, cfg)
    n = next(i for i, o in enumerate(orcs) if not o["ties"])
    o = orcs[n]
    g["tokens"][n][1] = (int(g["tokens"][n][1]) + 1) % cfg["V"]
    with pytest.raises(AssertionError, match="tokens"):
        parity.compare(g, orcs, list(range(cfg["N"])))
    # the same change where the oracle's draw was within the tie tolerance
    k = next(k for k, d in enumerate(o["decisions"]) if d[0] == "draft" and d[1] == 1)
    o["decisions"][k] = ("draft", 1, 5e-7)
    o["ties"].append(("draft", 1, 5e-7))
    g["tie_flags"][n] = int(g["tie_flags"][n]) | _near(2)
    st = parity.compare(g, orcs, list(range(cfg["N"])))
    assert st["diverged"] == 1 and st["precision_flips"] == 0


def test_a_flip_inside_the_precision_band_is_excused_and_counted():
    """A draw 2e-5 from its threshold is no tie (1e-6), but lies inside the
    kernels' precision band (1e-6 + NEAR_DRAW): a flip there is excused and
    counted; at 2e-3 it fails."""
    orcs, cfg = _oracle_run()
    orcs = copy.deepcopy(orcs)
    g = _as_gpu(orcs, cfg)
    n = next(i for i, o in enumerate(orcs) if not o["ties"])
    o = orcs[n]
    k = next(k for k, d in enumerate(o["decisions"]) if d[0] == "draft" and d[1] == 0)
    g["tokens"][n][0] = (int(g["tokens"][n][0]) + 1) % cfg["V"]
    g["tie_flags"][n] = int(g["tie_flags"][n]) | (2 << parity.NEAR_SHIFT)
    o["decisions"][k] = ("draft", 0, 2e-3)
    with pytest.raises(AssertionError, match="tokens"):
        parity.compare(g, orcs, list(range(cfg["N"])))
    o["decisions"][k] = ("draft", 0, 2e-5)
    st = parity.compare(g, orcs, list(range(cfg["N"])))
    assert st["precision_flips"] == 1
