"""Parity harness: run the CUDA step and the fp64 oracle on the same seeded
inputs and compare them with the agreed rules.

Integer outputs (latent category, draft tokens, accepted length, emitted
tokens) must be identical, except where the oracle finds a decision within
1e-6 of its threshold (a "tie"); the decisions that depend on a tie are
excluded.  Probabilities, overlaps, log-sum-exps and expected lengths must
agree within RTOL relative (plus a tiny absolute floor for values near 0).
"""
import numpy as np
import torch

from oracle import dblast_oracle as orc

RTOL = 1e-4
ATOL_PROB = 1e-7


def run_gpu(head_t, blk, T, Z_T, seed, pos, rnd, impl="auto", head=None, ws=None, mode="soft",
            top_k=0, top_p=0.0):
    from paper_2608_05448_gb300 import Head, Workspace, dblast_draft_and_verify
    head = head or Head.from_dict(head_t)
    N, B, _ = blk["hidden"].shape
    ws = ws or Workspace(head, N, B, blk["has_bonus"])
    dout, vout = dblast_draft_and_verify(head, ws, blk["hidden"], pos, rnd, T, Z_T, seed,
                                         blk["target"], blk["has_bonus"],
                                         anchor=blk.get("anchor"), impl=impl, mode=mode,
                                         top_k=top_k, top_p=top_p)
    torch.cuda.synchronize()
    out = {k: v.cpu() for k, v in dout.items()}
    out.update({k: v.cpu() for k, v in vout.items()})
    return out


def run_oracle(head_t, blk, T, Z_T, seed, pos, rnd, seqs, mode="soft", top_k=0, top_p=0.0):
    return orc.draft_and_verify(head_t, blk["hidden"], blk.get("anchor"), blk["target"],
                                blk["has_bonus"], T, Z_T, seed, pos.cpu().numpy(),
                                rnd.cpu().numpy(), seqs=seqs, mode=mode, top_k=top_k,
                                top_p=top_p)


def _close(name, got, want, rtol=RTOL, atol=ATOL_PROB):
    got = np.asarray(got, dtype=np.float64)
    want = np.asarray(want, dtype=np.float64)
    bad = np.abs(got - want) > atol + rtol * np.abs(want)
    if bad.any():
        i = np.argwhere(bad)[0]
        raise AssertionError("%s mismatch at %s: gpu %r oracle %r" %
                             (name, tuple(i), got[tuple(i)], want[tuple(i)]))


def compare(gpu, orc_list, seqs, stats=None):
    """Compare GPU outputs (dict of CPU tensors) with oracle dicts for `seqs`."""
    stats = stats if stats is not None else {}
    for key in ("sequences", "tie_sequences", "positions", "emitted_checked"):
        stats.setdefault(key, 0)
    for o, n in zip(orc_list, seqs):
        stats["sequences"] += 1
        B = len(o["tokens"])
        ties = o["ties"]
        if ties:
            stats["tie_sequences"] += 1
        if any(k == "zhat" for k, _, _ in ties):
            continue
        assert int(gpu["z_hat"][n]) == o["zhat"], ("z_hat", n)
        _close("pi", gpu["pi"][n], o["pi"], atol=1e-7)
        j = min([i for k, i, _ in ties if k in ("draft", "top_p")], default=B)
        _close("lse", gpu["lse"][n], o["lse"], rtol=1e-5, atol=1e-4)
        assert list(gpu["tokens"][n][:j].tolist()) == [int(x) for x in o["tokens"][:j]], \
            ("tokens", n, gpu["tokens"][n].tolist(), o["tokens"].tolist())
        jj = min(j + 1, B)
        _close("posterior", np.exp(gpu["logw"][n][:jj].double().numpy()),
               np.exp(o["logw"][:jj]), atol=1e-6)
        _close("q_tok", gpu["q_tok"][n][:j], o["q_tok"][:j])
        _close("p_tok", gpu["p_tok"][n][:j], o["p_tok"][:j])
        _close("accept_prob", gpu["accept_prob"][n][:j], o["accept_prob"][:j])
        _close("alpha", gpu["alpha"][n][:jj], o["alpha"][:jj], atol=1e-6)
        _close("lse_target", gpu["lse_target"][n], o["lse_target"], rtol=1e-5, atol=1e-4)
        if "collision" in gpu:
            _close("collision", gpu["collision"][n], o["collision"], atol=1e-7)
            _close("determinism", gpu["determinism"][n], o["determinism"], atol=1e-7)
        stats["positions"] += j
        if j == B:
            _close("exp_len", gpu["exp_len"][n], o["exp_len"], atol=1e-6)
            _close("alpha_len", gpu["alpha_len"][n], o["alpha_len"], atol=1e-6)
        if not ties:
            L = o["accepted"]
            assert int(gpu["accepted"][n]) == L, ("accepted", n, int(gpu["accepted"][n]), L)
            assert int(gpu["n_emitted"][n]) == o["n_emitted"], ("n_emitted", n)
            em = gpu["emitted"][n].tolist()
            assert em[:o["n_emitted"]] == o["emitted"], ("emitted", n, em, o["emitted"])
            assert all(x == -1 for x in em[o["n_emitted"]:])
            stats["emitted_checked"] += 1
    return stats


def compare_greedy(gpu, orc_list, seqs, stats=None):
    """Greedy-branch mode: as compare(), with the greedy argmax ties (top-two
    logit gap below the oracle's GREEDY_TIE_TOL, for a branch in C_i) ending
    the checked prefix, and every branch token checked where its gap is clear."""
    stats = stats if stats is not None else {}
    for key in ("sequences", "tie_sequences", "positions", "emitted_checked", "branch_tokens"):
        stats.setdefault(key, 0)
    for o, n in zip(orc_list, seqs):
        stats["sequences"] += 1
        B, K = o["xhat"].shape
        ties = o["ties"]
        if ties:
            stats["tie_sequences"] += 1
        clear = o["gap"] >= orc.GREEDY_TIE_TOL
        bt = gpu["branch_tokens"][n].numpy()
        assert (bt[clear] == o["xhat"][clear]).all(), ("branch_tokens", n)
        stats["branch_tokens"] += int(clear.sum())
        if any(k == "zhat" for k, _, _ in ties):
            continue
        assert int(gpu["z_hat"][n]) == o["zhat"], ("z_hat", n)
        _close("pi", gpu["pi"][n], o["pi"], atol=1e-7)
        j = min([i for k, i, _ in ties if k in ("greedy", "top_p")], default=B)
        assert list(gpu["tokens"][n][:j].tolist()) == [int(x) for x in o["tokens"][:j]], \
            ("tokens", n, gpu["tokens"][n].tolist(), o["tokens"].tolist())
        jj = min(j + 1, B)
        _close("posterior", np.exp(gpu["logw"][n][:jj].double().numpy()),
               np.exp(o["logw"][:jj]), atol=1e-6)
        _close("q_tok", gpu["q_tok"][n][:j], o["q_tok"][:j])
        _close("p_tok", gpu["p_tok"][n][:j], o["p_tok"][:j])
        _close("accept_prob", gpu["accept_prob"][n][:j], o["accept_prob"][:j])
        _close("alpha", gpu["alpha"][n][:j], o["alpha"][:j], atol=1e-6)
        _close("lse_target", gpu["lse_target"][n], o["lse_target"], rtol=1e-5, atol=1e-4)
        if "collision" in gpu:
            _close("collision", gpu["collision"][n], o["collision"], atol=1e-7)
            _close("determinism", gpu["determinism"][n], o["determinism"], atol=1e-7)
        stats["positions"] += j
        if j == B:
            _close("exp_len", gpu["exp_len"][n], o["exp_len"], atol=1e-6)
            _close("alpha_len", gpu["alpha_len"][n], o["alpha_len"], atol=1e-6)
        if not ties:
            L = o["accepted"]
            assert int(gpu["accepted"][n]) == L, ("accepted", n, int(gpu["accepted"][n]), L)
            assert int(gpu["n_emitted"][n]) == o["n_emitted"], ("n_emitted", n)
            em = gpu["emitted"][n].tolist()
            assert em[:o["n_emitted"]] == o["emitted"], ("emitted", n, em, o["emitted"])
            assert all(x == -1 for x in em[o["n_emitted"]:])
            stats["emitted_checked"] += 1
    return stats
