"""Parity harness: run the CUDA step and the fp64 oracle on the same seeded
inputs and compare them with the agreed rules.

Integer outputs (latent category, draft tokens, accepted length, emitted
tokens) are followed decision by decision along the oracle's path.  A
decision the GPU takes the other way must lie within its band of the
threshold: the tie tolerance (1e-6; 1e-4 on the logit gap of a greedy argmax)
plus the precision allowance of the kernels' arithmetic (NEAR_DRAW of
probability mass for an inverse-CDF draw, NEAR_ACCEPT relative for the
acceptance ratio).  The allowances come from the measured error of fp32
tensor-core accumulation over H bf16 products: vocabulary-head logits within
3.8e-5 of the exact ones at H = 4096, draw CDFs within 1.1e-5.  After such a
flip the decisions that depend on it are not compared; every other one is
exact.  Probabilities, overlaps, log-sum-exps and expected lengths must agree
within RTOL relative (plus a tiny absolute floor for values near 0).

The GPU's own tie report (`tie_flags`: per decision kind a tie bit, and the
same bit shifted by NEAR_SHIFT for "near", i.e. within the band) is checked
against the oracle's margins in both directions (check_tie_flags).

Every compare call also requires that its sequences were not skipped
wholesale: the accepted length and emitted tokens of at least three quarters
of them (and at least one) are compared exactly.
"""
import numpy as np
import torch

from oracle import dblast_oracle as orc

RTOL = 1e-4
ATOL_PROB = 1e-7

# tie_flags bits of include/dblast.h, by oracle decision kind; the near bit
# of a kind is its tie bit shifted left by NEAR_SHIFT
TIE_BITS = {"zhat": 1, "draft": 2, "greedy": 2, "accept": 4, "residual": 8, "bonus": 8,
            "residual_mass": 16, "top_p": 32}
NEAR_SHIFT = 8
# the kernels' precision allowances (the library's documented values): a draw
# may move by NEAR_DRAW of probability mass, an acceptance ratio by
# NEAR_ACCEPT relative
NEAR_DRAW = 5e-5
NEAR_ACCEPT = 1e-4
# minimum share of the sequences of one compare call whose accepted length and
# emitted tokens are compared exactly
MIN_CHECKED = 0.75


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


def run_gpu_split(head_t, blk, T, Z_T, seed, pos, rnd, impl="auto", head=None, ws=None,
                  mode="soft", top_k=0, top_p=0.0):
    """The same step through the two boundary calls: dblast_draft_block, then
    dblast_verify_block on the draft it left in the workspace."""
    from paper_2608_05448_gb300 import Head, Workspace, dblast_draft_block, dblast_verify_block
    head = head or Head.from_dict(head_t)
    N, B, _ = blk["hidden"].shape
    ws = ws or Workspace(head, N, B, blk["has_bonus"])
    dout = dblast_draft_block(head, ws, blk["hidden"], pos, rnd, T, Z_T, seed,
                              anchor=blk.get("anchor"), impl=impl, mode=mode)
    vout = dblast_verify_block(head, ws, blk["hidden"], pos, rnd, T, Z_T, seed, blk["target"],
                               blk["has_bonus"], anchor=blk.get("anchor"), impl=impl,
                               mode=mode, top_k=top_k, top_p=top_p)
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


# ------------------------------------------------------------ decisions
def _tol(kind):
    return orc.GREEDY_TIE_TOL if kind == "greedy" else orc.TIE_TOL


def _decision(o, kind, i):
    for d in o["decisions"]:
        if d[0] == kind and d[1] == i:
            return d
    return None


def _near_tol(d, o):
    """The band within which the kernels may take decision d the other way:
    its tie tolerance plus the precision allowance of the arithmetic behind it
    (NEAR_DRAW of probability mass for a draw, NEAR_ACCEPT relative for the
    acceptance ratio; the target filter and the greedy gap need none)."""
    kind, i, _ = d
    if kind == "greedy":
        return orc.GREEDY_TIE_TOL
    if kind == "top_p":
        return orc.TIE_TOL
    if kind == "accept":
        return orc.TIE_TOL + NEAR_ACCEPT
    if kind == "residual":  # margin in units of the residual mass R
        r = _decision(o, "residual_mass", i)
        R = r[2] if r is not None else 0.0
        return orc.TIE_TOL + NEAR_DRAW / R if R > 0.0 else np.inf
    return orc.TIE_TOL + NEAR_DRAW


def _is_tie(d):
    return d is not None and d[2] < _tol(d[0])


def _is_near(d, o):
    return d is not None and d[2] < _near_tol(d, o)


def _prereq(e, d):
    """True when decision e is taken before decision d and can change it (or
    whether d is taken at all).  Decisions are (kind, position, margin)."""
    ke, ie, _ = e
    kd, idd, _ = d
    if e is d or kd in ("zhat", "top_p"):
        return False  # the latent draw and the target filter depend on inputs only
    if ke == "zhat":
        return True
    if kd == "draft":
        return False  # soft draft tokens depend on z-hat alone
    if kd == "greedy":
        return ke == "greedy" and ie < idd  # C_i is fixed by the earlier greedy tokens
    # accept / residual_mass / residual / bonus at position idd
    if ke in ("draft", "greedy", "top_p"):
        return ie <= idd
    if ke == "accept":
        return ie < idd if kd == "accept" else True
    if ke == "residual_mass":
        return kd == "residual"
    return False


def _flip(d, o, n, stats, what):
    """The GPU took decision d the other way: allowed only inside its band."""
    assert _is_near(d, o), (what, n, d)
    stats["diverged"] += 1
    if not _is_tie(d):
        stats["precision_flips"] += 1


def check_tie_flags(flags, o, n, flipped=()):
    """The GPU's tie report of one sequence against the oracle's margins.

    Low byte: the decision was within TIE_TOL of its threshold by the
    kernel's own arithmetic; next byte ("near"): within TIE_TOL plus the
    kernel's precision allowance.  A tie bit implies its near bit.  Every
    oracle tie (on the path the GPU followed) must have its near bit set;
    with no decision taken the other way, a near bit must be clear when every
    decision of its kind is more than ten bands from its threshold, and a tie
    bit when every one is more than two bands away."""
    decs = o["decisions"]
    flags = int(flags)
    tie, near = flags & 0xFF, (flags >> NEAR_SHIFT) & 0xFF
    assert tie & ~near == 0, ("tie bit without its near bit", n, flags)
    for d in decs:
        if _is_tie(d) and not any(_prereq(e, d) for e in flipped):
            assert near & TIE_BITS[d[0]], ("tie flag not set", n, d, flags)
    if flipped:
        return
    for bit in sorted(set(TIE_BITS.values())):
        ds = [d for d in decs if TIE_BITS[d[0]] == bit]
        if all(d[2] > 10.0 * _near_tol(d, o) for d in ds):
            assert not near & bit, ("tie flag set without a near decision", n, bit, flags,
                                    [d for d in decs if d[2] < 1e-3])
        if all(d[2] > 2.0 * _near_tol(d, o) for d in ds):
            assert not tie & bit, ("tie flag set without a near decision", n, bit, flags,
                                   [d for d in decs if d[2] < 1e-3])


def _check_path(gpu, o, n, lim, stats, flipped):
    """Follow the decisions after the draft: acceptance, then the residual or
    bonus token.  lim: the first position whose acceptance test may run on
    another path (a draft or filter decision went the other way; B + 1 when
    none, and B when only the bonus row's filter cut differs).  Where the GPU
    and the oracle take a decision differently, it must lie in its band, and
    the comparison of everything after it stops there.  Returns True when the
    accepted length and the emitted tokens were compared in full."""
    B = len(o["tokens"])
    Lo, Lg = o["accepted"], int(gpu["accepted"][n])
    for i in range(B + 1):
        if i >= lim:
            return False  # the acceptance test at i runs on another path
        if i == B:
            break  # every draft accepted by both
        acc_o, acc_g = i < Lo, i < Lg
        if acc_o != acc_g:
            d = _decision(o, "accept", i)
            _flip(d, o, n, stats, "accepted")
            flipped.append(d)
            return False
        if not acc_o:
            break  # both reject at i
    assert Lg == Lo, ("accepted", n, Lg, Lo)
    em = gpu["emitted"][n].tolist()
    ne = int(gpu["n_emitted"][n])
    assert ne == o["n_emitted"], ("n_emitted", n, ne, o["n_emitted"])
    assert em[:Lo] == o["emitted"][:Lo], ("emitted", n, em, o["emitted"])
    assert all(x == -1 for x in em[ne:]), ("emitted padding", n, em)
    if ne > Lo and em[Lo] != o["emitted"][Lo]:  # the residual or bonus token
        kinds = ("residual", "residual_mass") if Lo < B else ("bonus",)
        ds = [_decision(o, k, Lo) for k in kinds]
        d = next((x for x in ds if _is_near(x, o)), ds[0])
        _flip(d, o, n, stats, "emitted")
        flipped.append(d)
        return False
    stats["emitted_checked"] += 1
    return True


def _filter_lim(o, B):
    """First row whose filtered target p may differ (a tied top-p cut)."""
    return min([d[1] for d in o["decisions"] if d[0] == "top_p" and _is_tie(d)], default=B + 1)


def _check_common(gpu, o, n, j, stats):
    """Floats along the checked prefix [0, j) of sequence n."""
    B = len(o["tokens"])
    jj = min(j + 1, B)
    _close("posterior", np.exp(gpu["logw"][n][:jj].double().numpy()),
           np.exp(o["logw"][:jj]), atol=1e-6)
    _close("q_tok", gpu["q_tok"][n][:j], o["q_tok"][:j])
    _close("p_tok", gpu["p_tok"][n][:j], o["p_tok"][:j])
    _close("accept_prob", gpu["accept_prob"][n][:j], o["accept_prob"][:j])
    _close("lse_target", gpu["lse_target"][n], o["lse_target"], rtol=1e-5, atol=1e-4)
    if "collision" in gpu:
        _close("collision", gpu["collision"][n], o["collision"], atol=1e-7)
        _close("determinism", gpu["determinism"][n], o["determinism"], atol=1e-7)
    stats["positions"] += j
    if j == B:
        _close("exp_len", gpu["exp_len"][n], o["exp_len"], atol=1e-6)
        _close("alpha_len", gpu["alpha_len"][n], o["alpha_len"], atol=1e-6)


def _finish(stats, start, nseq):
    checked = stats["emitted_checked"] - start
    need = max(1, int(MIN_CHECKED * nseq))
    assert checked >= need, ("too few sequences compared exactly", checked, nseq, stats)
    return stats


_KEYS = ("sequences", "tie_sequences", "positions", "emitted_checked", "tie_flags",
         "near_flags", "diverged", "precision_flips")


def _count_flags(gpu, o, n, stats):
    stats["sequences"] += 1
    if o["ties"]:
        stats["tie_sequences"] += 1
    f = int(gpu["tie_flags"][n])
    stats["tie_flags"] += int(f & 0xFF != 0)
    stats["near_flags"] += int(f != 0)


def compare(gpu, orc_list, seqs, stats=None):
    """Compare GPU outputs (dict of CPU tensors) with oracle dicts for `seqs`."""
    stats = stats if stats is not None else {}
    for key in _KEYS:
        stats.setdefault(key, 0)
    start = stats["emitted_checked"]
    for o, n in zip(orc_list, seqs):
        _count_flags(gpu, o, n, stats)
        B = len(o["tokens"])
        flipped = []
        _close("lse", gpu["lse"][n], o["lse"], rtol=1e-5, atol=1e-4)
        _close("lse_target", gpu["lse_target"][n], o["lse_target"], rtol=1e-5, atol=1e-4)
        if int(gpu["z_hat"][n]) != o["zhat"]:
            d = _decision(o, "zhat", -1)
            _flip(d, o, n, stats, "z_hat")
            check_tie_flags(gpu["tie_flags"][n], o, n, [d])
            continue
        _close("pi", gpu["pi"][n], o["pi"], atol=1e-7)
        # draft tokens depend on z-hat alone: each one is exact unless it
        # lies in its band
        j = B + 1  # first position on another path (B + 1: none)
        for i in range(B):
            if int(gpu["tokens"][n][i]) != int(o["tokens"][i]):
                d = _decision(o, "draft", i)
                assert _is_near(d, o), \
                    ("tokens", n, i, d, gpu["tokens"][n].tolist(), o["tokens"].tolist())
                if j > B:
                    _flip(d, o, n, stats, "tokens")
                flipped.append(d)
                j = min(j, i)
        lim = min(j, _filter_lim(o, B))
        _check_common(gpu, o, n, min(lim, B), stats)
        _close("alpha", gpu["alpha"][n][:min(lim + 1, B)], o["alpha"][:min(lim + 1, B)],
               atol=1e-6)
        _check_path(gpu, o, n, lim, stats, flipped)
        check_tie_flags(gpu["tie_flags"][n], o, n, flipped)
    return _finish(stats, start, len(seqs))


def compare_greedy(gpu, orc_list, seqs, stats=None):
    """Greedy-branch mode: as compare().  Every branch token whose top-two
    logit gap is clear of the tie band must be exact; a branch token that
    differs at a tie (gap below GREEDY_TIE_TOL) for a branch in C_i ends the
    comparison of what depends on it (C_j for j > i, q_greedy from i on)."""
    stats = stats if stats is not None else {}
    for key in _KEYS + ("branch_tokens",):
        stats.setdefault(key, 0)
    start = stats["emitted_checked"]
    for o, n in zip(orc_list, seqs):
        _count_flags(gpu, o, n, stats)
        B, K = o["xhat"].shape
        flipped = []
        clear = o["gap"] >= orc.GREEDY_TIE_TOL
        bt = gpu["branch_tokens"][n].numpy()
        assert (bt[clear] == o["xhat"][clear]).all(), ("branch_tokens", n)
        stats["branch_tokens"] += int(clear.sum())
        _close("lse_target", gpu["lse_target"][n], o["lse_target"], rtol=1e-5, atol=1e-4)
        if int(gpu["z_hat"][n]) != o["zhat"]:
            d = _decision(o, "zhat", -1)
            _flip(d, o, n, stats, "z_hat")
            check_tie_flags(gpu["tie_flags"][n], o, n, [d])
            continue
        _close("pi", gpu["pi"][n], o["pi"], atol=1e-7)
        # the first position where a branch of C_i took another greedy token
        # (only at a tie: the clear ones were checked above)
        C = o["consistent"]
        diff = (bt != o["xhat"]) & C
        j = int(np.argmax(diff.any(axis=1))) if diff.any() else B + 1
        if j <= B:
            d = ("greedy", j, float(np.min(np.where(diff[j], o["gap"][j], np.inf))))
            _flip(d, o, n, stats, "branch_tokens")
            flipped.append(d)
        jt = min(j, B)
        assert list(gpu["tokens"][n][:jt].tolist()) == [int(x) for x in o["tokens"][:jt]], \
            ("tokens", n, gpu["tokens"][n].tolist(), o["tokens"].tolist())
        lim = min(j, _filter_lim(o, B))
        _check_common(gpu, o, n, min(lim, B), stats)
        _close("alpha", gpu["alpha"][n][:min(lim, B)], o["alpha"][:min(lim, B)], atol=1e-6)
        _check_path(gpu, o, n, lim, stats, flipped)
        check_tie_flags(gpu["tie_flags"][n], o, n, flipped)
    return _finish(stats, start, len(seqs))
