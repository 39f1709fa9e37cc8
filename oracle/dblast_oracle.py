"""Plain fp64 CPU oracle for one DBLast draft+verify step.

TEST INFRASTRUCTURE ONLY.  It exists to check the CUDA path; nothing in the
product path imports it.  Only tests/, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may use it.  It shares no code with the CUDA
library (no kernels, headers, helpers, tables or pre/post-processing).

Everything is computed in float64 with numpy, in the direct form of the paper:
the branch hidden states h_{i,z} are materialised and pushed through the
vocabulary head, exactly as the definitions read; no blocking, fusion or
reordering is done beyond converting the vocabulary head to fp64 in row chunks
(a memory-management step of one matrix product).

Definitions followed (section / equation of the paper):

* Latent-mixture proposal q(x_{1:b}|y) = sum_z q(z|y) prod_i q_i(x_i|y,z)
  (Eq. 5, cp-drafter).
* Branch hidden states h_{i,z} = h_i + g_z(h_i) (Sec. 3.1, Architecture) with
  the reused vocabulary head giving q_i(.|y,z).  The expander is taken as
  rank r: g_z(h) = U_z (V_z^T h) + e_z.
* Category prior q_{Z_T}(z|y) = softmax(l(y)/Z_T) from a linear head on the
  block-anchor state (Sec. 3.1, "Drafter sampling during inference";
  Appendix A: Z_T = 0 selects the highest-prior category).
* Sampling: z-hat ~ q(z|y), then every position from q_i(.|y,z-hat) (Sec. 3.1,
  first paragraph of "Dependent Block Drafting and Verification").  Each draw
  is an inverse-CDF draw with one uniform (see ``inverse_cdf``).
* Category posterior (Eq. category-posterior) and the mixture next-token
  distribution (Eq. dep-next-token), which equal the prefix-marginal
  conditional of Eq. 1 / Eq. dep-conditional.
* Acceptance A_i = min(1, p/q) (Eq. 2), stop at the first rejection, residual
  draw from norm([p - q]_+), bonus token when the whole block is accepted
  (Algorithm 1; Appendix A, "Distributional correctness").
* Expected accepted length of the drafted block, sum_i prod_{j<=i} A_j
  (Eq. 3), and the overlap alpha_i = sum_v min(p_i(v), q(v|x_<i)).
* Training-side objectives, forward only (Sec. 3.2): block NLL (Eqs.
  independent-nll, dependent-nll) and the acceptance-oriented surrogate J_AL
  with r_l, S_l, l_tau (Eqs. acceptance-length-objective, subblock-objective)
  on given target blocks.
* Target sampling transform: temperature, top-k, top-p (Sec. 3.2, Sec. 4),
  applied to every target row before verification (filter_target).
* Target-block early determinism D_b and its M-sample estimator (App. B),
  for target rows that do not depend on the sampled prefix.
* Greedy-branch mode (Sec. 3.1, "Drafter sampling during inference"; App. A,
  "Greedy-Branch Proposal", "Prefix-Marginalized Conditional" and its
  verification algorithm): z-hat from the prior, the block is the greedy
  branch x-hat_{.,z-hat}, and verification uses the sparse conditional
  q_greedy over the consistent branches C_i.

Readings where the paper is silent (the same list is kept in the design notes):
the drafter's token distributions use the same temperature T as the target;
target rows are given inputs, independent of the drafted prefix; ties in
argmax go to the lowest index; an inverse-CDF draw takes the smallest index
whose cumulative mass exceeds u times the total; if a rejection leaves no
positive residual mass the replacement is drawn from p and flagged.
"""

import numpy as np

from .philox import (STREAM_ACCEPT, STREAM_DRAFT, STREAM_PRIOR,
                     STREAM_RESIDUAL, STREAM_TARGET, decision_uniform)

# decisions whose margin to the threshold is below this are "ties"
TIE_TOL = 1e-6


def f64(x):
    """Return x (torch tensor, numpy array or None) as a float64 numpy array."""
    if x is None:
        return None
    if hasattr(x, "detach"):
        import torch
        return x.detach().to(device="cpu", dtype=torch.float64).numpy()
    return np.asarray(x, dtype=np.float64)


def logsumexp(s, axis=-1):
    m = np.max(s, axis=axis, keepdims=True)
    m = np.where(np.isfinite(m), m, 0.0)
    with np.errstate(divide="ignore"):
        out = np.log(np.sum(np.exp(s - m), axis=axis, keepdims=True)) + m
    return np.squeeze(out, axis=axis)


def category_prior(Wp, bp, anchor, z_temperature):
    """Category logits l = Wp a (+ bp) and the prior pi = softmax(l / Z_T).

    Sec. 3.1 ("Drafter sampling during inference"): q_{Z_T}(z|y) =
    softmax(l_z(y)/Z_T).  Appendix A: for Z_T = 0 the highest-prior category is
    selected (one-hot; the lowest index on a tie).
    """
    ell = Wp @ anchor
    if bp is not None:
        ell = ell + bp
    if z_temperature == 0:
        pi = np.zeros_like(ell)
        pi[int(np.argmax(ell))] = 1.0
        return ell, pi
    s = ell / z_temperature
    e = np.exp(s - np.max(s))
    return ell, e / np.sum(e)


def inverse_cdf(weights, u):
    """One inverse-CDF draw from non-negative weights (not necessarily normalised).

    Returns (index, margin): index is the smallest v with
    sum_{v' <= v} w_{v'} > u * sum_v w_v; margin is the distance of u to the
    nearest edge of the chosen index's CDF interval, in normalised units.  If
    rounding leaves the target above every prefix sum, the last index with
    positive weight is returned with margin 0.
    """
    w = np.asarray(weights, dtype=np.float64)
    cum = np.cumsum(w)
    total = cum[-1]
    target = u * total
    idx = int(np.searchsorted(cum, target, side="right"))
    if idx >= w.shape[0]:
        nz = np.nonzero(w > 0)[0]
        return int(nz[-1]) if nz.size else w.shape[0] - 1, 0.0
    lo = cum[idx - 1] if idx > 0 else 0.0
    margin = min(target - lo, cum[idx] - target) / total
    return idx, margin


def branch_hidden(h, U, Vf, e):
    """h_{i,z} = h_i + U_z (V_z^T h_i) + e_z for every position i and branch z.

    Sec. 3.1 (Architecture): the category hidden expander maps h_i to K
    category-specific offsets g_z(h_i).  h: [B, H]; U, Vf: [K, H, r];
    e: [K, H] or None.  Returns [B, K, H].
    """
    B, H = h.shape
    K = U.shape[0]
    out = np.empty((B, K, H), dtype=np.float64)
    for z in range(K):
        code = h @ Vf[z]              # V_z^T h_i, [B, r]
        g = code @ U[z].T             # U_z code, [B, H]
        if e is not None:
            g = g + e[z]
        out[:, z, :] = h + g
    return out


def component_logits(W, hz, vbias, chunk=8192):
    """l_{i,z,v} = W_v . h_{i,z} (+ b_v): the reused vocabulary head on each branch.

    Sec. 3.1 (Architecture).  W is [V, H] (any dtype; converted to fp64 in row
    chunks), hz is [B, K, H].  Returns [B, K, V] in fp64.
    """
    B, K, H = hz.shape
    V = W.shape[0]
    flat = hz.reshape(B * K, H)
    out = np.empty((B * K, V), dtype=np.float64)
    for v0 in range(0, V, chunk):
        Wc = f64(W[v0:v0 + chunk])
        out[:, v0:v0 + Wc.shape[0]] = flat @ Wc.T
    if vbias is not None:
        out += vbias[None, :]
    return out.reshape(B, K, V)


def posterior(log_pi, logq_at_x):
    """Category posterior and its normaliser along the drafted prefix.

    Eq. category-posterior: q(z|y,x_<i) is proportional to
    q(z|y) prod_{j<i} q_j(x_j|y,z).  log_pi: [K]; logq_at_x: [B, K] with
    logq_at_x[j, z] = log q_j(x_j|y,z).  Returns log w: [B, K], normalised
    over z for every position i.
    """
    B, K = logq_at_x.shape
    logw = np.empty((B, K), dtype=np.float64)
    acc = np.array(log_pi, dtype=np.float64)
    for i in range(B):
        logw[i] = acc - logsumexp(acc)
        acc = acc + logq_at_x[i]
    return logw


def filter_target(t_row, T, top_k=0, top_p=0.0):
    """The target sampling transform: temperature, then top-k, then top-p.

    Sec. 3.2 / Sec. 4 (the target distribution after temperature, top-p and
    top-k; top-k 20 with top-p 0.8 or 0.95 in every evaluation).  Readings
    (the paper does not spell them out): top-k keeps the k largest logits,
    ties at the k-th value going to the lower token index, so exactly
    min(k, V) tokens stay (k = 0: off); top-p then orders the kept tokens by
    probability (the same order) and keeps each token whose preceding
    cumulative mass, renormalised over the top-k set, is below top_p (the
    smallest prefix reaching top_p; 0 or >= 1: off).  The result is
    renormalised over the kept set.  Returns (p' [V], kept token indices,
    margin of the top-p cut: the distance of top_p to the nearest cumulative
    mass that decides it, +inf when top-p is off).
    """
    t = f64(t_row)
    V = t.shape[0]
    st = t / T
    p = np.exp(st - logsumexp(st))
    order = np.lexsort((np.arange(V), -t))      # logit descending, index ascending
    kk = V if (top_k <= 0 or top_k >= V) else int(top_k)
    keep = order[:kk]
    margin = np.inf
    if 0.0 < top_p < 1.0:
        pk = p[keep] / np.sum(p[keep])
        before = np.concatenate([[0.0], np.cumsum(pk)[:-1]])
        n_keep = int(np.sum(before < top_p))
        margin = top_p - before[n_keep - 1]
        if n_keep < kk:
            margin = min(margin, before[n_keep] - top_p)
        keep = keep[:n_keep]
    out = np.zeros(V, dtype=np.float64)
    out[keep] = p[keep] / np.sum(p[keep])
    return out, keep, float(margin)


def target_distributions(target, T, top_k, top_p, ties, decisions=None):
    """p_i for every target row: softmax(t_i / T), filtered by top-k / top-p
    when either is on (filter_target); a top-p cut within TIE_TOL is recorded
    as a tie of kind "top_p" at row i, and every finite cut margin is listed
    in `decisions` when given.  Also returns the unfiltered natural
    log-sum-exp of t_i / T."""
    st = target / T
    lse_t = logsumexp(st, axis=-1)
    if top_k <= 0 and not (0.0 < top_p < 1.0):
        return np.exp(st - lse_t[:, None]), lse_t
    p = np.empty_like(st)
    for i in range(target.shape[0]):
        p[i], _, margin = filter_target(target[i], T, top_k, top_p)
        if decisions is not None and np.isfinite(margin):
            decisions.append(("top_p", i, margin))
        if margin < TIE_TOL:
            ties.append(("top_p", i, margin))
    return p, lse_t


def draft_and_verify_sequence(head, h, anchor, target, has_bonus, T, Z_T,
                              seed, n, pos, round_, top_k=0, top_p=0.0):
    """One draft+verify step for sequence n (all arrays fp64 numpy).

    head: dict with W [V,H] (any dtype), U, Vf [K,H,r], e [K,H]|None,
    Wp [K,H], bp [K]|None, vbias [V]|None.  h: [B,H]; anchor: [H]|None
    (None: h[0]); target: [B+has_bonus, V] target logits.
    """
    B, H = h.shape
    W = head["W"]
    a = h[0] if anchor is None else anchor
    ties = []
    decisions = []  # (kind, position, margin) of every decision taken

    # prior and latent category (Sec. 3.1; Appendix A)
    ell, pi = category_prior(head["Wp"], head["bp"], a, Z_T)
    u0 = decision_uniform(seed, STREAM_PRIOR, round_, n, pos)
    zhat, m0 = inverse_cdf(pi, u0)
    if Z_T != 0:
        decisions.append(("zhat", -1, m0))
        if m0 < TIE_TOL:
            ties.append(("zhat", -1, m0))
    with np.errstate(divide="ignore"):
        log_pi = np.log(pi)

    # branch distributions q_i(.|y,z) = softmax(l_{i,z}/T)
    hz = branch_hidden(h, head["U"], head["Vf"], head["e"])
    s = component_logits(W, hz, head["vbias"]) / T          # [B, K, V]
    lse = logsumexp(s, axis=-1)                               # [B, K]
    logq = s - lse[:, :, None]

    # draft block: every position from the z-hat branch
    tokens = np.empty(B, dtype=np.int64)
    for i in range(B):
        u1 = decision_uniform(seed, STREAM_DRAFT, round_, n, pos + i)
        tokens[i], m1 = inverse_cdf(np.exp(logq[i, zhat]), u1)
        decisions.append(("draft", i, m1))
        if m1 < TIE_TOL:
            ties.append(("draft", i, m1))

    # posterior weights and the mixture conditional q(.|y,x_<i)
    logq_at_x = logq[np.arange(B), :, tokens]                 # [B, K]
    logw = posterior(log_pi, logq_at_x)
    w = np.exp(logw)
    qmix = np.einsum("bk,bkv->bv", w, np.exp(logq))           # Eq. dep-next-token
    q_tok = qmix[np.arange(B), tokens]

    # target distributions p_i = softmax(t_i / T)
    p, lse_t = target_distributions(target, T, top_k, top_p, ties, decisions)  # [B+hb, V]
    p_tok = p[np.arange(B), tokens]

    alpha = np.sum(np.minimum(p[:B], qmix), axis=-1)
    ratio = p_tok / q_tok
    accept_prob = np.minimum(1.0, ratio)

    # sequential acceptance (Eq. 2; Algorithm 1)
    L = B
    for i in range(B):
        u2 = decision_uniform(seed, STREAM_ACCEPT, round_, n, pos + i)
        m2 = abs(u2 * q_tok[i] - p_tok[i]) / q_tok[i]
        decisions.append(("accept", i, m2))
        if m2 < TIE_TOL:
            ties.append(("accept", i, m2))
        if not (u2 < ratio[i]):
            L = i
            break

    emitted = list(int(x) for x in tokens[:L])
    extra = -1
    if L < B:
        # residual norm([p - q]_+) at the first rejected position
        u3 = decision_uniform(seed, STREAM_RESIDUAL, round_, n, pos + L)
        res = np.maximum(p[L] - qmix[L], 0.0)
        mass = float(np.sum(res))
        if mass > 0.0:
            extra, m3 = inverse_cdf(res, u3)
        else:
            extra, m3 = inverse_cdf(p[L], u3)
        decisions.append(("residual_mass", L, mass))
        decisions.append(("residual", L, m3))
        if mass < TIE_TOL:
            ties.append(("residual_mass", L, mass))
        if m3 < TIE_TOL:
            ties.append(("residual", L, m3))
    elif has_bonus:
        u3 = decision_uniform(seed, STREAM_RESIDUAL, round_, n, pos + B)
        extra, m3 = inverse_cdf(p[B], u3)
        decisions.append(("bonus", B, m3))
        if m3 < TIE_TOL:
            ties.append(("bonus", B, m3))
    if extra >= 0:
        emitted.append(int(extra))

    # Eq. 3 on the drafted block, and the same sum over the overlaps
    exp_len = float(np.sum(np.cumprod(accept_prob)))
    alpha_len = float(np.sum(np.cumprod(alpha)))

    first_tie = B + 1
    for kind, i, _ in ties:
        first_tie = min(first_tie, 0 if kind == "zhat" else i)

    return dict(pi=pi, ell=ell, zhat=int(zhat), tokens=tokens, lse=lse,
                logw=logw, q_tok=q_tok, p_tok=p_tok, accept_prob=accept_prob,
                alpha=alpha, accepted=L, emitted=emitted,
                n_emitted=len(emitted), exp_len=exp_len, alpha_len=alpha_len,
                lse_target=lse_t, ties=ties, decisions=decisions, first_tie=first_tie,
                collision=collision_probability(p[:B]),
                determinism=early_determinism_exact(p[:B]))


# ---------------------------------------------- training-side objectives (forward)
def block_nll(log_pi, logq_at_x):
    """Block negative log-likelihood of a target block under the proposal.

    Eq. dependent-nll: -log sum_z q(z|y) prod_i q_i(x*_i|y,z); with K = 1 it
    is Eq. independent-nll, -sum_i log q_i(x*_i|y).  log_pi: [K];
    logq_at_x: [b, K] with logq_at_x[i, z] = log q_i(x*_i|y,z).
    """
    with np.errstate(invalid="ignore"):
        return float(-logsumexp(log_pi + np.sum(logq_at_x, axis=0)))


def al_surrogate(q_cond, p_tok, tau):
    """The acceptance-oriented surrogate of one target block (Sec. 3.2).

    q_cond[i] = q(x*_i|y,x*_<i) (the proposal conditional, Eq.
    dep-next-token), p_tok[i] = p(x*_i|y,x*_<i).  A_j = min(1, p/q) (Eq. 2),
    r_l = q(x*_{1:l}|y) / p(x*_{1:l}|y) = prod_{j<=l} q_j / p_j (the prefix
    importance ratio), S_l = sum_{i<=l} prod_{j<=i} A_j, l_tau = the first l
    with r_l < tau (b if none), and J = sum_{l <= l_tau} (log r_l + log S_l)
    (Eq. subblock-objective for one sampled block; the loss is -J, Eq.
    training-loss).  Returns dict(A, r, S, l_tau (1-based), J, margin: the
    relative distance of the decisive r_l to tau).
    """
    q = np.asarray(q_cond, dtype=np.float64)
    p = np.asarray(p_tok, dtype=np.float64)
    b = q.shape[0]
    with np.errstate(divide="ignore"):
        A = np.minimum(1.0, p / q)
        r = np.cumprod(q / p)
    S = np.cumsum(np.cumprod(A))
    below = np.nonzero(r < tau)[0]
    l_tau = int(below[0]) + 1 if below.size else b
    with np.errstate(divide="ignore"):
        J = float(np.sum(np.log(r[:l_tau]) + np.log(S[:l_tau])))
    margin = float(np.min(np.abs(r[:l_tau] - tau)) / tau) if tau > 0 else np.inf
    return dict(A=A, r=r, S=S, l_tau=l_tau, J=J, margin=margin)


def al_objective_sequence(head, h, anchor, target, tokens, T, Z_T, tau,
                          top_k=0, top_p=0.0):
    """Forward pass of the training objectives on one given target block.

    tokens: the target block x*_{1:b} (sampled from the target); target:
    [b (+1), V] target logits whose first b rows give p_i.  The proposal is
    the soft latent mixture (Eq. 5) with the category prior at Z_T; its
    conditionals along x* are Eqs. category-posterior and dep-next-token.
    p is the target after the same filter as verification
    (target_distributions).  Returns block NLL (Eq. dependent-nll), the AL
    surrogate terms (al_surrogate), q_cond, p_tok and the ties of the
    top-p cuts and of the l_tau decision (kind "tau", within TIE_TOL).
    """
    b = len(tokens)
    a = h[0] if anchor is None else anchor
    ties = []
    _, pi = category_prior(head["Wp"], head["bp"], a, Z_T)
    with np.errstate(divide="ignore"):
        log_pi = np.log(pi)
    hz = branch_hidden(h, head["U"], head["Vf"], head["e"])
    s = component_logits(head["W"], hz, head["vbias"]) / T
    logq = s - logsumexp(s, axis=-1)[:, :, None]
    x = np.asarray(tokens, dtype=np.int64)
    logq_at_x = logq[np.arange(b), :, x]                        # [b, K]
    logw = posterior(log_pi, logq_at_x)
    q_cond = np.sum(np.exp(logw + logq_at_x), axis=-1)
    p, _ = target_distributions(target[:b], T, top_k, top_p, ties)
    p_tok = p[np.arange(b), x]
    al = al_surrogate(q_cond, p_tok, tau)
    if al["margin"] < TIE_TOL:
        ties.append(("tau", al["l_tau"] - 1, al["margin"]))
    return dict(nll=block_nll(log_pi, logq_at_x), q_cond=q_cond, p_tok=p_tok,
                ties=ties, **al)


# --------------------------------------------------------- greedy-branch mode
# Decisions whose top-two logit gap is below this are "ties" of the greedy
# argmax: the CUDA path forms the logits in fp32 (errors up to ~1e-5 at the
# Qwen3 shapes), so only gaps below 1e-4 may resolve differently.
GREEDY_TIE_TOL = 1e-4


def greedy_branch_tokens(logits):
    """x-hat_{i,z} = argmax_v q_i(v|y,z) for every position and branch.

    Sec. 3.1 ("Drafter sampling during inference"), Eq. greedy-branch-proposal:
    the greedy token of branch z at position i.  The argmax of q_i(.|y,z) =
    softmax(l_{i,z}/T) is the argmax of the logits l_{i,z} for any T > 0; ties
    go to the lowest index.  logits: [B, K, V].  Returns (xhat [B, K] int64,
    gap [B, K]: the largest logit minus the second largest, +inf if V = 1).
    """
    xhat = np.argmax(logits, axis=-1)
    if logits.shape[-1] < 2:
        return xhat, np.full(xhat.shape, np.inf)
    top2 = np.sort(logits, axis=-1)[..., -2:]
    return xhat, top2[..., 1] - top2[..., 0]


def consistent_branches(xhat, tokens):
    """Membership of the consistent-branch sets C_i(x_<i).

    App. A ("Prefix-Marginalized Conditional"): C_i = {z : x-hat_{j,z} = x_j
    for every j < i}.  xhat: [B, K]; tokens: [B].  Returns bool [B, K] with
    row i marking C_i (row 0 is every branch).
    """
    B, K = xhat.shape
    C = np.ones((B, K), dtype=bool)
    for i in range(1, B):
        C[i] = C[i - 1] & (xhat[i - 1] == tokens[i - 1])
    return C


def greedy_conditional(pi, xhat, C, V):
    """The sparse proposal conditional q_greedy(v|y,x_<i) at every position.

    App. A: pi-tilde_{i,z} = pi_z 1{z in C_i} / sum_{z' in C_i} pi_{z'} and
    q_greedy(v|y,x_<i) = sum_{z in C_i} pi-tilde_{i,z} 1{v = x-hat_{i,z}}
    (Eq. appendix-greedy-conditional).  pi: [K]; xhat, C: [B, K].  Returns
    (q [B, V] dense, with at most K non-zero entries per row; pit [B, K]).
    A prefix that no branch drafts (zero proposal mass) gets all-zero rows.
    """
    B, K = xhat.shape
    q = np.zeros((B, V), dtype=np.float64)
    pit = np.zeros((B, K), dtype=np.float64)
    for i in range(B):
        wz = np.where(C[i], pi, 0.0)
        tot = np.sum(wz)
        if not tot > 0.0:
            continue
        pit[i] = wz / tot
        for z in range(K):
            if C[i, z]:
                q[i, xhat[i, z]] += pit[i, z]
    return q, pit


def greedy_draft_and_verify_sequence(head, h, anchor, target, has_bonus, T, Z_T,
                                     seed, n, pos, round_, top_k=0, top_p=0.0):
    """One greedy-branch draft+verify step for sequence n (Algorithm 1 of App. A).

    Same inputs and outputs as draft_and_verify_sequence.  The category is
    drawn from the tempered prior as in the stochastic mode; the block is the
    greedy branch x_i = x-hat_{i,z-hat}; verification uses q_greedy (App. A)
    for the acceptance min(1, p/q) and the residual [p - q_greedy]_+, then the
    usual bonus token.  Extra outputs: xhat [B, K] (all K greedy branches),
    consistent [B, K] (C_i), gap [B, K] (top-two logit gaps).  "logw" holds
    log pi-tilde (the category posterior given the greedy prefix, -inf
    outside C_i).  A greedy argmax of a branch in C_i whose gap is below
    GREEDY_TIE_TOL is recorded as a tie of kind "greedy".
    """
    B, H = h.shape
    W = head["W"]
    V = W.shape[0]
    a = h[0] if anchor is None else anchor
    ties = []
    decisions = []  # (kind, position, margin) of every decision taken

    # prior and latent category, as in the stochastic mode
    ell, pi = category_prior(head["Wp"], head["bp"], a, Z_T)
    u0 = decision_uniform(seed, STREAM_PRIOR, round_, n, pos)
    zhat, m0 = inverse_cdf(pi, u0)
    if Z_T != 0:
        decisions.append(("zhat", -1, m0))
        if m0 < TIE_TOL:
            ties.append(("zhat", -1, m0))

    # all K greedy branches and the selected block
    hz = branch_hidden(h, head["U"], head["Vf"], head["e"])
    logits = component_logits(W, hz, head["vbias"])          # [B, K, V]
    xhat, gap = greedy_branch_tokens(logits)
    tokens = xhat[:, zhat].astype(np.int64)
    C = consistent_branches(xhat, tokens)
    for i in range(B):
        for z in range(xhat.shape[1]):
            if C[i, z]:
                decisions.append(("greedy", i, float(gap[i, z])))
                if gap[i, z] < GREEDY_TIE_TOL:
                    ties.append(("greedy", i, float(gap[i, z])))

    # the proposal conditional used by verification
    q, pit = greedy_conditional(pi, xhat, C, V)
    q_tok = q[np.arange(B), tokens]
    with np.errstate(divide="ignore"):
        logw = np.log(pit)

    # target distributions p_i = softmax(t_i / T)
    p, lse_t = target_distributions(target, T, top_k, top_p, ties, decisions)
    p_tok = p[np.arange(B), tokens]
    alpha = np.sum(np.minimum(p[:B], q), axis=-1)
    ratio = p_tok / q_tok
    accept_prob = np.minimum(1.0, ratio)

    L = B
    for i in range(B):
        u2 = decision_uniform(seed, STREAM_ACCEPT, round_, n, pos + i)
        m2 = abs(u2 * q_tok[i] - p_tok[i]) / q_tok[i]
        decisions.append(("accept", i, m2))
        if m2 < TIE_TOL:
            ties.append(("accept", i, m2))
        if not (u2 < ratio[i]):
            L = i
            break

    emitted = list(int(x) for x in tokens[:L])
    extra = -1
    if L < B:
        u3 = decision_uniform(seed, STREAM_RESIDUAL, round_, n, pos + L)
        res = np.maximum(p[L] - q[L], 0.0)
        mass = float(np.sum(res))
        if mass > 0.0:
            extra, m3 = inverse_cdf(res, u3)
        else:
            extra, m3 = inverse_cdf(p[L], u3)
        decisions.append(("residual_mass", L, mass))
        decisions.append(("residual", L, m3))
        if mass < TIE_TOL:
            ties.append(("residual_mass", L, mass))
        if m3 < TIE_TOL:
            ties.append(("residual", L, m3))
    elif has_bonus:
        u3 = decision_uniform(seed, STREAM_RESIDUAL, round_, n, pos + B)
        extra, m3 = inverse_cdf(p[B], u3)
        decisions.append(("bonus", B, m3))
        if m3 < TIE_TOL:
            ties.append(("bonus", B, m3))
    if extra >= 0:
        emitted.append(int(extra))

    exp_len = float(np.sum(np.cumprod(accept_prob)))
    alpha_len = float(np.sum(np.cumprod(alpha)))

    first_tie = B + 1
    for kind, i, _ in ties:
        first_tie = min(first_tie, 0 if kind == "zhat" else i)

    return dict(pi=pi, ell=ell, zhat=int(zhat), tokens=tokens, xhat=xhat,
                consistent=C, gap=gap, logw=logw, q_tok=q_tok, p_tok=p_tok,
                accept_prob=accept_prob, alpha=alpha, accepted=L,
                emitted=emitted, n_emitted=len(emitted), exp_len=exp_len,
                alpha_len=alpha_len, lse_target=lse_t, ties=ties, decisions=decisions,
                first_tie=first_tie, collision=collision_probability(p[:B]),
                determinism=early_determinism_exact(p[:B]))


# ------------------------------------------------- target-block early determinism
def target_probs(target_rows, T):
    """p_i = softmax(t_i / T) of each target row, fp64.  target_rows: [R, V]."""
    st = f64(target_rows) / T
    return np.exp(st - logsumexp(st, axis=-1)[:, None])


def collision_probability(p):
    """sum_v p(v)^2 of each row: the probability that two independent draws
    from p collide, i.e. E_{X ~ p}[p(X)] (App. B)."""
    return np.sum(p * p, axis=-1)


def early_determinism_exact(p_rows):
    """Target-block early determinism D_b(y) (App. B, Eq.
    appendix-early-determinism) for b = len(p_rows) target rows that do not
    depend on the sampled prefix (the synthetic targets here).

    D_b = E_{x ~ p}[(1/b) sum_j prod_{i<=j} p_i(x_i)].  With independent
    positions the expectation of each product is the product of the
    per-position collision probabilities, so
    D_b = (1/b) sum_j prod_{i<=j} sum_v p_i(v)^2.  p_rows: [b, V].
    """
    c = collision_probability(p_rows)
    return float(np.mean(np.cumprod(c)))


def early_determinism_estimate(p_rows, M, seed, n):
    """The M-sample estimator of App. B (Eq.
    appendix-early-determinism-estimator):
    D-hat_b = 1/(M b) sum_m sum_j prod_{i<=j} p_i(x_i^(m)),
    with M blocks x^(m) drawn from the target.  For prefix-independent rows
    x_i^(m) ~ p_i, each an inverse-CDF draw with the stream-4 uniform (round
    field = m, sequence n, position i).  Returns (D-hat, samples [M, b],
    ties: (m, i, margin) for draws within TIE_TOL of an edge).
    """
    b = p_rows.shape[0]
    samples = np.empty((M, b), dtype=np.int64)
    ties = []
    tot = 0.0
    for m in range(M):
        prod = 1.0
        for i in range(b):
            u = decision_uniform(seed, STREAM_TARGET, m, n, i)
            x, margin = inverse_cdf(p_rows[i], u)
            if margin < TIE_TOL:
                ties.append((m, i, margin))
            samples[m, i] = x
            prod *= p_rows[i, x]
            tot += prod
    return tot / (M * b), samples, ties


def prepare_head(head):
    """fp64 copies of the small head tensors; W is left as given (chunked later)."""
    out = {k: f64(head.get(k)) for k in ("U", "Vf", "e", "Wp", "bp", "vbias")}
    out["W"] = head["W"]
    return out


def draft_and_verify(head, hidden, anchor, target, has_bonus, T, Z_T, seed,
                     pos, round_, seqs=None, mode="soft", top_k=0, top_p=0.0):
    """Run the step for the sequences in ``seqs`` (default: all).

    hidden: [N, B, H]; anchor: [N, H] or None; target: [N, B+has_bonus, V];
    pos: [N] int; round_: [N] int; mode "soft" (tokens drawn from the branch
    distributions) or "greedy" (greedy branches, App. A); top_k / top_p: the
    target filter of filter_target (0: off).  Returns a list of
    per-sequence dicts (see draft_and_verify_sequence and
    greedy_draft_and_verify_sequence) in the order of ``seqs``.
    """
    step = {"soft": draft_and_verify_sequence,
            "greedy": greedy_draft_and_verify_sequence}[mode]
    hd = prepare_head(head)
    N = hidden.shape[0]
    seqs = range(N) if seqs is None else seqs
    out = []
    for n in seqs:
        h = f64(hidden[n])
        a = None if anchor is None else f64(anchor[n])
        t = f64(target[n])
        out.append(step(
            hd, h, a, t, bool(has_bonus), float(T), float(Z_T), int(seed),
            int(n), int(pos[n]), int(round_[n]), int(top_k), float(top_p)))
    return out


def expander_parameter_count(H, K, rank=None):
    """Parameters added by the category expander and the prior head.

    Table 1 (full-rank expander, one linear layer with bias per category, plus
    a linear prior head with bias): K H^2 + 2 K H + K.  With a rank-r expander
    U_z V_z^T + e_z the first term becomes 2 K H r.
    """
    expander = K * H * H if rank is None else 2 * K * H * rank
    return expander + K * H + (K * H + K)
