"""Seeded synthetic inputs for the DBLast draft+verify step.

This module only draws random tensors with the shapes, scales and structure of
the paper's workloads (Qwen3-4B / Qwen3-8B heads, block length around 15-16,
K mixture components, temperatures 0.6-1.5).  It is shared by the tests, the
bench and the oracle checks; it holds none of the step's own arithmetic
(sampling, posterior, verification).  The one derived input is the target
logits, which follow the stated recipe "the drafter's K-mixture logits plus
Gaussian noise": they are built here with plain torch ops in fp32 from the
generated head, and both the CUDA path and the oracle receive them as given.

No benchmark items, prompts or checkpoints are reproduced: the paper's
datasets (GSM8K, MT-Bench, HumanEval, creative writing) and trained weights
are not available, and these random inputs stand in for them.
"""

import math

import torch

QWEN_V = 151936

# name -> shape / generator parameters.  "vscale" is the std of V_z entries:
# "1/r" follows the tiny case literally (low-rank factors N(0, 1/r)); "1/H"
# gives unit-variance codes V_z^T h so the branch offset is as large as h.
CONFIGS = {
    "tiny": dict(V=64, H=32, B=3, K=2, r=2, N=8, T=1.0, Z_T=1.0, sigma=0.5,
                 zipf=None, vscale="1/r", dtype="f32", bonus=True, seed=0,
                 expander_bias=False),
    "qwen3_4b_b1": dict(V=QWEN_V, H=2560, B=16, K=8, r=16, N=1, T=1.0,
                        Z_T=1.0, sigma=1.0, zipf=1.1, vscale="1/H",
                        dtype="bf16", bonus=True, seed=1,
                        expander_bias=False),
    "qwen3_8b_b32": dict(V=QWEN_V, H=4096, B=16, K=8, r=16, N=32, T=1.0,
                         Z_T=1.0, sigma=0.7, zipf=1.1, vscale="1/H",
                         dtype="bf16", bonus=True, seed=2,
                         expander_bias=False),
    "sweep_k16": dict(V=QWEN_V, H=4096, B=16, K=16, r=32, N=64, T=1.0,
                      Z_T=1.0, sigma=0.3, zipf=1.1, vscale="1/H",
                      dtype="bf16", bonus=True, seed=3, expander_bias=False),
    "serve_b8": dict(V=QWEN_V, H=4096, B=8, K=8, r=16, N=256, T=1.0, Z_T=1.0,
                     sigma=0.7, zipf=1.1, vscale="1/H", dtype="bf16",
                     bonus=True, seed=4, expander_bias=False),
    "serve_b32": dict(V=QWEN_V, H=4096, B=32, K=8, r=16, N=256, T=1.0,
                      Z_T=1.0, sigma=0.7, zipf=1.1, vscale="1/H",
                      dtype="bf16", bonus=True, seed=5, expander_bias=False),
}


def config(name, **over):
    cfg = dict(CONFIGS[name])
    cfg.update(over)
    cfg["name"] = name
    return cfg


def _gen(seed, sub, device):
    g = torch.Generator(device=device)
    g.manual_seed((int(seed) * 1000003 + int(sub)) & ((1 << 63) - 1))
    return g


def _randn(shape, std, seed, sub, device):
    g = _gen(seed, sub, device)
    return torch.randn(shape, generator=g, device=device,
                       dtype=torch.float32) * std


def storage_dtype(cfg):
    return torch.float32 if cfg["dtype"] == "f32" else torch.bfloat16


def make_head(cfg, device="cpu"):
    """Vocabulary head, rank-r expander, prior head and vocabulary bias.

    W ~ N(0, 0.02^2) [V, H]; U_z ~ N(0, 1/r) [K, H, r]; V_z ~ N(0, vscale)
    [K, H, r]; prior head Wp ~ N(0, 1/(r H)) so that the category logits
    W_p a are N(0, 1/r) for a ~ N(0, 1); bp = 0.  Zipf-shaped vocabulary bias
    b_v = -s ln(1 + rank(v)) over a seeded permutation when cfg["zipf"] = s.
    Optional expander bias e_z ~ N(0, 1) [K, H].
    """
    V, H, K, r, seed = cfg["V"], cfg["H"], cfg["K"], cfg["r"], cfg["seed"]
    dt = storage_dtype(cfg)
    vstd = math.sqrt(1.0 / r) if cfg["vscale"] == "1/r" else math.sqrt(1.0 / H)
    head = {
        "W": _randn((V, H), 0.02, seed, 1, device).to(dt),
        "U": _randn((K, H, r), math.sqrt(1.0 / r), seed, 2, device).to(dt),
        "Vf": _randn((K, H, r), vstd, seed, 3, device).to(dt),
        "Wp": _randn((K, H), math.sqrt(1.0 / (r * H)), seed, 4,
                     device).to(dt),
        "bp": torch.zeros(K, dtype=torch.float32, device=device),
        "e": None,
        "vbias": None,
    }
    if cfg.get("expander_bias"):
        head["e"] = _randn((K, H), 1.0, seed, 5, device).to(dt)
    if cfg.get("zipf"):
        g = _gen(seed, 6, "cpu")
        perm = torch.randperm(V, generator=g)
        rank = torch.empty(V, dtype=torch.float64)
        rank[perm] = torch.arange(V, dtype=torch.float64)
        head["vbias"] = (-cfg["zipf"] * torch.log1p(rank)).to(
            torch.float32).to(device)
    return head


def _drafter_mixture_logprobs(head, h, cfg):
    """log sum_z pi_z softmax(W (h + U_z V_z^T h + e_z) + b) at temperature 1.

    Input recipe for the target logits only (fp32 torch); pi uses the
    category temperature Z_T = 1.  h: [N, B, H].  Returns [N, B, V].
    """
    W = head["W"].float()
    U, Vf = head["U"].float(), head["Vf"].float()
    N, B, H = h.shape
    K = U.shape[0]
    ell = h[:, 0, :] @ head["Wp"].float().T + head["bp"].float()
    logpi = torch.log_softmax(ell, dim=-1)                       # [N, K]
    out = None
    for z in range(K):
        hz = h + (h @ Vf[z]) @ U[z].T
        if head["e"] is not None:
            hz = hz + head["e"][z].float()
        lz = hz.reshape(N * B, H) @ W.T
        if head["vbias"] is not None:
            lz = lz + head["vbias"]
        lz = torch.log_softmax(lz, dim=-1).reshape(N, B, -1) + logpi[:, z,
                                                                      None,
                                                                      None]
        out = lz if out is None else torch.logaddexp(out, lz)
    return out


def make_block(cfg, head, round_idx=0, device="cpu", sigma=None):
    """Hidden states, optional anchor and target logits for one round.

    h ~ N(0, 1) [N, B, H].  Target rows t_{n,i} = drafter mixture
    log-probabilities + N(0, sigma^2) for i < B; the bonus row (i = B) is
    W g + b + N(0, sigma^2) with a fresh g ~ N(0, 1).  Stored in the config's
    dtype.  Anchor is None (the prior reads h[:, 0]).
    """
    N, B, H, V = cfg["N"], cfg["B"], cfg["H"], cfg["V"]
    seed = cfg["seed"] * 7919 + 101 * int(round_idx)
    sigma = cfg["sigma"] if sigma is None else sigma
    dt = storage_dtype(cfg)
    h = _randn((N, B, H), 1.0, seed, 11, device).to(dt)
    with torch.no_grad():
        t = _drafter_mixture_logprobs(head, h.float(), cfg)
        t = t + _randn((N, B, V), sigma, seed, 12, device)
        rows = [t]
        if cfg["bonus"]:
            g = _randn((N, H), 1.0, seed, 13, device)
            tb = g @ head["W"].float().T
            if head["vbias"] is not None:
                tb = tb + head["vbias"]
            tb = tb + _randn((N, V), sigma, seed, 14, device)
            rows.append(tb[:, None, :])
        target = torch.cat(rows, dim=1).to(dt).contiguous()
    return {"hidden": h.contiguous(), "anchor": None, "target": target,
            "has_bonus": bool(cfg["bonus"])}


def initial_state(cfg, device="cpu", prefix_len=37):
    """Per-sequence absolute positions and round counters before round 0."""
    N = cfg["N"]
    pos = torch.full((N,), prefix_len, dtype=torch.int64, device=device)
    pos += torch.arange(N, dtype=torch.int64, device=device) % 5
    rnd = torch.zeros(N, dtype=torch.int32, device=device)
    return pos, rnd
