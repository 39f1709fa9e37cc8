"""GPU parity of the training-side objectives, forward only (Sec. 3.2):
dblast_al_objective against the oracle's al_objective_sequence on target
blocks drawn from the (filtered) target."""
import numpy as np
import pytest
import torch

import synth
from oracle import dblast_oracle as orc
from tests.test_gpu_parity import SMALL, _skip_unsupported

pytestmark = pytest.mark.gpu

RTOL = 1e-4


def _target_blocks(target, B, T, top_k, top_p, seed):
    """x*_i drawn from the (filtered) target rows, as training data would be."""
    rng = np.random.default_rng(seed)
    N = target.shape[0]
    out = np.empty((N, B), dtype=np.int32)
    for n in range(N):
        p, _ = orc.target_distributions(orc.f64(target[n, :B]), T, top_k, top_p, [])
        for i in range(B):
            out[n, i] = rng.choice(p.shape[1], p=p[i] / p[i].sum())
    return torch.from_numpy(out)


def _case(cfg, T, Z_T, tau, impl, top_k=0, top_p=0.0, seqs=None, seed=0):
    from paper_2608_05448_gb300 import Head, Workspace, dblast_al_objective
    head_t = synth.make_head(cfg, "cuda")
    blk = synth.make_block(cfg, head_t, 0, "cuda")
    head = Head.from_dict(head_t)
    N, B = cfg["N"], cfg["B"]
    ws = Workspace(head, N, B, blk["has_bonus"])
    pos, rnd = synth.initial_state(cfg, "cuda")
    tokens = _target_blocks(blk["target"], B, T, top_k, top_p, seed)
    out = dblast_al_objective(head, ws, blk["hidden"], pos, rnd, T, Z_T, 5, tokens.cuda(),
                              blk["target"], blk["has_bonus"], tau=tau, top_k=top_k,
                              top_p=top_p, impl=impl)
    torch.cuda.synchronize()
    out = {k: v.cpu() for k, v in out.items()}
    hd = orc.prepare_head(head_t)
    seqs = range(N) if seqs is None else seqs
    for n in seqs:
        o = orc.al_objective_sequence(hd, orc.f64(blk["hidden"][n]), None,
                                      orc.f64(blk["target"][n]), tokens[n].tolist(), T, Z_T,
                                      tau, top_k, top_p)
        assert not any(k == "top_p" for k, _, _ in o["ties"])
        for key in ("q_cond", "p_tok", "A", "r", "S"):
            got = out["accept_prob" if key == "A" else key][n].double().numpy()
            np.testing.assert_allclose(got, o[key], rtol=RTOL, atol=1e-7, err_msg=key)
        assert abs(float(out["nll"][n]) - o["nll"]) <= RTOL * abs(o["nll"]) + 1e-4
        if not o["ties"]:
            assert int(out["l_tau"][n]) == o["l_tau"]
            assert abs(float(out["j_al"][n]) - o["J"]) <= RTOL * abs(o["J"]) + 1e-4
    return out


@pytest.mark.parametrize("impl", ["simt", "tcgen05"])
@pytest.mark.parametrize("name", ["ragged_e", "k1_b1", "b32_bf16", "k16_r32"])
def test_al_small_shapes(name, impl):
    over = dict(SMALL[name])
    cfg = synth.config(over.pop("base"), **over)
    _skip_unsupported(cfg, impl)
    _case(cfg, 1.0, 1.0, 0.1, impl)
    _case(cfg, 0.7, 1.0, 0.1, impl, top_k=20, top_p=0.8, seed=1)


def test_al_tiny_tau_edge_cases():
    cfg = synth.config("tiny")
    out = _case(cfg, 1.0, 1.0, 0.0, "auto")
    assert bool((out["l_tau"] == cfg["B"]).all())      # tau = 0 keeps every prefix
    _case(cfg, 1.0, 1.0, 1e6, "auto")                   # every r_1 below tau: l_tau = 1


@pytest.mark.parametrize("top", [(0, 0.0), (20, 0.95)])
def test_al_qwen3_8b_sampled(top):
    cfg = synth.config("qwen3_8b_b32")
    out = _case(cfg, 1.0, 1.0, 0.1, "tcgen05", top_k=top[0], top_p=top[1], seqs=[0, 31])
    assert bool(torch.isfinite(out["nll"]).all())
