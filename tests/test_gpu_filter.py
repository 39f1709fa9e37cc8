"""GPU parity of verification against the filtered target (temperature,
top-k, top-p; Sec. 3.2 and Sec. 4) in both drafting modes, through the C ABI
against the oracle.  A top-p cut within 1e-6 of top_p is a tie of the oracle
("top_p" at its row) and ends the checked prefix there."""
import pytest
import torch

import synth
from tests import parity
from tests.test_gpu_parity import SMALL, _skip_unsupported

pytestmark = pytest.mark.gpu

# the paper's target settings: (T, top_p) with top-k 20
PAPER = [(0.7, 0.8), (1.0, 0.95), (1.5, 0.95)]


def _case(cfg, T, Z_T, seed, impl, mode, top_k, top_p, seqs=None):
    head = synth.make_head(cfg, "cuda")
    blk = synth.make_block(cfg, head, 0, "cuda")
    pos, rnd = synth.initial_state(cfg, "cuda")
    pos0, rnd0 = pos.clone(), rnd.clone()
    gpu = parity.run_gpu(head, blk, T, Z_T, seed, pos, rnd, impl=impl, mode=mode,
                         top_k=top_k, top_p=top_p)
    seqs = list(range(cfg["N"])) if seqs is None else seqs
    orc = parity.run_oracle(head, blk, T, Z_T, seed, pos0, rnd0, seqs, mode=mode,
                            top_k=top_k, top_p=top_p)
    cmp = parity.compare_greedy if mode == "greedy" else parity.compare
    stats = cmp(gpu, orc, seqs)
    assert torch.equal(pos.cpu(), pos0.cpu() + gpu["n_emitted"].long())
    # every emitted extra token lies in the kept set: its filtered probability is positive
    return stats, gpu, orc


@pytest.mark.parametrize("mode", ["soft", "greedy"])
@pytest.mark.parametrize("impl", ["simt", "tcgen05"])
@pytest.mark.parametrize("name", ["ragged_e", "zt0", "b32_pair", "k16_r32"])
def test_filter_small_shapes(name, impl, mode):
    over = dict(SMALL[name])
    cfg = synth.config(over.pop("base"), **over)
    _skip_unsupported(cfg, impl)
    for seed, (T, tp) in enumerate(PAPER):
        _case(cfg, T, 1.0, seed, impl, mode, 20, tp)


@pytest.mark.parametrize("mode", ["soft", "greedy"])
def test_filter_top_k_only_and_top_p_only(mode):
    cfg = synth.config("tiny", V=200, N=6, B=5)
    _case(cfg, 1.0, 1.0, 3, "auto", mode, 7, 0.0)
    _case(cfg, 0.8, 1.0, 4, "auto", mode, 0, 0.9)      # top-p alone: V <= 256
    _case(cfg, 1.2, 0.0, 5, "auto", mode, 300, 0.5)    # top_k >= V: top-p over all


@pytest.mark.parametrize("mode", ["soft", "greedy"])
@pytest.mark.parametrize("T,top_p", PAPER)
def test_filter_qwen3_8b_paper_settings_sampled(mode, T, top_p):
    cfg = synth.config("qwen3_8b_b32")
    st, gpu, orc = _case(cfg, T, 1.0, 7, "tcgen05", mode, 20, top_p, seqs=[0, 31])
    assert st["sequences"] == 2


def test_filter_top_k_one_accepts_exactly_the_target_argmax():
    cfg = synth.config("qwen3_8b_b32", V=3000, H=128, K=4, r=8, B=8, N=16)
    head = synth.make_head(cfg, "cuda")
    blk = synth.make_block(cfg, head, 0, "cuda")
    top = blk["target"].float().argmax(-1).cpu()
    for mode in ("soft", "greedy"):
        pos, rnd = synth.initial_state(cfg, "cuda")
        gpu = parity.run_gpu(head, blk, 1.0, 1.0, 2, pos, rnd, mode=mode, top_k=1)
        for n in range(cfg["N"]):
            L = int(gpu["accepted"][n])
            em = gpu["emitted"][n].tolist()
            assert em[:L] == top[n, :L].tolist()
            ne = int(gpu["n_emitted"][n])
            assert em[ne - 1] == int(top[n, ne - 1])
        assert torch.allclose(gpu["collision"], torch.ones_like(gpu["collision"]))


@pytest.mark.parametrize("mode", ["soft", "greedy"])
def test_filter_qwen3_4b_single_sequence(mode):
    cfg = synth.config("qwen3_4b_b1")
    _case(cfg, 0.7, 1.0, 2, "tcgen05", mode, 20, 0.8)


@pytest.mark.parametrize("mode", ["soft", "greedy"])
def test_filter_serving_b32_sampled(mode):
    """Serving shapes (N=256, B=32): 8,448 filtered target rows per step."""
    cfg = synth.config("serve_b32")
    _case(cfg, 1.0, 1.0, 4, "tcgen05", mode, 20, 0.95, seqs=[0, 255])
