"""GPU parity of the greedy-branch mode (Sec. 3.1, "Drafter sampling during
inference"; App. A) through the C ABI against the oracle's greedy step.

Greedy argmax decisions are exact except where the oracle's top-two logit gap
is below its tie band; acceptance, residual and bonus draws follow the same
rules as the stochastic mode (tests/parity.py).
"""
import os

import pytest
import torch

import synth
from tests import parity
from tests.test_gpu_parity import SMALL, SMALL_T, _skip_unsupported

pytestmark = pytest.mark.gpu

IMPLS = ["simt", "tcgen05"]


def _case(cfg, T, Z_T, seed, impl, seqs=None, round_idx=0):
    head = synth.make_head(cfg, "cuda")
    blk = synth.make_block(cfg, head, round_idx, "cuda")
    pos, rnd = synth.initial_state(cfg, "cuda")
    pos0, rnd0 = pos.clone(), rnd.clone()
    gpu = parity.run_gpu(head, blk, T, Z_T, seed, pos, rnd, impl=impl, mode="greedy")
    seqs = list(range(cfg["N"])) if seqs is None else seqs
    orc = parity.run_oracle(head, blk, T, Z_T, seed, pos0, rnd0, seqs, mode="greedy")
    stats = parity.compare_greedy(gpu, orc, seqs)
    assert torch.equal(pos.cpu(), pos0.cpu() + gpu["n_emitted"].long())
    assert torch.equal(rnd.cpu(), rnd0.cpu() + 1)
    return stats, gpu


@pytest.mark.parametrize("T,Z_T", [(1.0, 1.0), (0.6, 0.0)])
def test_greedy_tiny_all_sequences(T, Z_T):
    cfg = synth.config("tiny")
    st, _ = _case(cfg, T, Z_T, seed=0, impl="auto")
    assert st["sequences"] == 8 and st["branch_tokens"] > 0


@pytest.mark.parametrize("impl", IMPLS)
@pytest.mark.parametrize("name", sorted(SMALL))
def test_greedy_small_shapes(name, impl):
    over = dict(SMALL[name])
    cfg = synth.config(over.pop("base"), **over)
    _skip_unsupported(cfg, impl)
    T, Z_T = SMALL_T[name]
    for seed in (1, 2):
        _case(cfg, T, Z_T, seed=seed, impl=impl)


@pytest.mark.parametrize("impl", IMPLS)
def test_greedy_qwen3_8b_batched(impl):
    """The headline shapes in greedy mode: all 32 sequences on the
    tensor-core path the bench times, two on the CUDA-core path."""
    cfg = synth.config("qwen3_8b_b32")
    _skip_unsupported(cfg, impl)
    seqs = None if impl == "tcgen05" else [0, 31]
    st, gpu = _case(cfg, 1.0, 1.0, seed=0, impl=impl, seqs=seqs)
    if impl == "tcgen05":
        assert st["sequences"] == 32
    # q_greedy sums pi over the consistent branches: a probability
    q = gpu["q_tok"]
    assert bool(((q > 0) & (q <= 1 + 1e-6)).all())


def test_greedy_split_calls_equal_fused_call():
    """dblast_draft_block + dblast_verify_block == dblast_draft_and_verify
    (decisions identical; the fused call computes the target statistics in the
    draft pass with another summation order, so floats agree within the parity
    tolerances)."""
    from paper_2608_05448_gb300 import (Head, Workspace, dblast_draft_and_verify,
                                        dblast_draft_block, dblast_verify_block)
    cfg = synth.config("qwen3_8b_b32", V=3000, H=128, K=6, r=8, B=7, N=5)
    head_t = synth.make_head(cfg, "cuda")
    head = Head.from_dict(head_t)
    blk = synth.make_block(cfg, head_t, 0, "cuda")
    outs = []
    for split in (False, True):
        ws = Workspace(head, cfg["N"], cfg["B"], True)
        pos, rnd = synth.initial_state(cfg, "cuda")
        args = (head, ws, blk["hidden"], pos, rnd, 0.8, 1.0, 9)
        if split:
            d = dblast_draft_block(*args, mode="greedy")
            v = dblast_verify_block(*args, blk["target"], True, mode="greedy")
        else:
            d, v = dblast_draft_and_verify(*args, blk["target"], True, mode="greedy")
        torch.cuda.synchronize()
        outs.append(({k: x.cpu() for k, x in d.items()}, {k: x.cpu() for k, x in v.items()},
                     pos.cpu()))
    for a, b in zip(outs[0][:2], outs[1][:2]):
        for k in a:
            if a[k].is_floating_point():
                atol = 1e-4 if k in ("lse_target", "lse") else 1e-6
                assert torch.allclose(a[k], b[k], rtol=1e-4, atol=atol, equal_nan=True), k
            else:
                assert torch.equal(a[k], b[k]), k
    assert torch.equal(outs[0][2], outs[1][2])


def test_greedy_cta_pair_matches_single_cta():
    """The CTA-pair and one-SM forms of the greedy draft pass give identical
    records, hence identical outputs."""
    cfg = synth.config("qwen3_8b_b32", V=5000, H=256, K=8, r=16, B=16, N=16)
    head = synth.make_head(cfg, "cuda")
    blk = synth.make_block(cfg, head, 0, "cuda")
    res = []
    for pair in ("1", "0"):
        os.environ["DBLAST_DRAFT_PAIR"] = pair
        try:
            pos, rnd = synth.initial_state(cfg, "cuda")
            res.append(parity.run_gpu(head, blk, 1.0, 1.0, 4, pos, rnd, impl="tcgen05",
                                      mode="greedy"))
        finally:
            os.environ.pop("DBLAST_DRAFT_PAIR", None)
    for k in res[0]:
        assert torch.equal(res[0][k], res[1][k]), k


@pytest.mark.parametrize("impl", IMPLS)
def test_greedy_four_rounds_carry_state(impl):
    from paper_2608_05448_gb300 import Head, Workspace
    cfg = synth.config("qwen3_8b_b32", V=2500, H=128, K=4, r=8, B=6, N=7)
    _skip_unsupported(cfg, impl)
    head_t = synth.make_head(cfg, "cuda")
    head = Head.from_dict(head_t)
    ws = Workspace(head, cfg["N"], cfg["B"], True)
    pos, rnd = synth.initial_state(cfg, "cuda")
    seqs = list(range(cfg["N"]))
    for rd in range(4):
        blk = synth.make_block(cfg, head_t, rd, "cuda")
        pos0, rnd0 = pos.clone(), rnd.clone()
        gpu = parity.run_gpu(head_t, blk, 1.0, 1.0, 11, pos, rnd, impl=impl, head=head, ws=ws,
                             mode="greedy")
        orc = parity.run_oracle(head_t, blk, 1.0, 1.0, 11, pos0, rnd0, seqs, mode="greedy")
        parity.compare_greedy(gpu, orc, seqs)
        assert torch.equal(pos.cpu(), pos0.cpu() + gpu["n_emitted"].long())
    assert int(rnd[0]) == 4


@pytest.mark.parametrize("impl", IMPLS)
def test_greedy_qwen3_4b_single_sequence_full(impl):
    cfg = synth.config("qwen3_4b_b1")
    _skip_unsupported(cfg, impl)
    _case(cfg, 1.0, 1.0, seed=3, impl=impl)


@pytest.mark.parametrize("K", [16, 1])
def test_greedy_entropy_sweep_sampled(K):
    """Entropy-sweep shapes at full size (N=64, r=32, V=151936), the K=16 drafter
    and the K=1 independent-block baseline, high-entropy cell."""
    cfg = synth.config("sweep_k16", K=K, sigma=1.0)
    _case(cfg, 1.5, 1.0, seed=8, impl="tcgen05", seqs=[0, 63])


def test_greedy_serving_batch_four_rounds_sampled():
    """Serving step at full size (N=256, B=8): state carried over four rounds,
    fresh hidden states and targets each round, sampled sequences checked."""
    from paper_2608_05448_gb300 import Head, Workspace
    cfg = synth.config("serve_b8")
    head_t = synth.make_head(cfg, "cuda")
    head = Head.from_dict(head_t)
    ws = Workspace(head, cfg["N"], cfg["B"], True)
    pos, rnd = synth.initial_state(cfg, "cuda")
    seqs = [3, 255]
    for rd in range(4):
        blk = synth.make_block(cfg, head_t, rd, "cuda")
        pos0, rnd0 = pos.clone(), rnd.clone()
        gpu = parity.run_gpu(head_t, blk, 1.0, 1.0, 21, pos, rnd, head=head, ws=ws, mode="greedy")
        orc = parity.run_oracle(head_t, blk, 1.0, 1.0, 21, pos0, rnd0, seqs, mode="greedy")
        parity.compare_greedy(gpu, orc, seqs)
        assert torch.equal(pos.cpu(), pos0.cpu() + gpu["n_emitted"].long())
        del blk, gpu
    assert int(rnd[0]) == 4
