"""GPU parity of the target-block early determinism (App. B) through the C
ABI: collision probabilities, D_b and the M-sample estimator of
dblast_target_determinism against the oracle, with the estimator's draws
bit-exact except where the oracle finds a draw within 1e-6 of a CDF edge."""
import numpy as np
import pytest
import torch

import synth
from oracle import dblast_oracle as orc

pytestmark = pytest.mark.gpu

RTOL = 1e-4


def _check(target, b, T, M, seed, seqs):
    from paper_2608_05448_gb300 import dblast_target_determinism
    out = dblast_target_determinism(target, b, T, M=M, seed=seed, samples=True)
    torch.cuda.synchronize()
    out = {k: v.cpu() for k, v in out.items()}
    ties_total = 0
    for n in seqs:
        p = orc.target_probs(target[n, :b].cpu(), T)
        np.testing.assert_allclose(out["collision"][n].double().numpy(),
                                   orc.collision_probability(p), rtol=RTOL, atol=1e-7)
        assert abs(float(out["d_exact"][n]) - orc.early_determinism_exact(p)) <= \
            RTOL * orc.early_determinism_exact(p) + 1e-7
        d_hat, smp, ties = orc.early_determinism_estimate(p, M, seed, n)
        ties_total += len(ties)
        tied = {m for m, _, _ in ties}
        for m in range(M):
            if m not in tied:
                assert out["samples"][n, m].tolist() == smp[m].tolist(), (n, m)
        if not ties:
            assert abs(float(out["d_hat"][n]) - d_hat) <= RTOL * d_hat + 1e-7
    return out, ties_total


def test_determinism_small_f32_all_sequences():
    g = torch.Generator().manual_seed(3)
    target = (torch.randn(5, 6, 1000, generator=g) * 1.5).cuda()
    _check(target, 4, 0.8, 20, 11, range(5))


def test_determinism_ragged_vocabulary_bf16():
    g = torch.Generator().manual_seed(4)
    target = (torch.randn(3, 9, 777, generator=g) * 2.0).to(torch.bfloat16).cuda()
    _check(target, 9, 1.0, 7, 5, range(3))


def test_determinism_qwen3_8b_target_paper_setting_sampled():
    """The paper's estimator setting (b = 15, M = 20) on the 8B-shaped target
    [32, 17, 151936] of the batched config; sequences 0 and 31 checked."""
    cfg = synth.config("qwen3_8b_b32")
    head = synth.make_head(cfg, "cuda")
    blk = synth.make_block(cfg, head, 0, "cuda")
    out, _ = _check(blk["target"], 15, 1.0, 20, 2024, [0, 31])
    assert bool(((out["d_exact"] > 0) & (out["d_exact"] <= 1)).all())


def test_determinism_one_hot_rows_are_fully_deterministic():
    target = torch.full((2, 3, 600), -1e4, dtype=torch.float32)
    target[:, :, 17] = 0.0
    target = target.cuda()
    from paper_2608_05448_gb300 import dblast_target_determinism
    out = dblast_target_determinism(target, 3, 1.0, M=4, seed=1, samples=True)
    torch.cuda.synchronize()
    assert torch.allclose(out["d_exact"].cpu(), torch.ones(2))
    assert torch.allclose(out["d_hat"].cpu(), torch.ones(2))
    assert bool((out["samples"] == 17).all())
