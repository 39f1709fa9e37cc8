"""GPU parity: the CUDA step through the C ABI against the fp64 oracle.

Every case draws seeded synthetic inputs (synth/), runs
dblast_draft_and_verify on cuda:0 and the oracle on the CPU, and compares
with tests/parity.py's rules: integer decisions bit-exact except counted
threshold ties, probabilities / overlaps / expected lengths within 1e-4
relative.
"""
import pytest
import torch

import synth
from tests import parity

pytestmark = pytest.mark.gpu

IMPLS = ["simt", "tcgen05"]


def _case(cfg, T, Z_T, seed, impl, seqs=None, round_idx=0, device="cuda"):
    head = synth.make_head(cfg, device)
    blk = synth.make_block(cfg, head, round_idx, device)
    pos, rnd = synth.initial_state(cfg, device)
    pos0, rnd0 = pos.clone(), rnd.clone()
    gpu = parity.run_gpu(head, blk, T, Z_T, seed, pos, rnd, impl=impl)
    seqs = list(range(cfg["N"])) if seqs is None else seqs
    orc = parity.run_oracle(head, blk, T, Z_T, seed, pos0, rnd0, seqs)
    stats = parity.compare(gpu, orc, seqs)
    # state update: pos += n_emitted, round += 1
    assert torch.equal(pos.cpu(), pos0.cpu() + gpu["n_emitted"].long())
    assert torch.equal(rnd.cpu(), rnd0.cpu() + 1)
    return stats


def _skip_unsupported(cfg, impl):
    rr = cfg["r"] + (1 if cfg.get("expander_bias") else 0)
    if impl == "tcgen05" and not (cfg["dtype"] == "bf16" and cfg["H"] % 64 == 0
                                  and cfg["K"] <= 16 and rr <= 32):
        pytest.skip("tensor-core path needs bf16, H % 64 == 0, K <= 16 and r (+1) <= 32")


@pytest.mark.parametrize("T,Z_T", [(1.0, 1.0), (0.6, 1.0), (1.5, 0.0)])
def test_tiny_config_all_sequences(T, Z_T):
    cfg = synth.config("tiny")
    st = _case(cfg, T, Z_T, seed=0, impl="auto")
    assert st["sequences"] == 8


SMALL = {
    # ragged vocabulary tail, expander bias, Zipf bias
    "ragged_e": dict(base="qwen3_8b_b32", V=1000, H=64, K=3, r=4, B=5, N=6,
                     expander_bias=True, sigma=0.7),
    # argmax prior, block of 16, 8 components
    "zt0": dict(base="qwen3_8b_b32", V=4099, H=128, K=8, r=16, B=16, N=3),
    # independent baseline K = 1 with B = 1
    "k1_b1": dict(base="qwen3_8b_b32", V=2048, H=64, K=1, r=8, B=1, N=5),
    # fp32, no bonus row, B = 32
    "f32_b32": dict(base="tiny", V=777, H=32, K=2, r=2, B=32, N=2, bonus=False),
    # many components, rank 32
    "k16_r32": dict(base="sweep_k16", V=3000, H=128, B=4, N=4),
    # the interface limits: B = 32 (one M tile, and two for the CTA pair) and
    # K = 32 with r = 64 (CUDA-core path only)
    "b32_bf16": dict(base="qwen3_8b_b32", V=2000, H=128, K=4, r=8, B=32, N=3),
    "b32_pair": dict(base="qwen3_8b_b32", V=2000, H=128, K=4, r=8, B=32, N=8),
    "k32_r64": dict(base="qwen3_8b_b32", V=1500, H=64, K=32, r=64, B=4, N=2),
}
SMALL_T = {"ragged_e": (0.8, 1.0), "zt0": (1.0, 0.0), "k1_b1": (1.5, 1.0),
           "f32_b32": (1.0, 0.7), "k16_r32": (0.7, 1.0), "b32_bf16": (1.0, 1.0),
           "b32_pair": (0.9, 1.0), "k32_r64": (1.2, 1.0)}


@pytest.mark.parametrize("impl", IMPLS)
@pytest.mark.parametrize("name", sorted(SMALL))
def test_small_shapes(name, impl):
    over = dict(SMALL[name])
    cfg = synth.config(over.pop("base"), **over)
    _skip_unsupported(cfg, impl)
    T, Z_T = SMALL_T[name]
    for seed in (1, 2):
        _case(cfg, T, Z_T, seed=seed, impl=impl)


@pytest.mark.parametrize("impl", IMPLS)
def test_four_rounds_carry_state(impl):
    from paper_2608_05448_gb300 import Head, Workspace
    cfg = synth.config("qwen3_8b_b32", V=2500, H=128, K=4, r=8, B=6, N=7)
    _skip_unsupported(cfg, impl)
    head_t = synth.make_head(cfg, "cuda")
    head = Head.from_dict(head_t)
    ws = Workspace(head, cfg["N"], cfg["B"], True)
    pos, rnd = synth.initial_state(cfg, "cuda")
    for rd in range(4):
        blk = synth.make_block(cfg, head_t, rd, "cuda")
        pos0, rnd0 = pos.clone(), rnd.clone()
        gpu = parity.run_gpu(head_t, blk, 1.0, 1.0, 11, pos, rnd, impl=impl, head=head, ws=ws)
        orc = parity.run_oracle(head_t, blk, 1.0, 1.0, 11, pos0, rnd0, list(range(cfg["N"])))
        parity.compare(gpu, orc, list(range(cfg["N"])))
        assert torch.equal(pos.cpu(), pos0.cpu() + gpu["n_emitted"].long())
        assert torch.equal(rnd.cpu(), rnd0.cpu() + 1)
    assert int(rnd[0]) == 4


def test_target_equal_to_drafter_accepts_every_token():
    """K = 1 and t = drafter logits (fp32): p = q, alpha = 1, all B accepted."""
    from oracle import dblast_oracle as orc
    cfg = synth.config("tiny", V=500, H=32, K=1, r=2, B=6, N=4)
    head = synth.make_head(cfg, "cuda")
    blk = synth.make_block(cfg, head, 0, "cuda")
    hd = orc.prepare_head(head)
    rows = []
    for n in range(cfg["N"]):
        h = orc.f64(blk["hidden"][n])
        l = orc.component_logits(head["W"], orc.branch_hidden(h, hd["U"], hd["Vf"], None),
                                 None)[:, 0, :]
        rows.append(torch.cat([torch.tensor(l), torch.tensor(l[:1])], 0))
    blk["target"] = torch.stack(rows).float().cuda().contiguous()
    pos, rnd = synth.initial_state(cfg, "cuda")
    gpu = parity.run_gpu(head, blk, 0.9, 1.0, 5, pos, rnd)
    assert (gpu["accepted"] == cfg["B"]).all()
    assert torch.allclose(gpu["alpha"], torch.ones_like(gpu["alpha"]), atol=1e-5)
    assert torch.allclose(gpu["exp_len"], torch.full_like(gpu["exp_len"], cfg["B"]), atol=1e-4)


def test_disjoint_target_rejects_first_token():
    cfg = synth.config("qwen3_8b_b32", V=1500, H=64, K=2, r=4, B=4, N=6)
    head = synth.make_head(cfg, "cuda")
    blk = synth.make_block(cfg, head, 0, "cuda")
    blk["target"] = (-4.0 * blk["target"].float()).to(torch.bfloat16).contiguous()
    pos, rnd = synth.initial_state(cfg, "cuda")
    pos0, rnd0 = pos.clone(), rnd.clone()
    gpu = parity.run_gpu(head, blk, 1.0, 1.0, 3, pos, rnd)
    assert (gpu["accepted"] == 0).sum() >= 4
    orc = parity.run_oracle(head, blk, 1.0, 1.0, 3, pos0, rnd0, list(range(cfg["N"])))
    parity.compare(gpu, orc, list(range(cfg["N"])))


@pytest.mark.parametrize("impl", IMPLS)
def test_qwen3_4b_single_sequence_full(impl):
    cfg = synth.config("qwen3_4b_b1")
    _skip_unsupported(cfg, impl)
    _case(cfg, 1.0, 1.0, seed=0, impl=impl)


@pytest.mark.parametrize("T", [1.0, 0.6])
def test_qwen3_8b_batched_all_sequences(T):
    """The headline workload in the launch configuration the bench times
    (tensor-core passes, N=32, B=16, K=8, r=16, H=4096, V=151936): every one
    of the 32 sequences against the oracle, at both temperatures."""
    cfg = synth.config("qwen3_8b_b32")
    st = _case(cfg, T, 1.0, seed=0, impl="auto")
    assert st["sequences"] == 32 and st["emitted_checked"] >= 28


def test_qwen3_8b_batched_simt_sampled():
    """The CUDA-core passes on the headline shapes, two sequences."""
    cfg = synth.config("qwen3_8b_b32")
    _case(cfg, 1.0, 1.0, seed=0, impl="simt", seqs=[0, 31])


@pytest.mark.parametrize("impl", IMPLS)
@pytest.mark.parametrize("bonus,top_k,top_p", [(True, 0, 0.0), (False, 0, 0.0), (True, 20, 0.95),
                                              (False, 20, 0.8)])
def test_soft_split_calls_match_oracle(impl, bonus, top_k, top_p):
    """dblast_draft_block, then dblast_verify_block on the workspace it left
    (Sec. 3.1 drafting, then Algorithm 1's verification), against the oracle
    element by element, with and without a bonus row and a target filter;
    and the fused call on the same inputs gives the same decisions."""
    cfg = synth.config("qwen3_8b_b32", V=6000, H=256, K=8, r=16, B=16, N=16, bonus=bonus)
    _skip_unsupported(cfg, impl)
    head = synth.make_head(cfg, "cuda")
    blk = synth.make_block(cfg, head, 0, "cuda")
    seqs = list(range(cfg["N"]))
    pos, rnd = synth.initial_state(cfg, "cuda")
    pos0, rnd0 = pos.clone(), rnd.clone()
    gpu = parity.run_gpu_split(head, blk, 0.9, 1.0, 12, pos, rnd, impl=impl, top_k=top_k,
                               top_p=top_p)
    orc = parity.run_oracle(head, blk, 0.9, 1.0, 12, pos0, rnd0, seqs, top_k=top_k, top_p=top_p)
    parity.compare(gpu, orc, seqs)
    assert torch.equal(pos.cpu(), pos0.cpu() + gpu["n_emitted"].long())
    assert torch.equal(rnd.cpu(), rnd0.cpu() + 1)
    posf, rndf = pos0.clone(), rnd0.clone()
    fused = parity.run_gpu(head, blk, 0.9, 1.0, 12, posf, rndf, impl=impl, top_k=top_k,
                           top_p=top_p)
    for k in ("z_hat", "tokens", "accepted", "emitted", "n_emitted", "tie_flags"):
        assert torch.equal(gpu[k], fused[k]), k


@pytest.mark.parametrize("T,sigma", [(0.7, 0.3), (1.5, 1.0)])
def test_entropy_sweep_k16_r32_sampled(T, sigma):
    """Entropy-sweep shapes at full size (N=64, K=16, r=32, V=151936), two cells."""
    cfg = synth.config("sweep_k16", sigma=sigma)
    _case(cfg, T, 1.0, seed=4, impl="tcgen05", seqs=[0, 63])


def test_entropy_sweep_k1_baseline_sampled():
    """The K=1 independent-block baseline of the sweep (same shapes, one component)."""
    cfg = synth.config("sweep_k16", K=1)
    _case(cfg, 1.0, 1.0, seed=5, impl="tcgen05", seqs=[7])


@pytest.mark.parametrize("B", [8, 32])
def test_serving_batch_four_rounds_sampled(B):
    """Serving step at full size (N=256, B=8 or 32): state carried over four
    rounds, each round with fresh hidden states and targets; sampled sequences
    checked against the oracle every round."""
    from paper_2608_05448_gb300 import Head, Workspace
    cfg = synth.config("serve_b8" if B == 8 else "serve_b32")
    head_t = synth.make_head(cfg, "cuda")
    head = Head.from_dict(head_t)
    ws = Workspace(head, cfg["N"], cfg["B"], True)
    pos, rnd = synth.initial_state(cfg, "cuda")
    seqs = [3, 255]
    rounds = 4 if B == 8 else 2
    for rd in range(rounds):
        blk = synth.make_block(cfg, head_t, rd, "cuda")
        pos0, rnd0 = pos.clone(), rnd.clone()
        gpu = parity.run_gpu(head_t, blk, 1.0, 1.0, 21, pos, rnd, head=head, ws=ws)
        orc = parity.run_oracle(head_t, blk, 1.0, 1.0, 21, pos0, rnd0, seqs)
        parity.compare(gpu, orc, seqs)
        assert torch.equal(pos.cpu(), pos0.cpu() + gpu["n_emitted"].long())
        assert torch.equal(rnd.cpu(), rnd0.cpu() + 1)
        del blk, gpu
    assert int(rnd[0]) == rounds


@pytest.mark.parametrize("mode,top_k,top_p", [("soft", 20, 0.95), ("greedy", 0, 0.0)])
def test_target_statistics_in_the_draft_pass_match_the_separate_kernel(mode, top_k, top_p):
    """The fused step computes the target statistics in the draft pass's idle
    warps (greedy mode, or a target filter on); with DBLAST_FUSE_TSTATS=0 a
    kernel of its own does.  Decisions are
    identical and the floats agree within the parity tolerances (another
    summation order)."""
    import os
    cfg = synth.config("qwen3_8b_b32", V=6000, H=128, K=4, r=8, B=9, N=6)
    head = synth.make_head(cfg, "cuda")
    blk = synth.make_block(cfg, head, 0, "cuda")
    res = []
    for fuse in ("1", "0"):
        os.environ["DBLAST_FUSE_TSTATS"] = fuse
        try:
            pos, rnd = synth.initial_state(cfg, "cuda")
            res.append(parity.run_gpu(head, blk, 0.9, 1.0, 6, pos, rnd, impl="tcgen05", mode=mode,
                                      top_k=top_k, top_p=top_p))
        finally:
            os.environ.pop("DBLAST_FUSE_TSTATS", None)
    for k in res[0]:
        a, b = res[0][k], res[1][k]
        if a.is_floating_point():
            atol = 1e-4 if k in ("lse_target", "lse") else 1e-6
            assert torch.allclose(a, b, rtol=1e-4, atol=atol, equal_nan=True), k
        else:
            assert torch.equal(a, b), k
