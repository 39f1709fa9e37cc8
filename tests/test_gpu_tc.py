"""Tensor-core (tcgen05) prep GEMM against the CUDA-core one, and the
bounded-wait status of the tensor-core pass."""
import os

import pytest
import torch

import synth

pytestmark = pytest.mark.gpu


def _wu(head, cfg):
    rr = cfg["r"] + (1 if cfg.get("expander_bias") else 0)
    n = cfg["V"] * cfg["K"] * rr
    return head.prep[: 4 * n].view(torch.float32).reshape(cfg["V"], cfg["K"], rr).clone()


@pytest.mark.parametrize("over", [dict(V=1000, H=128, K=3, r=4, expander_bias=True),
                                  dict(V=4096, H=256, K=8, r=16),
                                  dict(V=2944, H=512, K=16, r=32)])
def test_tc_prep_matches_cuda_core_prep(over, monkeypatch):
    from paper_2608_05448_gb300 import Head
    cfg = synth.config("qwen3_8b_b32", **over)
    head_t = synth.make_head(cfg, "cuda")
    h_tc = Head.from_dict(head_t)
    monkeypatch.setenv("DBLAST_PREP_SIMT", "1")
    h_simt = Head.from_dict(head_t)
    monkeypatch.delenv("DBLAST_PREP_SIMT")
    torch.cuda.synchronize()
    a, b = _wu(h_tc, cfg), _wu(h_simt, cfg)
    # exact-input bf16 products, fp32 accumulation in different orders
    assert torch.allclose(a, b, rtol=1e-5, atol=1e-5 * float(b.abs().max())), \
        float((a - b).abs().max())
    # and against an fp64 product
    W = head_t["W"].double()
    U = head_t["U"].double()
    ref = torch.einsum("vh,khr->vkr", W, U)
    assert torch.allclose(a[:, :, :cfg["r"]].double(), ref, rtol=1e-5,
                          atol=1e-5 * float(ref.abs().max()))


@pytest.mark.parametrize("over", [dict(V=20000, H=512, K=8, r=16, B=16, N=32),   # 4 M tiles
                                  dict(V=3001, H=256, K=3, r=4, B=5, N=40,        # 2 M tiles
                                       expander_bias=True)])
def test_draft_pass_cta_pair_matches_single_cta(over, monkeypatch):
    """The CTA-pair draft pass (cta_group::2 MMAs of 256 rows, B split between
    the two SMs) computes the same products in the same order as the one-SM
    pass: the oracle checks sampled sequences, and every output must equal
    the one-SM schedule's bit for bit."""
    from tests import parity
    cfg = synth.config("qwen3_8b_b32", **over)
    head = synth.make_head(cfg, "cuda")
    blk = synth.make_block(cfg, head, 0, "cuda")
    runs = {}
    for c in ("0", "1"):
        monkeypatch.setenv("DBLAST_DRAFT_PAIR", c)
        pos, rnd = synth.initial_state(cfg, "cuda")
        runs[c] = parity.run_gpu(head, blk, 0.8, 1.0, 7, pos, rnd, impl="tcgen05")
    pos0, rnd0 = synth.initial_state(cfg, "cuda")
    seqs = [0, cfg["N"] // 2 - 1, cfg["N"] - 1]
    orc = parity.run_oracle(head, blk, 0.8, 1.0, 7, pos0, rnd0, seqs)
    parity.compare(runs["1"], orc, seqs)
    for k, v in runs["0"].items():
        assert torch.equal(v, runs["1"][k]), k
