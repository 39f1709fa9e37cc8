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
