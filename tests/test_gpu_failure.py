"""Failure detection without a GPU fault: every device-side wait of the
tensor-core passes is bounded.  dblast_set_wait_limit(1) makes the waits give
up at once; the kernels then record a timeout in the workspace, drain their
copies and MMAs, free TMEM and return, so the step reports
DBLAST_ERR_TIMEOUT through dblast_device_status and the context stays usable:
the next step with the default limit matches the oracle."""
import pytest
import torch

import synth
from tests import parity

pytestmark = pytest.mark.gpu

DBLAST_OK, DBLAST_ERR_TIMEOUT = 0, 5


@pytest.mark.parametrize("N,B", [(4, 8), (16, 16)])   # one-SM form, then the CTA pair
def test_bounded_waits_report_a_timeout_and_the_context_survives(N, B):
    from paper_2608_05448_gb300 import (Head, Workspace, dblast_device_status,
                                        dblast_draft_and_verify, dblast_set_wait_limit)
    cfg = synth.config("qwen3_8b_b32", V=3000, H=128, K=4, r=8, B=B, N=N)
    head_t = synth.make_head(cfg, "cuda")
    head = Head.from_dict(head_t)
    blk = synth.make_block(cfg, head_t, 0, "cuda")
    ws = Workspace(head, N, B, True)
    pos, rnd = synth.initial_state(cfg, "cuda")
    dblast_set_wait_limit(1)
    try:
        dblast_draft_and_verify(head, ws, blk["hidden"], pos, rnd, 1.0, 1.0, 3, blk["target"],
                                True, impl="tcgen05")
        torch.cuda.synchronize()
    finally:
        dblast_set_wait_limit(0)
    assert dblast_device_status(ws) == DBLAST_ERR_TIMEOUT
    assert dblast_device_status(ws) == DBLAST_OK          # the record was cleared
    # the same workspace and context, default limit: a correct step
    pos, rnd = synth.initial_state(cfg, "cuda")
    pos0, rnd0 = pos.clone(), rnd.clone()
    gpu = parity.run_gpu(head_t, blk, 1.0, 1.0, 3, pos, rnd, impl="tcgen05", head=head, ws=ws)
    assert dblast_device_status(ws) == DBLAST_OK
    orc = parity.run_oracle(head_t, blk, 1.0, 1.0, 3, pos0, rnd0, list(range(N)))
    parity.compare(gpu, orc, list(range(N)))
