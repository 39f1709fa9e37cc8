"""Device-side index checks (dblast_set_checks): a data-dependent token index
outside [0, V) is recorded in the workspace status word and reported as
DBLAST_ERR_BOUNDS, without a trap (the access uses the clamped index); a
normal step with the checks on reports nothing and matches the oracle."""
import pytest
import torch

import synth
from tests import parity

pytestmark = pytest.mark.gpu

DBLAST_OK, DBLAST_ERR_BOUNDS = 0, 7


def _al_call(cfg, tokens):
    from paper_2608_05448_gb300 import Head, Workspace, dblast_al_objective
    head_t = synth.make_head(cfg, "cuda")
    blk = synth.make_block(cfg, head_t, 0, "cuda")
    head = Head.from_dict(head_t)
    ws = Workspace(head, cfg["N"], cfg["B"], blk["has_bonus"])
    pos, rnd = synth.initial_state(cfg, "cuda")
    out = dblast_al_objective(head, ws, blk["hidden"], pos, rnd, 1.0, 1.0, 5, tokens.cuda(),
                              blk["target"], blk["has_bonus"], tau=0.1)
    torch.cuda.synchronize()
    return ws, out


def test_out_of_range_given_tokens_are_reported_with_checks_on():
    from paper_2608_05448_gb300 import dblast_device_status, dblast_set_checks
    cfg = synth.config("tiny")
    tokens = torch.randint(0, cfg["V"], (cfg["N"], cfg["B"]), dtype=torch.int32,
                           generator=torch.Generator().manual_seed(3))
    bad = tokens.clone()
    bad[1, 0] = cfg["V"] + 3
    bad[2, 1] = -1
    dblast_set_checks(True)
    try:
        ws, out = _al_call(cfg, bad)
        assert dblast_device_status(ws) == DBLAST_ERR_BOUNDS
        assert dblast_device_status(ws) == DBLAST_OK        # the record was cleared
        assert bool(torch.isfinite(out["nll"]).all())        # clamped, not trapped
        ws, _ = _al_call(cfg, tokens)                        # in-range tokens: nothing
        assert dblast_device_status(ws) == DBLAST_OK
    finally:
        dblast_set_checks(False)
    ws, _ = _al_call(cfg, bad)                               # checks off: not recorded
    assert dblast_device_status(ws) == DBLAST_OK


@pytest.mark.parametrize("mode", ["soft", "greedy"])
def test_step_with_checks_on_matches_oracle(mode):
    from paper_2608_05448_gb300 import (Head, Workspace, dblast_device_status,
                                        dblast_set_checks)
    cfg = synth.config("qwen3_8b_b32", V=3001, H=128, K=4, r=8, B=8, N=4)
    head_t = synth.make_head(cfg, "cuda")
    blk = synth.make_block(cfg, head_t, 0, "cuda")
    head = Head.from_dict(head_t)
    ws = Workspace(head, cfg["N"], cfg["B"], blk["has_bonus"])
    pos, rnd = synth.initial_state(cfg, "cuda")
    pos0, rnd0 = pos.clone(), rnd.clone()
    seqs = list(range(cfg["N"]))
    dblast_set_checks(True)
    try:
        gpu = parity.run_gpu(head_t, blk, 0.8, 1.0, 2, pos, rnd, head=head, ws=ws, mode=mode)
        assert dblast_device_status(ws) == DBLAST_OK
    finally:
        dblast_set_checks(False)
    orc = parity.run_oracle(head_t, blk, 0.8, 1.0, 2, pos0, rnd0, seqs, mode=mode)
    if mode == "greedy":
        parity.compare_greedy(gpu, orc, seqs)
    else:
        parity.compare(gpu, orc, seqs)
