"""The no-allocation entry point dblast_target_lse_noalloc against the
workspace-based step.

Some callers cannot allocate device memory when they call in, for example a
plugin that runs inside another engine's enqueue step, where cudaMalloc would
synchronise the device and bypass the engine's memory pool.  This entry point
uses only a static device array inside the library.  The test calls it twice
in a row through the C ABI, on different inputs and temperatures, and checks
each result against the lse_target output of dblast_draft_and_verify, within
the log-sum-exp tolerance of the parity tests.  This file is collected last on
purpose.
"""
import ctypes

import numpy as np
import pytest
import torch

import synth
from tests import parity

pytestmark = pytest.mark.gpu


def test_noalloc_lse_matches_workspace_step_on_two_calls():
    from paper_2608_05448_gb300.binding import dblast_target_lse_noalloc
    cfg = synth.config("qwen3_8b_b32", H=256, K=4, r=8, B=8, N=6)   # full vocabulary
    head = synth.make_head(cfg, "cuda")
    for T, rd in ((1.0, 0), (0.7, 1)):
        blk = synth.make_block(cfg, head, rd, "cuda")
        pos, rnd = synth.initial_state(cfg, "cuda")
        ref = parity.run_gpu(head, blk, T, 1.0, 0, pos, rnd)["lse_target"].reshape(-1)
        out = torch.full((ref.numel(),), float("nan"), dtype=torch.float32, device="cuda")
        assert dblast_target_lse_noalloc(blk["target"], T, out) == 0
        torch.cuda.synchronize()
        got = out.cpu().double().numpy()
        want = ref.double().numpy()
        assert np.all(np.abs(got - want) <= 1e-4 + 1e-5 * np.abs(want))


def test_noalloc_rejects_rows_beyond_the_static_scratch():
    from paper_2608_05448_gb300 import binding
    lib = binding.lib()
    fake = ctypes.c_void_p(1 << 20)   # never dereferenced: the size check comes first
    V = 151936
    rows = binding.NOALLOC_MAX_RECORDS // 1187 + 1
    assert lib.dblast_target_lse_noalloc(fake, rows, V, 0, 1.0, fake, None) == 3
    assert lib.dblast_target_lse_noalloc(fake, rows - 1, V, 0, 0.0, fake, None) == 1
