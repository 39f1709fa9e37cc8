"""Pins for the oracle's Philox4x32-10 and decision uniforms (CPU only)."""
import json
import os
import subprocess
import sys
import textwrap

import numpy as np
import pytest

from oracle.philox import (decision_uniform, philox4x32_10, word_to_uniform)

CASES = [
    # (counter, seed)
    ((0, 0, 0, 0), 0),
    ((1, 2, 3, 4), 12345),
    ((0xFFFFFFFF, 0xFFFFFFFF, 0xFFFFFFFF, 0xFFFFFFFF), 0xFFFFFFFFFFFFFFFF),
    ((7, 37, 5, (3 << 24) | 17), 0x0123456789ABCDEF),
    ((0x243F6A88, 0x85A308D3, 0x13198A2E, 0x03707344), 0x299F31D0A4093822),
]

_TRITON_SCRIPT = textwrap.dedent("""
    import json, os, sys
    os.environ["TRITON_INTERPRET"] = "1"
    import torch
    import triton
    import triton.language as tl

    @triton.jit
    def k(out_ptr, cin_ptr, seed_lo, seed_hi):
        c0 = tl.load(cin_ptr + 0)
        c1 = tl.load(cin_ptr + 1)
        c2 = tl.load(cin_ptr + 2)
        c3 = tl.load(cin_ptr + 3)
        seed = (seed_hi.to(tl.uint64) << 32) | seed_lo.to(tl.uint64)
        a, b, c, d = tl.philox(seed, c0, c1, c2, c3, 10)
        tl.store(out_ptr + 0, a.to(tl.int32, bitcast=True))
        tl.store(out_ptr + 1, b.to(tl.int32, bitcast=True))
        tl.store(out_ptr + 2, c.to(tl.int32, bitcast=True))
        tl.store(out_ptr + 3, d.to(tl.int32, bitcast=True))

    res = []
    for ctr, seed in json.loads(sys.argv[1]):
        cin = torch.tensor([c - (1 << 32) if c >= (1 << 31) else c
                            for c in ctr], dtype=torch.int32)
        out = torch.zeros(4, dtype=torch.int32)
        lo, hi = seed & 0xFFFFFFFF, seed >> 32
        k[(1,)](out, cin, lo, hi)
        res.append([x & 0xFFFFFFFF for x in out.tolist()])
    print(json.dumps(res))
""")


def test_philox_matches_triton_interpreter():
    """Philox4x32-10 equals Triton's own implementation, run on the CPU."""
    pytest.importorskip("triton")
    env = dict(os.environ, TRITON_INTERPRET="1")
    arg = json.dumps([[list(c), s] for c, s in CASES])
    proc = subprocess.run([sys.executable, "-c", _TRITON_SCRIPT, arg],
                          capture_output=True, text=True, env=env, timeout=300)
    if proc.returncode != 0:
        pytest.skip("triton interpreter unavailable: " + proc.stderr[-300:])
    ref = json.loads(proc.stdout.strip().splitlines()[-1])
    for (ctr, seed), want in zip(CASES, ref):
        key = (seed & 0xFFFFFFFF, seed >> 32)
        assert list(philox4x32_10(ctr, key)) == want, (ctr, seed)


def test_uniform_open_interval_and_exact_in_fp32():
    for w in (0, 1, 511, 512, 0x7FFFFFFF, 0xFFFFFE00, 0xFFFFFFFF):
        u = word_to_uniform(w)
        assert 0.0 < u < 1.0
        assert float(np.float32(u)) == u
    assert word_to_uniform(0) == 2.0 ** -24
    assert word_to_uniform(0xFFFFFFFF) == 1.0 - 2.0 ** -24


def test_decision_uniforms_are_distinct_across_streams_rounds_positions():
    us = set()
    for stream in range(4):
        for rnd in range(3):
            for pos in range(5):
                for seq in range(3):
                    us.add(decision_uniform(7, stream, rnd, seq, pos))
    assert len(us) == 4 * 3 * 5 * 3


def test_uniforms_are_uniform():
    """Kolmogorov-Smirnov check of 4000 decision uniforms."""
    from scipy import stats
    u = [decision_uniform(99, 1, 0, 3, p) for p in range(4000)]
    assert stats.kstest(u, "uniform").pvalue > 1e-3
