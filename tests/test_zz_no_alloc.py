"""The no-allocation entry point dblast_target_lse_noalloc against the oracle.

Some callers cannot allocate device memory when they call in, for example a
plugin that runs inside another engine's enqueue step, where cudaMalloc would
synchronise the device and bypass the engine's memory pool.  This entry point
uses only a static device array inside the library.  The tests call it through
the C ABI, twice in a row on different inputs and temperatures, and compare
each result with the oracle's log-sum-exp of t / T (fp64), within the
log-sum-exp tolerance of the parity tests; and, in a process of its own, once
more after a cudaDeviceReset, which gives the device a new context (the
library must look the array's address up again).  This file is collected last
on purpose.
"""
import ctypes
import os
import subprocess
import sys
import textwrap

import numpy as np
import pytest
import torch

import synth
from oracle import dblast_oracle as orc

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _oracle_lse(target, T):
    t = orc.f64(target)
    return orc.logsumexp(t.reshape(-1, t.shape[-1]) / T, axis=-1)


def test_noalloc_lse_matches_oracle_on_two_calls():
    from paper_2608_05448_gb300.binding import dblast_target_lse_noalloc
    cfg = synth.config("qwen3_8b_b32", H=256, K=4, r=8, B=8, N=6)   # full vocabulary
    head = synth.make_head(cfg, "cuda")
    for T, rd in ((1.0, 0), (0.7, 1)):
        blk = synth.make_block(cfg, head, rd, "cuda")
        want = _oracle_lse(blk["target"], T)
        out = torch.full((want.size,), float("nan"), dtype=torch.float32, device="cuda")
        assert dblast_target_lse_noalloc(blk["target"], T, out) == 0
        torch.cuda.synchronize()
        got = out.cpu().double().numpy()
        assert np.all(np.abs(got - want) <= 1e-4 + 1e-5 * np.abs(want)), \
            float(np.max(np.abs(got - want)))


_RESET_SCRIPT = textwrap.dedent("""
    import ctypes, sys
    import numpy as np
    lib = ctypes.CDLL(sys.argv[1])
    rt = None
    for line in open("/proc/self/maps"):
        if "libcudart.so" in line:
            rt = ctypes.CDLL(line.split()[-1])
            break
    assert rt is not None, "libcudart not loaded by the library"
    rows, V, T = 5, 3000, 0.8
    rng = np.random.default_rng(7)
    out = []
    for call in range(2):
        t = (rng.standard_normal((rows, V)) * 3.0).astype(np.float32)
        dt, do = ctypes.c_void_p(), ctypes.c_void_p()
        assert rt.cudaMalloc(ctypes.byref(dt), ctypes.c_size_t(t.nbytes)) == 0
        assert rt.cudaMalloc(ctypes.byref(do), ctypes.c_size_t(4 * rows)) == 0
        assert rt.cudaMemcpy(dt, t.ctypes.data_as(ctypes.c_void_p), ctypes.c_size_t(t.nbytes), 1) == 0
        st = lib.dblast_target_lse_noalloc(dt, rows, V, 1, ctypes.c_float(T), do, None)
        assert st == 0, st
        assert rt.cudaDeviceSynchronize() == 0
        got = np.empty(rows, dtype=np.float32)
        assert rt.cudaMemcpy(got.ctypes.data_as(ctypes.c_void_p), do, ctypes.c_size_t(4 * rows), 2) == 0
        s = t.astype(np.float64) / T
        m = s.max(axis=1, keepdims=True)
        want = (np.log(np.exp(s - m).sum(axis=1, keepdims=True)) + m)[:, 0]
        assert np.all(np.abs(got - want) <= 1e-4 + 1e-5 * np.abs(want)), (call, got, want)
        out.append(float(got[0]))
        if call == 0:
            assert rt.cudaDeviceReset() == 0   # ends this process's context on the device
    print("reset ok", out)
""")


def test_noalloc_after_device_reset_in_a_fresh_process():
    from paper_2608_05448_gb300 import build
    r = subprocess.run([sys.executable, "-c", _RESET_SCRIPT, build.LIB], capture_output=True,
                       text=True, timeout=300, cwd=ROOT)
    assert r.returncode == 0 and "reset ok" in r.stdout, r.stdout + r.stderr


def test_noalloc_rejects_rows_beyond_the_static_scratch():
    from paper_2608_05448_gb300 import binding
    lib = binding.lib()
    fake = ctypes.c_void_p(1 << 20)   # never dereferenced: the size check comes first
    V = 151936
    rows = binding.NOALLOC_MAX_RECORDS // 1187 + 1
    assert lib.dblast_target_lse_noalloc(fake, rows, V, 0, 1.0, fake, None) == 3
    assert lib.dblast_target_lse_noalloc(fake, rows - 1, V, 0, 0.0, fake, None) == 1
