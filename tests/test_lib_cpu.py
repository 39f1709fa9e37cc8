"""Host-side checks of libdblast that need no GPU: it builds, loads, exports
every entry point declared in include/dblast.h, sizes its buffers and rejects
bad arguments before any CUDA call."""
import ctypes
import os
import re

import pytest

from paper_2608_05448_gb300 import binding as bd

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def header_functions():
    src = open(os.path.join(ROOT, "include", "dblast.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(dblast_[a-z_]+)\s*\(", src)))


def test_library_exports_every_declared_function():
    names = header_functions()
    assert len(names) >= 10
    lib = bd.lib()
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(bd.EXPORTS)
    assert lib.dblast_version().startswith(b"dblast")


def fake_head(V=151936, H=4096, K=8, r=16, e=False):
    p = ctypes.c_void_p(1 << 20)  # 16-byte aligned placeholder, never dereferenced
    return bd.CHead(V, H, K, r, 0, p, p, p, p if e else None, p, None, None, p, 0)


def test_prep_and_workspace_sizes():
    lib = bd.lib()
    h = fake_head()
    prep = lib.dblast_prep_bytes(ctypes.byref(h))
    V, K, rr = 151936, 8, 16
    assert prep >= V * K * rr * 4 + V * K * 2 * 16 * 2
    he = fake_head(e=True)
    assert lib.dblast_prep_bytes(ctypes.byref(he)) > prep   # r+1 -> padded to 32
    ws = lib.dblast_workspace_bytes(ctypes.byref(h), 32, 16, 1)
    assert ws >= 32 * 16 * V * 4            # fp32 stash of the base logits
    assert ws < 32 * 16 * V * 4 * 1.35      # everything else is small next to it
    assert lib.dblast_workspace_bytes(ctypes.byref(h), 32, 16, 0) == ws
    # a small vocabulary with many components: the stash region, which first
    # holds up to 16 split-K partials of the codes [M, K r], is sized for them
    hs = fake_head(V=3000, H=4096, K=16, r=32)
    M = 4 * 4
    assert lib.dblast_workspace_bytes(ctypes.byref(hs), 4, 4, 1) >= 16 * M * 16 * 32 * 4


def _args(N=2, B=3, T=1.0, zt=1.0):
    p = ctypes.c_void_p(1 << 20)
    return bd.CBlockArgs(N, B, T, zt, 0, p, None, p, p, 0)


@pytest.mark.parametrize("mutate,status", [
    (lambda h, a: setattr(h, "K", 0), 1),
    (lambda h, a: setattr(h, "K", 33), 1),
    (lambda h, a: setattr(h, "r", 65), 1),
    (lambda h, a: setattr(h, "H", 12), 1),
    (lambda h, a: setattr(h, "W", None), 1),
    (lambda h, a: setattr(h, "W", 1 << 20 | 4), 1),
    (lambda h, a: setattr(a, "B", 33), 1),
    (lambda h, a: setattr(a, "N", 0), 1),
    (lambda h, a: setattr(a, "temperature", 0.0), 1),
    (lambda h, a: setattr(a, "z_temperature", -1.0), 1),
    (lambda h, a: setattr(a, "hidden", None), 1),
    (lambda h, a: setattr(h, "prep_bytes", 0), 3),
    (lambda h, a: setattr(a, "mode", 2), 1),
    (lambda h, a: setattr(a, "mode", -1), 1),
])
def test_bad_arguments_are_rejected_before_launch(mutate, status):
    lib = bd.lib()
    h = fake_head(V=1000, H=64, K=4, r=8)
    h.prep_bytes = lib.dblast_prep_bytes(ctypes.byref(h))
    a = _args()
    mutate(h, a)
    d = bd.CDraftOut()
    ws = ctypes.c_void_p(1 << 20)
    got = lib.dblast_draft_block(ctypes.byref(h), ctypes.byref(a), ctypes.byref(d), ws,
                                 1 << 40, None)
    assert got == status


def test_workspace_too_small_is_rejected():
    lib = bd.lib()
    h = fake_head(V=1000, H=64, K=4, r=8)
    h.prep_bytes = lib.dblast_prep_bytes(ctypes.byref(h))
    a = _args()
    need = lib.dblast_workspace_bytes(ctypes.byref(h), 2, 3, 1)
    d = bd.CDraftOut()
    got = lib.dblast_draft_block(ctypes.byref(h), ctypes.byref(a), ctypes.byref(d),
                                 ctypes.c_void_p(1 << 20), need - 1, None)
    assert got == 3
    v = bd.CVerifyOut()
    got = lib.dblast_verify_block(ctypes.byref(h), ctypes.byref(a), ctypes.byref(v),
                                  ctypes.c_void_p(1 << 20), need, None)
    assert got == 1   # verify needs target logits


def test_status_strings():
    lib = bd.lib()
    for s in range(8):
        assert lib.dblast_status_string(s)
        assert not lib.dblast_status_string(s).startswith(b"unknown")
    assert bd.STATUS_NAMES[7] == "bounds"


def test_check_switch_is_host_only():
    # toggling the device-side index checks touches no device state
    bd.dblast_set_checks(True)
    bd.dblast_set_checks(False)


@pytest.mark.parametrize("kw,status", [
    (dict(b=0), 1), (dict(b=33, rows=40), 1), (dict(b=6, rows=5), 1),
    (dict(M=0, d_hat=True), 1), (dict(T=0.0), 1), (dict(ws_bytes=0), 3),
])
def test_determinism_bad_arguments_are_rejected_before_launch(kw, status):
    lib = bd.lib()
    a = dict(N=2, rows=5, b=4, V=100, T=1.0, M=3, d_hat=False, ws_bytes=1 << 30)
    a.update(kw)
    p = ctypes.c_void_p(1 << 20)
    got = lib.dblast_target_determinism(p, 0, a["N"], a["rows"], a["b"], a["V"], a["T"],
                                        a["M"], 0, p, p, p if a["d_hat"] else None, None, p,
                                        a["ws_bytes"], None)
    assert got == status
    assert lib.dblast_determinism_workspace_bytes(2, 17, 15, 151936, 20) > 2 * 17 * 1187 * 8


@pytest.mark.parametrize("top_k,top_p,status", [
    (-1, 0.0, 1), (0, float("nan"), 1), (0, -0.5, 1),
    (300, 0.0, 2),        # more than 256 kept tokens
    (0, 0.9, 2),          # top-p over the whole 1000-token vocabulary
    (20, 0.9, 0), (2000, 0.0, 0), (0, 1.0, 0),
])
def test_filter_arguments_are_checked_before_launch(top_k, top_p, status):
    lib = bd.lib()
    h = fake_head(V=1000, H=64, K=4, r=8)
    h.prep_bytes = lib.dblast_prep_bytes(ctypes.byref(h))
    a = _args()
    p = ctypes.c_void_p(1 << 20)
    v = bd.CVerifyOut()
    v.target = p
    v.top_k = top_k
    v.top_p = top_p
    need = lib.dblast_workspace_bytes(ctypes.byref(h), 2, 3, 1)
    # an accepted filter gets as far as the workspace check (3), with a buffer one byte short
    got = lib.dblast_verify_block(ctypes.byref(h), ctypes.byref(a), ctypes.byref(v), p,
                                  need - 1, None)
    assert got == (3 if status == 0 else status)


@pytest.mark.parametrize("mutate,status", [
    (lambda a, al: setattr(al, "tokens", None), 1),
    (lambda a, al: setattr(al, "target", None), 1),
    (lambda a, al: setattr(al, "tau", -0.1), 1),
    (lambda a, al: setattr(al, "tau", float("inf")), 1),
    (lambda a, al: setattr(a, "mode", 1), 1),        # the objectives use the soft proposal
    (lambda a, al: setattr(al, "top_k", 300), 2),
    (lambda a, al: None, 3),                          # accepted: stops at the short workspace
])
def test_al_objective_arguments_are_checked_before_launch(mutate, status):
    lib = bd.lib()
    h = fake_head(V=1000, H=64, K=4, r=8)
    h.prep_bytes = lib.dblast_prep_bytes(ctypes.byref(h))
    a = _args()
    p = ctypes.c_void_p(1 << 20)
    al = bd.CAlArgs()
    al.tokens, al.target, al.has_bonus, al.tau = p, p, 1, 0.1
    mutate(a, al)
    need = lib.dblast_workspace_bytes(ctypes.byref(h), 2, 3, 1)
    got = lib.dblast_al_objective(ctypes.byref(h), ctypes.byref(a), ctypes.byref(al), p,
                                  need - 1, None)
    assert got == status


def test_no_cluster_multicast_copies_in_the_kernels():
    # every CTA copies its own operand boxes: no bulk or tensor copy in the
    # sources uses cluster multicast (the library also runs as independent
    # replicas, one per GPU)
    csrc = os.path.join(ROOT, "paper_2608_05448_gb300", "csrc")
    for name in sorted(os.listdir(csrc)):
        if not name.endswith((".cu", ".cuh")):
            continue
        for line in open(os.path.join(csrc, name)):
            if "cp.async.bulk" in line:
                assert "multicast" not in line, (name, line.strip())
