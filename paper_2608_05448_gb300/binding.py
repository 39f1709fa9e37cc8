"""ctypes binding of libdblast (include/dblast.h).

Argument marshalling only: torch tensors are checked for device, dtype and
layout and passed as raw device pointers with the current CUDA stream; every
step of the computation runs in the library's CUDA kernels.  There is no CPU
fallback: if the library cannot be loaded, importing this module raises.
"""
import ctypes
import os

import torch

from . import build as _build

DBLAST_OK = 0
STATUS_NAMES = {0: "ok", 1: "invalid argument", 2: "unsupported",
                3: "workspace", 4: "cuda", 5: "timeout", 6: "no device", 7: "bounds"}
DTYPES = {torch.bfloat16: 0, torch.float32: 1}
IMPLS = {"auto": 0, "simt": 1, "tcgen05": 2}
MODES = {"soft": 0, "greedy": 1}

TIE_ZHAT, TIE_DRAFT, TIE_ACCEPT, TIE_RESID, TIE_RMASS, TIE_TOPP = 1, 2, 4, 8, 16, 32


class DBLastError(RuntimeError):
    def __init__(self, status, where):
        self.status = status
        super().__init__("%s failed: %s (%d)" % (where, STATUS_NAMES.get(status, "?"),
                                                 status))


class CHead(ctypes.Structure):
    _fields_ = [("V", ctypes.c_int), ("H", ctypes.c_int), ("K", ctypes.c_int),
                ("r", ctypes.c_int), ("dtype", ctypes.c_int),
                ("W", ctypes.c_void_p), ("U", ctypes.c_void_p),
                ("Vf", ctypes.c_void_p), ("e", ctypes.c_void_p),
                ("Wp", ctypes.c_void_p), ("bp", ctypes.c_void_p),
                ("vbias", ctypes.c_void_p), ("prep", ctypes.c_void_p),
                ("prep_bytes", ctypes.c_size_t)]


class CBlockArgs(ctypes.Structure):
    _fields_ = [("N", ctypes.c_int), ("B", ctypes.c_int),
                ("temperature", ctypes.c_float), ("z_temperature", ctypes.c_float),
                ("seed", ctypes.c_uint64), ("hidden", ctypes.c_void_p),
                ("anchor", ctypes.c_void_p), ("pos", ctypes.c_void_p),
                ("round", ctypes.c_void_p), ("impl", ctypes.c_int),
                ("mode", ctypes.c_int)]


class CDraftOut(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in
                ("z_hat", "pi", "tokens", "lse", "logw", "q_tok", "branch_tokens")]


class CAlArgs(ctypes.Structure):
    _fields_ = [("tokens", ctypes.c_void_p), ("target", ctypes.c_void_p),
                ("has_bonus", ctypes.c_int), ("top_k", ctypes.c_int), ("top_p", ctypes.c_float),
                ("tau", ctypes.c_float)] + [
        (n, ctypes.c_void_p) for n in ("nll", "j_al", "l_tau", "r", "S", "accept_prob",
                                       "q_cond", "p_tok", "tie_flags")]


class CStats(ctypes.Structure):
    _fields_ = [("calls", ctypes.c_uint64), ("kernel_launches", ctypes.c_uint64),
                ("tc_launches", ctypes.c_uint64),
                ("timed_draft", ctypes.c_uint64), ("timed_verify", ctypes.c_uint64),
                ("draft_pass_ms", ctypes.c_double), ("verify_pass_ms", ctypes.c_double)]


class CVerifyOut(ctypes.Structure):
    _fields_ = [("target", ctypes.c_void_p), ("has_bonus", ctypes.c_int)] + [
        (n, ctypes.c_void_p) for n in
        ("p_tok", "accept_prob", "alpha", "lse_target", "accepted", "emitted",
         "n_emitted", "exp_len", "alpha_len", "tie_flags", "collision", "determinism")] + [
        ("top_k", ctypes.c_int), ("top_p", ctypes.c_float)]
    POINTERS = 12  # the output pointers after (target, has_bonus)


EXPORTS = ["dblast_prep_bytes", "dblast_workspace_bytes", "dblast_head_prepare",
           "dblast_draft_block", "dblast_verify_block", "dblast_draft_and_verify",
           "dblast_device_status", "dblast_set_wait_limit", "dblast_set_checks", "dblast_stats_reset",
           "dblast_stats_get", "dblast_target_lse_noalloc", "dblast_status_string",
           "dblast_version", "dblast_determinism_workspace_bytes", "dblast_target_determinism",
           "dblast_al_objective"]


def load_library(path=None, build_if_missing=True):
    """Load libdblast.so (building it first when it is missing or stale)."""
    if path is None:
        path = _build.LIB
        if build_if_missing and not _build.up_to_date():
            _build.build()
    if not os.path.exists(path):
        raise ImportError("libdblast.so not found at %s; run the build first" % path)
    lib = ctypes.CDLL(path)
    P, S = ctypes.POINTER, ctypes.c_size_t
    lib.dblast_prep_bytes.argtypes = [P(CHead)]
    lib.dblast_prep_bytes.restype = S
    lib.dblast_workspace_bytes.argtypes = [P(CHead), ctypes.c_int, ctypes.c_int, ctypes.c_int]
    lib.dblast_workspace_bytes.restype = S
    lib.dblast_head_prepare.argtypes = [P(CHead), ctypes.c_void_p]
    lib.dblast_head_prepare.restype = ctypes.c_int
    lib.dblast_draft_block.argtypes = [P(CHead), P(CBlockArgs), P(CDraftOut),
                                       ctypes.c_void_p, S, ctypes.c_void_p]
    lib.dblast_draft_block.restype = ctypes.c_int
    lib.dblast_verify_block.argtypes = [P(CHead), P(CBlockArgs), P(CVerifyOut),
                                        ctypes.c_void_p, S, ctypes.c_void_p]
    lib.dblast_verify_block.restype = ctypes.c_int
    lib.dblast_draft_and_verify.argtypes = [P(CHead), P(CBlockArgs), P(CDraftOut),
                                            P(CVerifyOut), ctypes.c_void_p, S,
                                            ctypes.c_void_p]
    lib.dblast_draft_and_verify.restype = ctypes.c_int
    lib.dblast_device_status.argtypes = [ctypes.c_void_p, ctypes.c_void_p]
    lib.dblast_device_status.restype = ctypes.c_int
    lib.dblast_set_wait_limit.argtypes = [ctypes.c_uint32]
    lib.dblast_set_wait_limit.restype = None
    lib.dblast_set_checks.argtypes = [ctypes.c_int]
    lib.dblast_set_checks.restype = None
    lib.dblast_stats_reset.argtypes = [ctypes.c_int]
    lib.dblast_stats_reset.restype = None
    lib.dblast_stats_get.argtypes = [P(CStats)]
    lib.dblast_stats_get.restype = ctypes.c_int
    lib.dblast_target_lse_noalloc.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_int,
                                              ctypes.c_int, ctypes.c_float, ctypes.c_void_p,
                                              ctypes.c_void_p]
    lib.dblast_target_lse_noalloc.restype = ctypes.c_int
    lib.dblast_al_objective.argtypes = [P(CHead), P(CBlockArgs), P(CAlArgs), ctypes.c_void_p, S,
                                        ctypes.c_void_p]
    lib.dblast_al_objective.restype = ctypes.c_int
    lib.dblast_determinism_workspace_bytes.argtypes = [ctypes.c_int] * 5
    lib.dblast_determinism_workspace_bytes.restype = S
    lib.dblast_target_determinism.argtypes = [
        ctypes.c_void_p, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
        ctypes.c_float, ctypes.c_int, ctypes.c_uint64, ctypes.c_void_p, ctypes.c_void_p,
        ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, S, ctypes.c_void_p]
    lib.dblast_target_determinism.restype = ctypes.c_int
    lib.dblast_status_string.argtypes = [ctypes.c_int]
    lib.dblast_status_string.restype = ctypes.c_char_p
    lib.dblast_version.argtypes = []
    lib.dblast_version.restype = ctypes.c_char_p
    return lib


_LIB = None


def lib():
    global _LIB
    if _LIB is None:
        _LIB = load_library()
    return _LIB


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream():
    return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)


def _check(status, where):
    if status != DBLAST_OK:
        raise DBLastError(status, where)


def _cuda_contig(t, name, dtype=None):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("%s must be a CUDA tensor" % name)
    if dtype is not None and t.dtype != dtype:
        raise ValueError("%s must be %s, got %s" % (name, dtype, t.dtype))
    if not t.is_contiguous():
        raise ValueError("%s must be contiguous" % name)
    return t


class Head:
    """Drafter head on the device plus its prep buffer (dblast_head_prepare)."""

    def __init__(self, W, U, Vf, Wp, bp=None, e=None, vbias=None, prepare=True):
        dt = W.dtype
        if dt not in DTYPES:
            raise ValueError("head dtype must be bf16 or fp32")
        V, H = W.shape
        K, H2, r = U.shape
        if H2 != H or tuple(Vf.shape) != (K, H, r) or tuple(Wp.shape) != (K, H):
            raise ValueError("inconsistent head shapes")
        self.tensors = dict(W=_cuda_contig(W, "W", dt), U=_cuda_contig(U, "U", dt),
                            Vf=_cuda_contig(Vf, "Vf", dt), Wp=_cuda_contig(Wp, "Wp", dt),
                            e=_cuda_contig(e, "e", dt),
                            bp=_cuda_contig(bp, "bp", torch.float32),
                            vbias=_cuda_contig(vbias, "vbias", torch.float32))
        self.V, self.H, self.K, self.r, self.dtype = V, H, K, r, dt
        self.c = CHead(V, H, K, r, DTYPES[dt], *[_ptr(self.tensors[k]) for k in
                                                  ("W", "U", "Vf", "e", "Wp", "bp",
                                                   "vbias")], None, 0)
        nbytes = lib().dblast_prep_bytes(ctypes.byref(self.c))
        self.prep = torch.empty(nbytes, dtype=torch.uint8, device=W.device)
        self.c.prep = self.prep.data_ptr()
        self.c.prep_bytes = nbytes
        if prepare:
            _check(lib().dblast_head_prepare(ctypes.byref(self.c), _stream()),
                   "dblast_head_prepare")

    @classmethod
    def from_dict(cls, d, **kw):
        return cls(d["W"], d["U"], d["Vf"], d["Wp"], bp=d.get("bp"), e=d.get("e"),
                   vbias=d.get("vbias"), **kw)

    def workspace_bytes(self, N, B, has_bonus=True):
        return lib().dblast_workspace_bytes(ctypes.byref(self.c), N, B, int(has_bonus))


class Workspace:
    """Caller-owned scratch buffer for N sequences of block B."""

    def __init__(self, head, N, B, has_bonus=True, device=None):
        self.nbytes = head.workspace_bytes(N, B, has_bonus)
        self.buf = torch.zeros(self.nbytes, dtype=torch.uint8,
                               device=device or head.tensors["W"].device)
        self.N, self.B = N, B

    @property
    def ptr(self):
        return ctypes.c_void_p(self.buf.data_ptr())


def _block_args(head, hidden, pos, round_, T, Z_T, seed, anchor, impl, mode="soft"):
    N, B, H = hidden.shape
    if H != head.H:
        raise ValueError("hidden size mismatch")
    _cuda_contig(hidden, "hidden", head.dtype)
    _cuda_contig(anchor, "anchor", head.dtype)
    _cuda_contig(pos, "pos", torch.int64)
    if round_.dtype not in (torch.int32, getattr(torch, "uint32", torch.int32)):
        raise ValueError("round must be int32/uint32")
    _cuda_contig(round_, "round")
    return CBlockArgs(N, B, float(T), float(Z_T), int(seed) & ((1 << 64) - 1),
                      _ptr(hidden), _ptr(anchor), _ptr(pos), _ptr(round_), IMPLS[impl],
                      MODES[mode])


def alloc_draft_out(N, B, K, device, mode="soft"):
    """Draft outputs; "lse" only in soft mode, "branch_tokens" only in greedy mode."""
    f, i = torch.float32, torch.int32
    out = dict(z_hat=torch.empty(N, dtype=i, device=device),
               pi=torch.empty(N, K, dtype=f, device=device),
               tokens=torch.empty(N, B, dtype=i, device=device),
               logw=torch.empty(N, B, K, dtype=f, device=device),
               q_tok=torch.empty(N, B, dtype=f, device=device))
    if mode == "greedy":
        out["branch_tokens"] = torch.empty(N, B, K, dtype=i, device=device)
    else:
        out["lse"] = torch.empty(N, B, K, dtype=f, device=device)
    return out


def alloc_verify_out(N, B, has_bonus, device):
    f, i = torch.float32, torch.int32
    Bt = B + int(has_bonus)
    return dict(p_tok=torch.empty(N, B, dtype=f, device=device),
                accept_prob=torch.empty(N, B, dtype=f, device=device),
                alpha=torch.empty(N, B, dtype=f, device=device),
                lse_target=torch.empty(N, Bt, dtype=f, device=device),
                accepted=torch.empty(N, dtype=i, device=device),
                emitted=torch.empty(N, B + 1, dtype=i, device=device),
                n_emitted=torch.empty(N, dtype=i, device=device),
                exp_len=torch.empty(N, dtype=f, device=device),
                alpha_len=torch.empty(N, dtype=f, device=device),
                tie_flags=torch.empty(N, dtype=i, device=device),
                collision=torch.empty(N, B, dtype=f, device=device),
                determinism=torch.empty(N, dtype=f, device=device))


def _draft_struct(d):
    if d is None:
        return CDraftOut()
    return CDraftOut(*[_ptr(d.get(k)) for k, _ in CDraftOut._fields_])


def _verify_struct(target, has_bonus, v, top_k=0, top_p=0.0):
    v = v or {}
    names = [k for k, _ in CVerifyOut._fields_[2:2 + CVerifyOut.POINTERS]]
    return CVerifyOut(_ptr(target), int(has_bonus), *[_ptr(v.get(k)) for k in names],
                      int(top_k), float(top_p))


def dblast_draft_block(head, ws, hidden, pos, round_, T, Z_T, seed, anchor=None,
                       impl="auto", out=None, mode="soft"):
    args = _block_args(head, hidden, pos, round_, T, Z_T, seed, anchor, impl, mode)
    N, B, _ = hidden.shape
    out = out if out is not None else alloc_draft_out(N, B, head.K, hidden.device, mode)
    d = _draft_struct(out)
    _check(lib().dblast_draft_block(ctypes.byref(head.c), ctypes.byref(args),
                                    ctypes.byref(d), ws.ptr, ws.nbytes, _stream()),
           "dblast_draft_block")
    return out


def dblast_verify_block(head, ws, hidden, pos, round_, T, Z_T, seed, target, has_bonus,
                        anchor=None, impl="auto", out=None, mode="soft", top_k=0, top_p=0.0):
    args = _block_args(head, hidden, pos, round_, T, Z_T, seed, anchor, impl, mode)
    N, B, _ = hidden.shape
    _cuda_contig(target, "target", head.dtype)
    if tuple(target.shape) != (N, B + int(has_bonus), head.V):
        raise ValueError("target must be [N, B + has_bonus, V]")
    out = out if out is not None else alloc_verify_out(N, B, has_bonus, hidden.device)
    v = _verify_struct(target, has_bonus, out, top_k, top_p)
    _check(lib().dblast_verify_block(ctypes.byref(head.c), ctypes.byref(args),
                                     ctypes.byref(v), ws.ptr, ws.nbytes, _stream()),
           "dblast_verify_block")
    return out


def dblast_draft_and_verify(head, ws, hidden, pos, round_, T, Z_T, seed, target,
                            has_bonus, anchor=None, impl="auto", dout=None, vout=None,
                            mode="soft", top_k=0, top_p=0.0):
    """One fused draft+verify step; returns (draft_out, verify_out) dicts.
    mode: "soft" (sampled draft tokens) or "greedy" (greedy branches);
    top_k / top_p: the target filter (0: off)."""
    args = _block_args(head, hidden, pos, round_, T, Z_T, seed, anchor, impl, mode)
    N, B, _ = hidden.shape
    _cuda_contig(target, "target", head.dtype)
    if tuple(target.shape) != (N, B + int(has_bonus), head.V):
        raise ValueError("target must be [N, B + has_bonus, V]")
    dout = dout if dout is not None else alloc_draft_out(N, B, head.K, hidden.device, mode)
    vout = vout if vout is not None else alloc_verify_out(N, B, has_bonus, hidden.device)
    d = _draft_struct(dout)
    v = _verify_struct(target, has_bonus, vout, top_k, top_p)
    _check(lib().dblast_draft_and_verify(ctypes.byref(head.c), ctypes.byref(args),
                                         ctypes.byref(d), ctypes.byref(v), ws.ptr,
                                         ws.nbytes, _stream()),
           "dblast_draft_and_verify")
    return dout, vout


def dblast_device_status(ws):
    return lib().dblast_device_status(ws.ptr, _stream())


def dblast_set_wait_limit(spins):
    lib().dblast_set_wait_limit(int(spins))


def dblast_set_checks(enable):
    """Device-side index checks of later calls on (True) or off."""
    lib().dblast_set_checks(1 if enable else 0)


def dblast_stats_reset(enable_pass_timing=True):
    """Zero the counters; time every n-th pass with CUDA events (True = 1,
    False = 0 = off)."""
    lib().dblast_stats_reset(int(enable_pass_timing))


def dblast_stats_get():
    st = CStats()
    _check(lib().dblast_stats_get(ctypes.byref(st)), "dblast_stats_get")
    return {k: getattr(st, k) for k, _ in CStats._fields_}


NOALLOC_MAX_RECORDS = 1 << 20


def dblast_target_lse_noalloc(target, temperature, lse_out):
    """Natural log-sum-exp of target / T per row through the no-allocation
    entry point: its only scratch is the library's static device array, and
    the caller provides the output.  target: CUDA [..., V] bf16/fp32 logits;
    lse_out: CUDA fp32 with one entry per row.  Returns the C status code."""
    _cuda_contig(target, "target")
    _cuda_contig(lse_out, "lse_out", torch.float32)
    V = target.shape[-1]
    rows = target.numel() // V
    if lse_out.numel() != rows:
        raise ValueError("lse_out must have one entry per row")
    return lib().dblast_target_lse_noalloc(_ptr(target), rows, V, DTYPES[target.dtype],
                                           float(temperature), _ptr(lse_out), _stream())


def dblast_target_determinism(target, b, temperature, M=0, seed=0, samples=False, ws=None):
    """Target-block early determinism of target logits [N, rows, V] (App. B):
    returns a dict with collision [N, b], d_exact [N] and, for M >= 1, the
    M-sample estimate d_hat [N] (and the drawn blocks [N, M, b] if samples)."""
    _cuda_contig(target, "target")
    if target.dtype not in DTYPES or target.dim() != 3:
        raise ValueError("target must be a bf16/fp32 [N, rows, V] tensor")
    N, rows, V = target.shape
    dev = target.device
    f = torch.float32
    out = dict(collision=torch.empty(N, b, dtype=f, device=dev),
               d_exact=torch.empty(N, dtype=f, device=dev))
    if M >= 1:
        out["d_hat"] = torch.empty(N, dtype=f, device=dev)
        if samples:
            out["samples"] = torch.empty(N, M, b, dtype=torch.int32, device=dev)
    nbytes = lib().dblast_determinism_workspace_bytes(N, rows, b, V, int(M))
    if ws is None or ws.numel() < nbytes:
        ws = torch.empty(max(nbytes, 1), dtype=torch.uint8, device=dev)
    _check(lib().dblast_target_determinism(
        _ptr(target), DTYPES[target.dtype], N, rows, int(b), V, float(temperature), int(M),
        int(seed) & ((1 << 64) - 1), _ptr(out["collision"]), _ptr(out["d_exact"]),
        _ptr(out.get("d_hat")), _ptr(out.get("samples")), _ptr(ws), nbytes, _stream()),
        "dblast_target_determinism")
    return out


def dblast_al_objective(head, ws, hidden, pos, round_, T, Z_T, seed, tokens, target, has_bonus,
                        tau=0.1, top_k=0, top_p=0.0, anchor=None, impl="auto"):
    """Forward pass of the training-side objectives on given target blocks
    tokens [N, B] (int32): block NLL, J_AL and its terms (r, S, l_tau, A,
    q_cond, p_tok).  Returns a dict of CUDA tensors."""
    args = _block_args(head, hidden, pos, round_, T, Z_T, seed, anchor, impl, "soft")
    N, B, _ = hidden.shape
    _cuda_contig(tokens, "tokens", torch.int32)
    _cuda_contig(target, "target", head.dtype)
    if tuple(tokens.shape) != (N, B) or tuple(target.shape) != (N, B + int(has_bonus), head.V):
        raise ValueError("tokens must be [N, B] and target [N, B + has_bonus, V]")
    dev = hidden.device
    f = torch.float32
    out = dict(nll=torch.empty(N, dtype=f, device=dev), j_al=torch.empty(N, dtype=f, device=dev),
               l_tau=torch.empty(N, dtype=torch.int32, device=dev),
               r=torch.empty(N, B, dtype=f, device=dev), S=torch.empty(N, B, dtype=f, device=dev),
               accept_prob=torch.empty(N, B, dtype=f, device=dev),
               q_cond=torch.empty(N, B, dtype=f, device=dev),
               p_tok=torch.empty(N, B, dtype=f, device=dev),
               tie_flags=torch.empty(N, dtype=torch.int32, device=dev))
    al = CAlArgs(_ptr(tokens), _ptr(target), int(has_bonus), int(top_k), float(top_p), float(tau),
                 *[_ptr(out[k]) for k, _ in CAlArgs._fields_[6:]])
    _check(lib().dblast_al_objective(ctypes.byref(head.c), ctypes.byref(args), ctypes.byref(al),
                                     ws.ptr, ws.nbytes, _stream()), "dblast_al_objective")
    return out
