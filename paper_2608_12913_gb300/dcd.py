"""Thin ctypes binding of libdcd.so (include/dcd.h), same entry-point names.

Argument marshalling only: every step of the verification runs in the CUDA
library.  Tensors are torch CUDA tensors (torch provides device memory and
streams); the library never sees a torch type.  There is no CPU fallback: if
the library cannot be built or loaded, or no CUDA device is present, the calls
raise.
"""

from __future__ import annotations

import ctypes
import os
import threading
from typing import Optional

import torch

from . import build as _build

DCD_OK = 0
DCD_F32, DCD_BF16 = 0, 1
DEVERR_BITS = {0x1: "bad_parent", 0x2: "bad_token", 0x4: "nonfinite", 0x8: "timeout", 0x10: "bad_param"}
MAX_NODES = 1024

_lock = threading.Lock()
_lib = None


class DcdShape(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int32), ("N", ctypes.c_int32), ("V", ctypes.c_int64),
                ("logits_dtype", ctypes.c_int32), ("flags", ctypes.c_int32),
                ("ld_logits", ctypes.c_int64), ("ld_q", ctypes.c_int64)]


class DcdError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} ({status})")


def library_path() -> str:
    return _build.LIB


def load(build_if_missing: bool = True):
    """Loads (building first if needed) libdcd.so and declares its C signatures."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        path = _build.LIB
        if build_if_missing:
            path = _build.build()
        if not os.path.exists(path):
            raise RuntimeError(f"libdcd.so is not built ({path})")
        lib = ctypes.CDLL(path)
        P, I32, U64, SZ = ctypes.c_void_p, ctypes.c_int32, ctypes.c_uint64, ctypes.c_size_t
        SH = ctypes.POINTER(DcdShape)
        lib.dcd_workspace_bytes.argtypes = [SH]
        lib.dcd_workspace_bytes.restype = SZ
        lib.dcd_verify_greedy.argtypes = [SH, P, P, P, P, P, P, P, P, P, P, P, P, P, SZ, P]
        lib.dcd_verify_sample.argtypes = [SH, P, P, P, P, P, P, P, P, U64, U64, P, P, P, P, P, P, P, P, SZ, P]
        lib.dcd_score_rows.argtypes = [SH, P, P, P, P, P, P, P, P, U64, U64, P, P, P, P, SZ, P]
        lib.dcd_verify_sample_noalloc.argtypes = [SH, P, P, P, P, P, P, P, P, U64, U64, P, P, P, P, P, P, P, P]
        lib.dcd_verify_sample_noalloc.restype = I32
        lib.dcd_score_rows_ex.argtypes = [SH, P, P, P, P, P, P, P, P, U64, U64, P, P, P, P, SZ, P,
                                          ctypes.c_int, ctypes.c_int, ctypes.c_int64]
        lib.dcd_tree_walk.argtypes = [SH, P, P, P, P, SZ, P]
        lib.dcd_upload_q_rows.argtypes = [SH, P, P, P, P, P]
        lib.dcd_upload_q_rows.restype = I32
        lib.dcd_fused_workspace_bytes.argtypes = [SH]
        lib.dcd_fused_workspace_bytes.restype = SZ
        lib.dcd_verify_fused_lmhead.argtypes = [SH, P, I32, P, P, I32, P, P, P, P, P, P, P, P, P, P, P, SZ, P]
        lib.dcd_verify_fused_lmhead_ex.argtypes = [SH, P, I32, P, P, I32, P, P, P, P, P, P, P, P, P, P, P, P, SZ,
                                                   P, P, P]
        lib.dcd_diagnostics_workspace_bytes.argtypes = [SH]
        lib.dcd_diagnostics_workspace_bytes.restype = SZ
        lib.dcd_row_diagnostics.argtypes = [SH, P, P, P, P, P, P, P, P, P, P, SZ, P]
        lib.dcd_row_diagnostics_ex.argtypes = [SH, P, P, P, P, P, P, P, P, P, P, SZ, P, P, P]
        lib.dcd_get_device_error.argtypes = [P, P, ctypes.POINTER(ctypes.c_uint32)]
        lib.dcd_status_string.argtypes = [ctypes.c_int]
        lib.dcd_status_string.restype = ctypes.c_char_p
        lib.dcd_version.restype = ctypes.c_int
        for name in ("dcd_verify_greedy", "dcd_verify_sample", "dcd_score_rows", "dcd_score_rows_ex",
                     "dcd_tree_walk", "dcd_get_device_error", "dcd_verify_fused_lmhead",
                     "dcd_verify_fused_lmhead_ex", "dcd_row_diagnostics", "dcd_row_diagnostics_ex"):
            getattr(lib, name).restype = I32
        _lib = lib
        return lib


def status_string(status: int) -> str:
    return load().dcd_status_string(int(status)).decode()


def _check(status: int, where: str):
    if status != DCD_OK:
        raise DcdError(status, where)


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _require(t, name, dtype=None, device=None, shape=None):
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch tensor")
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor (the library has no CPU path)")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if device is not None and t.device != device:
        raise ValueError(f"{name} is on {t.device}, expected {device}")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} has shape {tuple(t.shape)}, expected {tuple(shape)}")


def _logits_dtype(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return DCD_BF16
    if t.dtype == torch.float32:
        return DCD_F32
    raise TypeError(f"logits must be bfloat16 or float32, got {t.dtype}")


DCD_SIBLINGS_DISTINCT = 0x1


def make_shape(B: int, N: int, V: int, dtype: int, ld: Optional[int] = None, ldq: Optional[int] = None,
               flags: int = 0) -> DcdShape:
    return DcdShape(B, N, V, dtype, flags, V if ld is None else ld, (V if ldq is None else ldq))


def workspace_bytes(B: int, N: int, V: int, dtype: int = DCD_BF16) -> int:
    sh = make_shape(B, N, V, dtype)
    n = load().dcd_workspace_bytes(ctypes.byref(sh))
    if n == 0:
        raise ValueError("invalid shape")
    return int(n)


def alloc_workspace(B: int, N: int, V: int, device, dtype: int = DCD_BF16) -> torch.Tensor:
    ws = torch.zeros(workspace_bytes(B, N, V, dtype), dtype=torch.uint8, device=device)
    assert ws.data_ptr() % 256 == 0
    return ws


def alloc_outputs(B: int, N: int, device, V: Optional[int] = None, residual: bool = False) -> dict:
    out = dict(
        accept_len=torch.empty(B, dtype=torch.int32, device=device),
        accept_path=torch.empty((B, N), dtype=torch.int32, device=device),
        bonus=torch.empty(B, dtype=torch.int32, device=device),
        cd_logprob=torch.empty((B, N), dtype=torch.float32, device=device),
        cd_argmax=torch.empty((B, N), dtype=torch.int32, device=device),
        cd_lse=torch.empty((B, N), dtype=torch.float32, device=device),
    )
    if residual:
        out["residual"] = torch.empty((B, V), dtype=torch.float32, device=device)
    return out


def _check_outputs(o: dict, B: int, N: int, V: int, device) -> dict:
    """A caller's output tensors: each must have the dtype, device and shape the library writes, and
    be contiguous (the library writes them as dense arrays)."""
    specs = {"accept_len": (torch.int32, (B,)), "accept_path": (torch.int32, (B, N)), "bonus": (torch.int32, (B,)),
             "cd_logprob": (torch.float32, (B, N)), "cd_argmax": (torch.int32, (B, N)),
             "cd_lse": (torch.float32, (B, N)), "residual": (torch.float32, (B, V))}
    for k in ("accept_len", "accept_path", "bonus"):
        if k not in o:
            raise ValueError(f"out must hold {k!r}")
    for k, t in o.items():
        if k in specs:
            dtype, shape = specs[k]
            _require(t, f"out[{k!r}]", dtype, device, shape)
            if not t.is_contiguous():
                raise ValueError(f"out[{k!r}] must be contiguous")
    return o


def _require_vec(t, name, B: int, device):
    _require(t, name, torch.float32, device, (B,))
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")


class _Call:
    """Validated arguments of one verification call."""

    def __init__(self, z_exp, z_ama, tokens, parents, alpha, beta, q=None, temperature=None, distinct=False):
        _require(z_exp, "z_exp")
        dev = z_exp.device
        if z_exp.dim() != 2 or z_exp.stride(1) != 1:
            raise ValueError("z_exp must be a 2-D tensor with unit stride along the vocabulary")
        _require(z_ama, "z_ama", dtype=z_exp.dtype, device=dev, shape=z_exp.shape)
        if z_ama.stride() != z_exp.stride():
            raise ValueError("z_exp and z_ama must share one row stride")
        _require(tokens, "tokens", dtype=torch.int32, device=dev)
        if tokens.dim() != 2 or not tokens.is_contiguous():
            raise ValueError("tokens must be a contiguous [B, N] int32 tensor")
        B, N = tokens.shape
        V = z_exp.shape[1]
        if z_exp.shape[0] != B * N:
            raise ValueError(f"z_exp has {z_exp.shape[0]} rows, expected B*N = {B * N}")
        _require(parents, "parents", dtype=torch.int32, device=dev, shape=(B, N))
        if not parents.is_contiguous():
            raise ValueError("parents must be contiguous")
        _require_vec(alpha, "alpha", B, dev)
        if beta is not None:
            _require_vec(beta, "beta", B, dev)
        ldq = None
        if q is not None:
            _require(q, "q", dtype=torch.float32, device=dev)
            if q.dim() != 2 or q.shape[0] != B * N or q.shape[1] != V or q.stride(1) != 1:
                raise ValueError("q must be a [B*N, V] float32 tensor with unit stride along the vocabulary")
            ldq = q.stride(0)
        if temperature is not None:
            _require_vec(temperature, "temperature", B, dev)
        self.device = dev
        self.B, self.N, self.V = B, N, V
        self.shape = make_shape(B, N, V, _logits_dtype(z_exp), z_exp.stride(0), ldq,
                                DCD_SIBLINGS_DISTINCT if distinct else 0)
        self.args = (z_exp, z_ama, q, tokens, parents, alpha, beta, temperature)

    def workspace(self, workspace):
        need = load().dcd_workspace_bytes(ctypes.byref(self.shape))
        if workspace is None:
            return torch.empty(need, dtype=torch.uint8, device=self.device)
        _require(workspace, "workspace", dtype=torch.uint8, device=self.device)
        if workspace.numel() < need:
            raise ValueError(f"workspace has {workspace.numel()} bytes, needs {need}")
        return workspace

    def outputs(self, out, residual=False):
        if out is None:
            return alloc_outputs(self.B, self.N, self.device, self.V, residual)
        return _check_outputs(out, self.B, self.N, self.V, self.device)


def dcd_verify_greedy(z_exp, z_ama, tokens, parents, alpha, beta=None, *, out=None, workspace=None,
                      stream=None) -> dict:
    """Greedy CD verification; returns accept_len, accept_path, bonus, cd_logprob, cd_argmax, cd_lse."""
    c = _Call(z_exp, z_ama, tokens, parents, alpha, beta)
    ws = c.workspace(workspace)
    o = c.outputs(out)
    st = load().dcd_verify_greedy(
        ctypes.byref(c.shape), _ptr(z_exp), _ptr(z_ama), _ptr(tokens), _ptr(parents), _ptr(alpha), _ptr(beta),
        _ptr(o["accept_len"]), _ptr(o["accept_path"]), _ptr(o["bonus"]), _ptr(o.get("cd_logprob")),
        _ptr(o.get("cd_argmax")), _ptr(o.get("cd_lse")), _ptr(ws), ws.numel(), _stream(stream))
    _check(st, "dcd_verify_greedy")
    o["workspace"] = ws
    return o


def dcd_verify_sample(z_exp, z_ama, q, tokens, parents, alpha, temperature, seed: int, offset: int, beta=None, *,
                      residual: bool = False, out=None, workspace=None, stream=None, distinct: bool = False) -> dict:
    """Speculative-sampling CD verification (greedy for sequences with temperature 0)."""
    c = _Call(z_exp, z_ama, tokens, parents, alpha, beta, q=q, temperature=temperature, distinct=distinct)
    ws = c.workspace(workspace)
    o = c.outputs(out, residual=residual)
    st = load().dcd_verify_sample(
        ctypes.byref(c.shape), _ptr(z_exp), _ptr(z_ama), _ptr(q), _ptr(tokens), _ptr(parents), _ptr(alpha),
        _ptr(beta), _ptr(temperature), int(seed) & (2 ** 64 - 1), int(offset) & (2 ** 64 - 1),
        _ptr(o["accept_len"]), _ptr(o["accept_path"]), _ptr(o["bonus"]), _ptr(o.get("cd_logprob")),
        _ptr(o.get("cd_argmax")), _ptr(o.get("cd_lse")), _ptr(o.get("residual") if residual else None), _ptr(ws),
        ws.numel(), _stream(stream))
    _check(st, "dcd_verify_sample")
    o["workspace"] = ws
    return o


def dcd_verify_sample_noalloc(z_exp, z_ama, q, tokens, parents, alpha, temperature, seed: int, offset: int,
                              beta=None, *, residual: bool = False, out=None, stream=None, distinct: bool = False) -> dict:
    """dcd_verify_sample with the library's built-in scratch instead of a caller workspace.

    For callers that cannot allocate device memory (see include/dcd.h).  Calls that overlap on the
    GPU share that scratch and race; the caller serialises them.
    """
    c = _Call(z_exp, z_ama, tokens, parents, alpha, beta, q=q, temperature=temperature, distinct=distinct)
    o = c.outputs(out, residual=residual)
    st = load().dcd_verify_sample_noalloc(
        ctypes.byref(c.shape), _ptr(z_exp), _ptr(z_ama), _ptr(q), _ptr(tokens), _ptr(parents), _ptr(alpha),
        _ptr(beta), _ptr(temperature), int(seed) & (2 ** 64 - 1), int(offset) & (2 ** 64 - 1),
        _ptr(o["accept_len"]), _ptr(o["accept_path"]), _ptr(o["bonus"]), _ptr(o.get("cd_logprob")),
        _ptr(o.get("cd_argmax")), _ptr(o.get("cd_lse")), _ptr(o.get("residual") if residual else None),
        _stream(stream))
    _check(st, "dcd_verify_sample_noalloc")
    return o


def dcd_score_rows(z_exp, z_ama, tokens, parents, alpha, beta=None, q=None, temperature=None, seed: int = 0,
                   offset: int = 0, *, out=None, workspace=None, stream=None, stages: int = 0,
                   plain_loads: bool = False, distinct: bool = False, poll_limit_cycles: int = 0) -> dict:
    """The per-row step alone (records stay in the workspace); see dcd_tree_walk."""
    c = _Call(z_exp, z_ama, tokens, parents, alpha, beta, q=q, temperature=temperature, distinct=distinct)
    ws = c.workspace(workspace)
    o = c.outputs(out)
    lib = load()
    common = (ctypes.byref(c.shape), _ptr(z_exp), _ptr(z_ama), _ptr(q), _ptr(tokens), _ptr(parents), _ptr(alpha),
              _ptr(beta), _ptr(temperature), int(seed) & (2 ** 64 - 1), int(offset) & (2 ** 64 - 1),
              _ptr(o.get("cd_logprob")), _ptr(o.get("cd_argmax")), _ptr(o.get("cd_lse")), _ptr(ws), ws.numel(),
              _stream(stream))
    if stages or plain_loads or poll_limit_cycles:
        st = lib.dcd_score_rows_ex(*common, int(stages), int(bool(plain_loads)), int(poll_limit_cycles))
    else:
        st = lib.dcd_score_rows(*common)
    _check(st, "dcd_score_rows")
    o["workspace"] = ws
    return o


def dcd_tree_walk(B: int, N: int, V: int, out: dict, workspace, stream=None) -> dict:
    """Tree walk over the records a previous dcd_score_rows left in `workspace`."""
    sh = make_shape(B, N, V, DCD_BF16)
    st = load().dcd_tree_walk(ctypes.byref(sh), _ptr(out["accept_len"]), _ptr(out["accept_path"]),
                              _ptr(out["bonus"]), _ptr(workspace), workspace.numel(), _stream(stream))
    _check(st, "dcd_tree_walk")
    return out


def fused_workspace_bytes(B: int, N: int, V: int) -> int:
    sh = make_shape(B, N, V, DCD_BF16)
    n = load().dcd_fused_workspace_bytes(ctypes.byref(sh))
    if n == 0:
        raise ValueError("invalid shape")
    return int(n)


def dcd_verify_fused_lmhead(h_exp, w_exp, h_ama, w_ama, tokens, parents, alpha, beta=None, *, out=None,
                            workspace=None, stream=None, gemm_events=None) -> dict:
    """Greedy CD verification fused with the two LM heads (logits h W^T never materialised).

    h_exp [B*N, H_exp], w_exp [V, H_exp], h_ama [B*N, H_ama], w_ama [V, H_ama]: bf16, row-major.
    beta: fp32 [B] plausibility thresholds (two tensor-core sweeps) or None (beta = 0, one sweep).
    Returns accept_len, accept_path, bonus, cd_logprob, cd_argmax, cd_lse (and the workspace).
    `gemm_events` = (start, stop) torch.cuda.Event pair recorded around the tensor-core sweeps.
    """
    _require(h_exp, "h_exp", dtype=torch.bfloat16)
    dev = h_exp.device
    for t, name in ((h_exp, "h_exp"), (w_exp, "w_exp"), (h_ama, "h_ama"), (w_ama, "w_ama")):
        _require(t, name, dtype=torch.bfloat16, device=dev)
        if t.dim() != 2 or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous 2-D tensor")
    B, N = tokens.shape
    R, H_exp = h_exp.shape
    V = w_exp.shape[0]
    H_ama = h_ama.shape[1]
    if R != B * N or h_ama.shape[0] != R or tuple(w_exp.shape) != (V, H_exp) or tuple(w_ama.shape) != (V, H_ama):
        raise ValueError("inconsistent shapes for the fused LM-head call")
    _require(tokens, "tokens", torch.int32, dev)
    if tokens.dim() != 2 or not tokens.is_contiguous():
        raise ValueError("tokens must be a contiguous [B, N] int32 tensor")
    _require(parents, "parents", torch.int32, dev, (B, N))
    if not parents.is_contiguous():
        raise ValueError("parents must be contiguous")
    _require_vec(alpha, "alpha", B, dev)
    if beta is not None:
        _require_vec(beta, "beta", B, dev)
    sh = make_shape(B, N, V, DCD_BF16)
    if workspace is None:
        workspace = torch.empty(fused_workspace_bytes(B, N, V), dtype=torch.uint8, device=dev)
    o = alloc_outputs(B, N, dev) if out is None else _check_outputs(out, B, N, V, dev)
    ev0 = ev1 = None
    if gemm_events is not None:
        for e in gemm_events:
            if not e.cuda_event:  # torch creates the event at its first record
                e.record()
        ev0, ev1 = (ctypes.c_void_p(e.cuda_event) for e in gemm_events)
    st = load().dcd_verify_fused_lmhead_ex(
        ctypes.byref(sh), _ptr(h_exp), H_exp, _ptr(w_exp), _ptr(h_ama), H_ama, _ptr(w_ama), _ptr(tokens),
        _ptr(parents), _ptr(alpha), _ptr(beta), _ptr(o["accept_len"]), _ptr(o["accept_path"]), _ptr(o["bonus"]),
        _ptr(o.get("cd_logprob")), _ptr(o.get("cd_argmax")), _ptr(o.get("cd_lse")), _ptr(workspace),
        workspace.numel(), _stream(stream), ev0, ev1)
    _check(st, "dcd_verify_fused_lmhead")
    o["workspace"] = workspace
    return o




def diagnostics_workspace_bytes(B: int, N: int, V: int) -> int:
    sh = make_shape(B, N, V, DCD_BF16)
    n = load().dcd_diagnostics_workspace_bytes(ctypes.byref(sh))
    if n == 0:
        raise ValueError("invalid shape")
    return int(n)


DIAG_COLS = 8
DIAG_FIELDS = ("lse_p", "lse_q", "signal", "e_q", "e_e", "kl_e_p", "kl_p_q", "kl_p_cd")


def dcd_row_diagnostics(z_exp, z_ama, B: int, N: int, *, q=None, xstar=None, cd_lse=None, alpha=None, beta=None,
                        temperature=None, out=None, workspace=None, stream=None, pass_events=None) -> torch.Tensor:
    """Per-row diagnostics [B*N, 8] (columns DIAG_FIELDS): lse_p, lse_q, the signal
    |log pi_p(x*) - log pi_q(x*)| at x* = xstar (the CD argmax), E_{pi_q}[log pi_p - log pi_q],
    with the drafter's distribution q: E_q[log pi_p - log pi_q] and D_KL(q || pi_p); then
    D_KL(pi_p || pi_q) and, given the verification call's cd_lse and alpha (and its beta and
    temperature, if any), D_KL(pi_p || pi_CD) by the decomposition lemma of App. B.

    z_exp, z_ama: [B*N, ld] bf16 or fp32 logits (row stride = their stride); q: [B*N, ldq] fp32
    or None; xstar: int32 [B*N] or [B, N], or None; cd_lse: fp32 [B*N] or [B, N], or None;
    alpha / beta / temperature: fp32 [B] or None.  `pass_events` = (start, stop) torch.cuda.Event
    pair recorded around the streaming pass.
    """
    _require(z_exp, "z_exp")
    dev = z_exp.device
    _require(z_ama, "z_ama", z_exp.dtype, dev, tuple(z_exp.shape))
    if z_exp.dim() != 2 or z_exp.stride(1) != 1 or z_ama.stride() != z_exp.stride():
        raise ValueError("z_exp / z_ama must be 2-D with unit column stride and equal strides")
    R, V = z_exp.shape
    if R != B * N:
        raise ValueError(f"z_exp has {R} rows, expected B*N = {B * N}")
    ldq = None
    if q is not None:
        _require(q, "q", torch.float32, dev)
        if q.dim() != 2 or q.shape[0] != R or q.shape[1] != V or q.stride(1) != 1:
            raise ValueError("q must be [B*N, V] with unit column stride")
        ldq = q.stride(0)
    if xstar is not None:
        _require(xstar, "xstar", torch.int32, dev)
        if xstar.numel() != R or not xstar.is_contiguous():
            raise ValueError("xstar must be a contiguous int32 tensor of B*N tokens")
    if (cd_lse is None) != (alpha is None):
        raise ValueError("cd_lse and alpha go together (the lemma of App. B needs both)")
    if cd_lse is not None:
        _require(cd_lse, "cd_lse", torch.float32, dev)
        if cd_lse.numel() != R or not cd_lse.is_contiguous():
            raise ValueError("cd_lse must be a contiguous fp32 tensor of B*N values")
        _require_vec(alpha, "alpha", B, dev)
        if beta is not None:
            _require_vec(beta, "beta", B, dev)
        if temperature is not None:
            _require_vec(temperature, "temperature", B, dev)
    sh = make_shape(B, N, V, _logits_dtype(z_exp), ld=z_exp.stride(0), ldq=ldq)
    if workspace is None:
        workspace = torch.empty(diagnostics_workspace_bytes(B, N, V), dtype=torch.uint8, device=dev)
    if out is None:
        out = torch.empty(R, DIAG_COLS, dtype=torch.float32, device=dev)
    else:
        _require(out, "out", torch.float32, dev, (R, DIAG_COLS))
        if not out.is_contiguous():
            raise ValueError("out must be contiguous")
    ev0 = ev1 = None
    if pass_events is not None:
        for e in pass_events:
            if not e.cuda_event:
                e.record()
        ev0, ev1 = (ctypes.c_void_p(e.cuda_event) for e in pass_events)
    st = load().dcd_row_diagnostics_ex(ctypes.byref(sh), _ptr(z_exp), _ptr(z_ama), _ptr(q), _ptr(xstar),
                                       _ptr(cd_lse), _ptr(alpha), _ptr(beta), _ptr(temperature), _ptr(out),
                                       _ptr(workspace), workspace.numel(), _stream(stream), ev0, ev1)
    _check(st, "dcd_row_diagnostics")
    return out


def dcd_get_device_error(workspace: torch.Tensor, stream=None) -> int:
    """Synchronises the stream and returns the device error bits of the last call on `workspace`."""
    bits = ctypes.c_uint32(0)
    st = load().dcd_get_device_error(_ptr(workspace), _stream(stream), ctypes.byref(bits))
    if st not in (DCD_OK, -6):
        raise DcdError(st, "dcd_get_device_error")
    return int(bits.value)


def version() -> int:
    return int(load().dcd_version())


def sampled_row_ranges(temperature: torch.Tensor, N: int, parents: Optional[torch.Tensor] = None) -> list:
    """Row ranges [start, stop), adjacent rows merged, of the rows whose q the kernels read: the
    rows of sequences with a positive temperature (sequence b owns rows b*N .. b*N+N-1), and of
    those, when `parents` [B, N] is given, only the rows of nodes with at least one child (a
    leaf draws its terminal token from pi_CD alone)."""
    t = temperature.detach().to("cpu").reshape(-1)
    par = None if parents is None else parents.detach().to("cpu").reshape(t.numel(), N)
    ranges = []
    for b in range(t.numel()):
        if not float(t[b]) > 0.0:
            continue
        if par is None:
            rows = range(b * N, (b + 1) * N)
        else:
            has_child = torch.zeros(N, dtype=torch.bool)
            p = par[b, 1:].long()
            has_child[p[(p >= 0) & (p < N)]] = True
            rows = (b * N + n for n in range(N) if bool(has_child[n]))
        for g in rows:
            if ranges and ranges[-1][1] == g:
                ranges[-1][1] = g + 1
            else:
                ranges.append([g, g + 1])
    return [tuple(r) for r in ranges]


def upload_inputs(host: dict, dst: dict, N: int, stream=None) -> int:
    """Copies one call's inputs from host tensors (pinned, for asynchronous copies) into the
    matching device tensors on `stream`, and returns the bytes copied.  Every tensor is copied whole
    except ``q``, of which only the rows the verification reads are copied (sampled_row_ranges:
    rows of sampled sequences whose node has a child); the other rows may hold anything on the
    device.  `host` must hold ``temperature`` and ``parents`` when it holds ``q``."""
    stream = stream if stream is not None else torch.cuda.current_stream()
    nbytes = 0
    with torch.cuda.stream(stream):
        for k, h in host.items():
            if k != "q" and h is not None:
                dst[k].copy_(h, non_blocking=True)
                nbytes += h.numel() * h.element_size()
    h = host.get("q")
    if h is not None:
        ranges = sampled_row_ranges(host["temperature"], N, host["parents"])
        nbytes += sum(r1 - r0 for r0, r1 in ranges) * h.shape[1] * h.element_size()
        d = dst["q"]
        if h.is_pinned() and h.dim() == 2 and h.stride(1) == 1 and d.stride() == h.stride():
            # one launch: the SMs read the rows through the pinned buffer's device mapping (after
            # parents and temperature, copied above on the same stream)
            B = host["temperature"].numel()
            sh = make_shape(B, N, h.shape[1], DCD_BF16, ldq=h.stride(0))
            st = load().dcd_upload_q_rows(ctypes.byref(sh), ctypes.c_void_p(h.data_ptr()), _ptr(d),
                                          _ptr(dst["parents"]), _ptr(dst["temperature"]), _stream(stream))
            _check(st, "dcd_upload_q_rows")
        else:
            with torch.cuda.stream(stream):
                for r0, r1 in ranges:
                    d[r0:r1].copy_(h[r0:r1], non_blocking=True)
    return nbytes
