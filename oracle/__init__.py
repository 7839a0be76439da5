"""CPU oracle of the CD verification step (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline leg
may import this package.  The product path (the CUDA library and its binding)
never imports it and shares no code with it.

The arithmetic lives in ``dcd_oracle.c`` (plain fp64 C, OpenMP over rows); this
module compiles it with gcc on first use and wraps it with ctypes.

Parity status of each function (what pins it, see tests/test_oracle_pins.py):
* ``row_logpi``   -- pinned: product-form brute force of Eq. 1, alpha = 0 reduces to
                     log-softmax, KL-decomposition lemma (App. B), mask invariants.
* ``row_chain``   -- pinned: exact enumeration of the lossless theorem (App. B.3).
* ``verify``      -- pinned: greedy paths fixed by construction, chain reduction to
                     Algorithm 1, Monte-Carlo lossless check, T -> 0 limit.
* ``philox``      -- pinned: Random123 known-answer vectors (tests/golden).
"""

from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "dcd_oracle.c")
_LIB_PATH = os.path.join(_HERE, "_build", "libdcd_oracle.so")
_lock = threading.Lock()
_lib = None

DTYPE_CODE = {"f32": 0, "bf16": 1, "f64": 2}


class OracleRow(ctypes.Structure):
    _fields_ = [
        ("cd_lse", ctypes.c_double),
        ("log_zcd", ctypes.c_double),
        ("gap_argmax", ctypes.c_double),
        ("gap_mask", ctypes.c_double),
        ("gap_accept", ctypes.c_double),
        ("gap_race", ctypes.c_double),
        ("argmax", ctypes.c_int32),
        ("acc_child", ctypes.c_int32),
        ("term_token", ctypes.c_int32),
        ("n_tests", ctypes.c_int32),
    ]


ROW_DTYPE = np.dtype([
    ("cd_lse", np.float64), ("log_zcd", np.float64), ("gap_argmax", np.float64),
    ("gap_mask", np.float64), ("gap_accept", np.float64), ("gap_race", np.float64),
    ("argmax", np.int32), ("acc_child", np.int32), ("term_token", np.int32), ("n_tests", np.int32),
])
assert ROW_DTYPE.itemsize == ctypes.sizeof(OracleRow)


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (OpenMP when available); returns the library path."""
    os.makedirs(os.path.dirname(_LIB_PATH), exist_ok=True)
    if not force and os.path.exists(_LIB_PATH) and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC):
        return _LIB_PATH
    base = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", _SRC, "-lm", "-o", _LIB_PATH + ".tmp"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True, capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(_LIB_PATH + ".tmp", _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P, I32, I64, U64, D = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_uint64, ctypes.c_double
            lib.dcd_oracle_philox4x32_10.argtypes = [P, P, P]
            lib.dcd_oracle_u01.argtypes = [ctypes.c_uint32]
            lib.dcd_oracle_u01.restype = D
            lib.dcd_oracle_accept_uniform.argtypes = [U64, U64, ctypes.c_uint32]
            lib.dcd_oracle_accept_uniform.restype = D
            lib.dcd_oracle_race_uniform.argtypes = [U64, U64, ctypes.c_uint32, I64]
            lib.dcd_oracle_race_uniform.restype = D
            lib.dcd_oracle_block_uniform.argtypes = [U64, U64, ctypes.c_uint32, I64]
            lib.dcd_oracle_block_uniform.restype = D
            lib.dcd_oracle_row_logpi.argtypes = [I64, ctypes.c_int, P, P, D, D, D, P, P, P, P, P, P, P]
            lib.dcd_oracle_row_chain.argtypes = [I64, ctypes.c_int, P, P, D, D, D, P, ctypes.c_int, P, ctypes.c_int,
                                                 P, P]
            lib.dcd_oracle_verify.argtypes = [I32, I32, I64, ctypes.c_int, I64, P, P, P, P, P, P, P, P, I64,
                                              U64, U64, P, ctypes.c_int, ctypes.c_int, P, P, P, P, P, P]
            lib.dcd_oracle_max_threads.restype = ctypes.c_int
            lib.dcd_oracle_row_diagnostics.argtypes = [I64, ctypes.c_int, P, P, P, ctypes.c_int32, ctypes.c_double,
                                                       P]
            _lib = lib
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _logits(z, dtype: str) -> np.ndarray:
    """Accepts numpy arrays or torch tensors; bf16 tensors are passed as raw 16-bit patterns."""
    try:
        import torch  # noqa: WPS433 -- only for unwrapping tensors handed in by tests
        if isinstance(z, torch.Tensor):
            z = z.detach().cpu().contiguous()
            if z.dtype == torch.bfloat16:
                return z.view(torch.int16).numpy().view(np.uint16)
            z = z.numpy()
    except ImportError:
        pass
    z = np.ascontiguousarray(z)
    want = {"f32": np.float32, "bf16": np.uint16, "f64": np.float64}[dtype]
    if z.dtype != want:
        raise TypeError(f"logits dtype {z.dtype} does not match {dtype}")
    return z


def max_threads() -> int:
    return int(_load().dcd_oracle_max_threads())


def philox(ctr, key) -> np.ndarray:
    c = np.asarray(ctr, dtype=np.uint32)
    k = np.asarray(key, dtype=np.uint32)
    o = np.zeros(4, dtype=np.uint32)
    _load().dcd_oracle_philox4x32_10(_ptr(c), _ptr(k), _ptr(o))
    return o


def u01(w: int) -> float:
    return float(_load().dcd_oracle_u01(int(w) & 0xFFFFFFFF))


def accept_uniform(seed: int, offset: int, G: int) -> float:
    return float(_load().dcd_oracle_accept_uniform(seed, offset, G))


def race_uniform(seed: int, offset: int, G: int, x: int) -> float:
    return float(_load().dcd_oracle_race_uniform(seed, offset, G, x))


def block_uniform(seed: int, offset: int, G: int, k: int) -> float:
    return float(_load().dcd_oracle_block_uniform(seed, offset, G, k))


def row_logpi(zp, zq, alpha: float, beta: float = 0.0, T: float = 1.0, dtype: str = "f64") -> dict:
    """log pi_CD,T over the vocabulary of one row, plus its normalisers and argmax."""
    zp = _logits(zp, dtype)
    zq = _logits(zq, dtype)
    V = zp.shape[-1]
    out = np.empty(V, dtype=np.float64)
    vals = {k: ctypes.c_double() for k in ("lse_p", "lse_q", "log_zcd", "cd_lse", "gap_argmax")}
    arg = ctypes.c_int32()
    rc = _load().dcd_oracle_row_logpi(
        V, DTYPE_CODE[dtype], _ptr(zp), _ptr(zq), float(alpha), float(beta), float(T), _ptr(out),
        ctypes.byref(vals["lse_p"]), ctypes.byref(vals["lse_q"]), ctypes.byref(vals["log_zcd"]),
        ctypes.byref(vals["cd_lse"]), ctypes.byref(arg), ctypes.byref(vals["gap_argmax"]))
    if rc != 0:
        raise ValueError(f"oracle row_logpi failed: {rc}")
    res = {k: v.value for k, v in vals.items()}
    res["logpi"] = out
    res["argmax"] = arg.value
    return res


def row_chain(zp, zq, alpha: float, beta: float, T: float, q, child_tokens, dtype: str = "f64",
              distinct: bool = False):
    """Sibling-rejection chain run to its end: (ratios[m], final residual r_m[V]).  `distinct`:
    siblings drawn without replacement (each sees q without the earlier siblings' tokens)."""
    zp = _logits(zp, dtype)
    zq = _logits(zq, dtype)
    V = zp.shape[-1]
    q = np.ascontiguousarray(q, dtype=np.float32)
    ct = np.ascontiguousarray(child_tokens, dtype=np.int32)
    ratios = np.empty(max(1, len(ct)), dtype=np.float64)
    r = np.empty(V, dtype=np.float64)
    rc = _load().dcd_oracle_row_chain(V, DTYPE_CODE[dtype], _ptr(zp), _ptr(zq), float(alpha), float(beta),
                                      float(T), _ptr(q), len(ct), _ptr(ct), int(distinct), _ptr(ratios), _ptr(r))
    if rc != 0:
        raise ValueError(f"oracle row_chain failed: {rc}")
    return ratios[: len(ct)], r


def verify(*, B: int, N: int, V: int, dtype: str, z_exp, z_ama, tokens, parents, alpha, beta=None,
           temperature=None, q=None, seed: int = 0, offset: int = 0, ld=None, ldq=None,
           nthreads: int = 1, want_residual: bool = False, seq_ids=None, distinct: bool = False) -> dict:
    """Full verification of B sequences x N nodes (see dcd_oracle_verify in the C source)."""
    zp = _logits(z_exp, dtype)
    zq = _logits(z_ama, dtype)
    ld = V if ld is None else ld

    def _np(a, dt):
        if a is None:
            return None
        try:
            import torch
            if isinstance(a, torch.Tensor):
                a = a.detach().cpu().numpy()
        except ImportError:
            pass
        return np.ascontiguousarray(a, dtype=dt)

    tok = _np(tokens, np.int32).reshape(-1)
    par = _np(parents, np.int32).reshape(-1)
    al = _np(alpha, np.float32)
    be = _np(beta, np.float32)
    te = _np(temperature, np.float32)
    qq = _np(q, np.float32)
    sid = _np(seq_ids, np.int32)
    ldq = (V if ldq is None else ldq) if qq is not None else 0
    R = B * N
    accept_len = np.zeros(B, dtype=np.int32)
    path = np.zeros(R, dtype=np.int32)
    bonus = np.zeros(B, dtype=np.int32)
    logprob = np.zeros(R, dtype=np.float64)
    rows = np.zeros(R, dtype=ROW_DTYPE)
    residual = np.zeros((B, V), dtype=np.float64) if want_residual else None
    rc = _load().dcd_oracle_verify(
        B, N, V, DTYPE_CODE[dtype], ld, _ptr(zp), _ptr(zq), _ptr(tok), _ptr(par), _ptr(al), _ptr(be),
        _ptr(te), _ptr(qq), ldq, seed, offset, _ptr(sid), int(distinct), nthreads, _ptr(accept_len), _ptr(path),
        _ptr(bonus),
        _ptr(logprob), _ptr(rows), _ptr(residual))
    if rc != 0:
        raise ValueError(f"oracle verify failed: {rc}")
    return dict(accept_len=accept_len, accept_path=path.reshape(B, N), bonus=bonus,
                cd_logprob=logprob.reshape(B, N), rows=rows.reshape(B, N), residual=residual)


def verify_workload(w, nthreads: int = 1, want_residual: bool = False, seqs=None, distinct: bool = False) -> dict:
    """Runs ``verify`` on a workloads.Workload (optionally on a subset of its sequences)."""
    import torch
    B, N, V = w.B, w.N, w.V
    sel = list(range(B)) if seqs is None else list(seqs)
    rows = torch.cat([torch.arange(b * N, (b + 1) * N) for b in sel]).to(w.z_exp.device)
    zp = w.z_exp[rows].cpu()
    zq = w.z_ama[rows].cpu()
    q = None if w.q is None else w.q[rows.to(w.q.device)].cpu()
    return verify(B=len(sel), N=N, V=V, dtype=w.dtype, z_exp=zp, z_ama=zq,
                  tokens=w.tokens.cpu()[sel], parents=w.parents.cpu()[sel], alpha=w.alpha.cpu()[sel],
                  beta=w.beta.cpu()[sel], temperature=w.temperature.cpu()[sel], q=q, seed=w.seed,
                  offset=w.offset, nthreads=nthreads, want_residual=want_residual, seq_ids=np.asarray(sel),
                  distinct=distinct)


def margin_fn(zp_row, za_row, alpha: float, beta: float) -> float:
    """Decision margin of one row for the input generator: min(top-2 score gap, mask distance)."""
    r = row_logpi(np.asarray(zp_row, dtype=np.float64), np.asarray(za_row, dtype=np.float64), alpha, beta, 0.0)
    gap = r["gap_argmax"]
    if beta > 0:
        lp = np.asarray(zp_row, dtype=np.float64)
        m = lp.max()
        gap = min(gap, float(np.min(np.abs(lp - m - np.log(beta)))))
    return gap


def fused_logits(h, w, chunk: int = 8192) -> np.ndarray:
    """z = h w^T in fp64 from the exact bf16 values (the fused LM-head variant's logits), h
    [rows, H] and w [V, H]: a library matrix product, taken over blocks of `chunk` vocabulary
    rows to bound host memory."""
    import torch
    hh = (h.detach().cpu() if isinstance(h, torch.Tensor) else torch.as_tensor(h)).to(torch.float64).numpy()
    V = w.shape[0]
    out = np.empty((hh.shape[0], V), dtype=np.float64)
    for v0 in range(0, V, chunk):
        v1 = min(V, v0 + chunk)
        wb = w[v0:v1]
        wb = (wb.detach().cpu() if isinstance(wb, torch.Tensor) else torch.as_tensor(wb)).to(torch.float64).numpy()
        out[:, v0:v1] = hh @ wb.T
    return out


def verify_fused_workload(w, nthreads: int = 1, seqs=None) -> dict:
    """``verify`` of a fused LM-head workload: logits from ``fused_logits`` (fp64), greedy, with the
    workload's beta (the plausibility mask) when any is nonzero."""
    B, N = w.B, w.N
    sel = list(range(B)) if seqs is None else list(seqs)
    rows = np.concatenate([np.arange(b * N, (b + 1) * N) for b in sel])
    import torch
    ridx = torch.as_tensor(rows, device=w.h_exp.device)
    zp = fused_logits(w.h_exp[ridx], w.w_exp)
    zq = fused_logits(w.h_ama[ridx], w.w_ama)
    beta = None
    if getattr(w, "beta", None) is not None and bool((w.beta != 0).any()):
        beta = w.beta.cpu()[sel]
    return verify(B=len(sel), N=N, V=w.V, dtype="f64", z_exp=zp, z_ama=zq,
                  tokens=w.tokens.cpu()[sel], parents=w.parents.cpu()[sel], alpha=w.alpha.cpu()[sel],
                  beta=beta, temperature=None, nthreads=nthreads, seq_ids=np.asarray(sel))


def row_diagnostics(zp, zq, xstar: int, q=None, dtype: str = "f64", alpha=None) -> dict:
    """Per-row diagnostics (see dcd_oracle_row_diagnostics): lse_p, lse_q, signal at x*, e_q,
    kl_p_q = D_KL(pi_p || pi_q); with the drafter's distribution q: e_e and kl_e_p; with the
    contrast strength alpha: kl_p_cd = D_KL(pi_p || pi_CD) of the untruncated T = 1 target."""
    zp = _logits(zp, dtype)
    zq = _logits(zq, dtype)
    V = zp.shape[-1]
    qq = None if q is None else np.ascontiguousarray(q, dtype=np.float32)
    out = np.empty(8, dtype=np.float64)
    a = -1.0 if alpha is None else float(alpha)
    rc = _load().dcd_oracle_row_diagnostics(V, DTYPE_CODE[dtype], _ptr(zp), _ptr(zq), _ptr(qq), int(xstar), a,
                                            _ptr(out))
    if rc != 0:
        raise ValueError(f"oracle row_diagnostics failed: {rc}")
    return dict(zip(("lse_p", "lse_q", "signal", "e_q", "e_e", "kl_e_p", "kl_p_q", "kl_p_cd"), out))
