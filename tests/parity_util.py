"""Shared helpers of the GPU-versus-oracle parity tests.

Bars (stated once, used by every parity test):
* token ids, argmax, accepted lengths, accepted paths, bonus tokens and the per-row
  acceptance records: bit-exact;
* cd_logprob and cd_lse (the CD scores): within 1e-4 absolute (fp32 on the GPU
  against the fp64 oracle);
* the residual a bonus was drawn from: total variation within 1e-5.

Where floating point decides an integer, the two sides decide in different
precisions (fp32 kernel, fp64 oracle).  The oracle reports every decision's
margin; a row whose margin is below what fp32 can resolve is "ambiguous": its
decision is not compared, and a sequence whose oracle path crosses an ambiguous
row is only checked for validity.  Inputs drawn with the margin rule have none.
"""

from __future__ import annotations

import numpy as np
import torch

import oracle
from paper_2608_12913_gb300 import dcd

SCORE_TOL = 1e-4
TV_TOL = 1e-5
# margins below which fp32 and fp64 may legitimately decide differently
AMB_ARGMAX = 2e-5
AMB_ACCEPT = 1e-5
AMB_RACE = 1e-4
AMB_MASK = 1e-5


def records(ws: torch.Tensor, R: int):
    """Per-row records the kernels leave in the workspace (after the 256-byte header, R 4-byte
    part counters padded to 16 bytes and R 64-byte residual-pass records)."""
    off = 256 + (4 * R + 15) // 16 * 16 + 64 * R
    raw = ws[off:off + 16 * R].cpu().numpy().view(np.int32).reshape(R, 4)
    return dict(acc_child=raw[:, 0].copy(), term_token=raw[:, 1].copy(), status=raw[:, 2].view(np.uint32).copy())


def run_gpu(w, *, sampled: bool, residual: bool = False, stages: int = 0, plain: bool = False, offset=None,
            out=None, workspace=None, distinct: bool = False):
    dev = torch.device("cuda")
    wd = w.to(dev)
    off = w.offset if offset is None else offset
    if stages or plain:
        q = None
        temp = None
        if sampled:
            q = wd.q if wd.q is not None else torch.zeros_like(wd.z_exp, dtype=torch.float32)
            temp = wd.temperature
        o = dcd.dcd_score_rows(wd.z_exp, wd.z_ama, wd.tokens, wd.parents, wd.alpha, wd.beta, q=q, temperature=temp,
                               seed=w.seed, offset=off, stages=stages, plain_loads=plain, out=out,
                               workspace=workspace, distinct=distinct)
        dcd.dcd_tree_walk(w.B, w.N, w.V, o, o["workspace"])
    elif sampled:
        q = wd.q if wd.q is not None else torch.zeros_like(wd.z_exp, dtype=torch.float32)
        o = dcd.dcd_verify_sample(wd.z_exp, wd.z_ama, q, wd.tokens, wd.parents, wd.alpha, wd.temperature, w.seed, off,
                                  wd.beta, residual=residual, out=out, workspace=workspace, distinct=distinct)
    else:
        o = dcd.dcd_verify_greedy(wd.z_exp, wd.z_ama, wd.tokens, wd.parents, wd.alpha, wd.beta, out=out,
                                  workspace=workspace)
    torch.cuda.synchronize()
    res = {k: v.cpu().numpy() for k, v in o.items() if k != "workspace"}
    res["records"] = records(o["workspace"], w.B * w.N)
    res["error_bits"] = dcd.dcd_get_device_error(o["workspace"])
    return res


# The fused LM-head forms its logits itself: bf16 products accumulated in fp32 over K = H (8192
# at full size).  That rounding is about sqrt(K / 16) * 2^-24 * sum_k |h_k w_k| ~ 1.4e-4 of a
# logit at full size (sum |h w| ~ 100), against the oracle's exact fp64 logits.
# * FUSED_AMB_MASK: margin to the plausibility threshold within which the two may mask a token
#   differently;
# * FUSED_SCORE_TOL: the score bar of a masked fused row.  With beta > 0 few tokens make up P_beta
#   and the normaliser follows the GEMM's rounding of one or two logits, (1 + 2 alpha) x 1.4e-4
#   at alpha = 0.1, where an unmasked row's normaliser averages it over many tokens (those keep
#   the 1e-4 bar).
FUSED_AMB_MASK = 2e-4
FUSED_SCORE_TOL = 3e-4


def fused_records(ws: torch.Tensor, R: int):
    """Per-row records of the fused LM-head step (after the 256-byte header, 3 x R x 8 child
    entries of 4 bytes and R 4-byte row statuses padded to 16 bytes)."""
    off = 256 + 96 * R + (4 * R + 15) // 16 * 16
    raw = ws[off:off + 16 * R].cpu().numpy().view(np.int32).reshape(R, 4)
    return dict(acc_child=raw[:, 0].copy(), term_token=raw[:, 1].copy(), status=raw[:, 2].view(np.uint32).copy())


def run_fused_gpu(w, beta=None) -> dict:
    """The fused LM-head call on workload `w` (with the plausibility thresholds `beta`, a tensor
    [B], or none), results on the host in the layout `compare` takes."""
    o = dcd.dcd_verify_fused_lmhead(w.h_exp, w.w_exp, w.h_ama, w.w_ama, w.tokens, w.parents, w.alpha, beta)
    torch.cuda.synchronize()
    res = {k: v.cpu().numpy() for k, v in o.items() if k != "workspace"}
    res["records"] = fused_records(o["workspace"], w.B * w.N)
    res["error_bits"] = dcd.dcd_get_device_error(o["workspace"])
    return res


def compare(w, gpu: dict, ref: dict, seqs=None, check_residual: bool = False, max_amb_frac: float = 0.05,
            amb_mask: float = AMB_MASK, score_tol: float = SCORE_TOL):
    """Asserts parity of GPU outputs (all sequences of `w`, or the subset `seqs`) with the oracle's.

    `amb_mask` is the margin to the plausibility threshold below which a row's mask is taken as
    unresolved.  With materialised logits both sides test the same values and AMB_MASK covers
    fp32 against fp64 evaluation; the fused LM-head forms the logits itself in fp32, so its
    callers pass the GEMM's rounding instead.  Such a row's scores are not compared either (one
    token on the other side of the threshold moves its normaliser)."""
    B, N = w.B, w.N
    sel = np.arange(B) if seqs is None else np.asarray(seqs)
    rows_ref = ref["rows"]  # [len(sel), N]
    gsel = (sel[:, None] * N + np.arange(N)[None, :]).reshape(-1)
    rr = rows_ref.reshape(-1)
    mask_amb = rr["gap_mask"] < amb_mask
    amb = ((rr["gap_argmax"] < AMB_ARGMAX) | (rr["gap_accept"] < AMB_ACCEPT) | (rr["gap_race"] < AMB_RACE) |
           mask_amb)
    assert gpu["error_bits"] == 0, f"device error bits {gpu['error_bits']:#x}"
    assert np.all(gpu["records"]["status"][gsel] == 0)

    # Eq. 1 scores, within tolerance everywhere the mask is resolved
    lse_g = gpu["cd_lse"].reshape(-1)[gsel].astype(np.float64)
    lse_err = np.where(mask_amb, 0.0, np.abs(lse_g - rr["cd_lse"]))
    assert lse_err.max() <= score_tol, f"cd_lse max error {lse_err.max():.3g}"
    lp_g = gpu["cd_logprob"][sel].astype(np.float64)
    lp_r = ref["cd_logprob"]
    # a node's score comes from its parent's row
    par = w.parents.cpu().numpy()[sel] if hasattr(w.parents, "cpu") else np.asarray(w.parents)[sel]
    row_amb = mask_amb.reshape(len(sel), N)
    node_amb = np.zeros_like(row_amb)
    node_amb[:, 1:] = np.take_along_axis(row_amb, np.clip(par[:, 1:], 0, N - 1), axis=1)
    both_inf = np.isneginf(lp_g) & np.isneginf(lp_r)
    assert np.array_equal(np.isneginf(lp_g) & ~node_amb, np.isneginf(lp_r) & ~node_amb), "plausibility masks differ"
    with np.errstate(invalid="ignore"):
        lp_err = np.where(both_inf | node_amb, 0.0, np.abs(lp_g - lp_r))
    assert lp_err.max() <= score_tol, f"cd_logprob max error {lp_err.max():.3g}"

    # integer decisions per row: bit-exact where the margin is resolvable in fp32
    arg_g = gpu["cd_argmax"].reshape(-1)[gsel]
    ok_arg = rr["gap_argmax"] >= AMB_ARGMAX
    assert np.array_equal(arg_g[ok_arg], rr["argmax"][ok_arg]), "cd_argmax mismatch"
    acc_g = gpu["records"]["acc_child"][gsel]
    term_g = gpu["records"]["term_token"][gsel]
    bad = np.nonzero((acc_g != rr["acc_child"]) & ~amb)[0]
    assert bad.size == 0, f"accepted-child mismatch at rows {gsel[bad][:8]}: gpu {acc_g[bad][:8]} " \
                          f"oracle {rr['acc_child'][bad][:8]} gap_accept {rr['gap_accept'][bad][:8]}"
    bad = np.nonzero((term_g != rr["term_token"]) & ~amb)[0]
    assert bad.size == 0, f"terminal-token mismatch at rows {gsel[bad][:8]}: gpu {term_g[bad][:8]} " \
                          f"oracle {rr['term_token'][bad][:8]} gap_race {rr['gap_race'][bad][:8]}"

    # sequences
    amb_rows = amb.reshape(len(sel), N)
    n_amb = 0
    for i, b in enumerate(sel):
        path = ref["accept_path"][i]
        on = path[path >= 0]
        if amb_rows[i, on].any():
            n_amb += 1
            # validity only: a path of real parent-child links from the root
            gp = gpu["accept_path"][b]
            L = gpu["accept_len"][b]
            assert gp[0] == 0 and np.all(gp[L + 1:] == -1)
            par = w.parents[b].cpu().numpy()
            for k in range(1, L + 1):
                assert par[gp[k]] == gp[k - 1]
            continue
        assert gpu["accept_len"][b] == ref["accept_len"][i], f"accept_len mismatch in sequence {b}"
        assert np.array_equal(gpu["accept_path"][b], ref["accept_path"][i]), f"path mismatch in sequence {b}"
        assert gpu["bonus"][b] == ref["bonus"][i], f"bonus mismatch in sequence {b}"
        if check_residual:
            tv = 0.5 * np.abs(gpu["residual"][b].astype(np.float64) - ref["residual"][i]).sum()
            assert tv <= TV_TOL, f"residual TV {tv:.3g} in sequence {b}"
    assert n_amb <= max(1, int(max_amb_frac * len(sel))), f"{n_amb} ambiguous sequences"
    return dict(ambiguous_rows=int(amb.sum()), ambiguous_seqs=n_amb, max_lse_err=float(lse_err.max()),
                max_logprob_err=float(lp_err.max()))
