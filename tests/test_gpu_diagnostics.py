"""GPU parity of the per-row diagnostics (lse_p, lse_q, the signal at the CD argmax, the
alignment terms E_{pi_q}[log pi_p - log pi_q], E_q[log pi_p - log pi_q] and D_KL(q || pi_p) of
Sec. 3.1 / App. C, D_KL(pi_p || pi_q), and D_KL(pi_p || pi_CD) of App. B's decomposition lemma)
against the oracle's fp64 definitions on the same rounded inputs.  The oracle sums
D_KL(pi_p || pi_CD) term by term from Eq. 1; the library forms it from the verification call's
cd_lse by the lemma, so the comparison also checks the lemma on the GPU's numbers.

Bar (DIAG_TOL): |gpu - oracle| <= 1e-4 * max(1, |oracle|) per value.  The kernel accumulates in
fp32 over at most 16384 tokens a CTA (8 to 64 terms a thread, then tree merges) and merges the
chunks in fp32; every linear sum is taken relative to the row's first logit, so with inputs of
logit spread below 30 its rounding stays near 1e-5 of the quantities' scale.  NaN where the definition gives none (no q, no or out-of-range x*) must match
exactly."""

import numpy as np
import pytest
import torch

import oracle
from paper_2608_12913_gb300 import dcd, workloads

pytestmark = pytest.mark.gpu

DIAG_TOL = 1e-4


def _oracle_rows(zp, zq, q, xstar, rows, dtype, alpha=None, lemma=None):
    """Oracle diagnostics of `rows`; alpha[i] (or None) is the contrast strength of row i's
    sequence, and lemma[i] says whether its call's target was untruncated at T = 1 (else the
    last column is NaN, as the library reports it)."""
    out = np.full((len(rows), dcd.DIAG_COLS), np.nan)
    for i, g in enumerate(rows):
        x = int(xstar[g]) if xstar is not None else 0
        ok = xstar is not None and 0 <= x < zp.shape[1]
        a = None if alpha is None or (lemma is not None and not lemma[i]) else float(alpha[i])
        d = oracle.row_diagnostics(zp[g], zq[g], x if ok else 0, q=None if q is None else q[g].numpy(), dtype=dtype,
                                   alpha=a)
        out[i] = [d[k] for k in dcd.DIAG_FIELDS]
        if not ok:
            out[i, 2] = np.nan
    return out


def _compare(gpu, ref):
    gpu = gpu.astype(np.float64)
    assert np.array_equal(np.isnan(gpu), np.isnan(ref)), "NaN pattern differs"
    fin = ~np.isnan(ref)
    err = np.abs(gpu[fin] - ref[fin]) / np.maximum(1.0, np.abs(ref[fin]))
    assert err.max() <= DIAG_TOL, f"max scaled error {err.max():.3g}"
    return float(err.max())


def _inputs(B, V, dtype, seed, levels=(1, 4, 8)):
    w = workloads.generate(name="diag", B=B, V=V, dtype=dtype, temperatures=(1.0,), levels=levels, seed=seed)
    return w


def test_diagnostics_full_vocab_with_q_and_cd_argmax():
    # 2 x 60-node trees at V = 128256 (bf16): q on every row with children, zero rows on leaves;
    # x* is the CD argmax that a greedy verification call reports for each node
    w = workloads.make_config(2, B=2)
    dev = torch.device("cuda")
    wd = w.to(dev)
    R = w.B * w.N
    o = dcd.dcd_verify_greedy(wd.z_exp, wd.z_ama, wd.tokens, wd.parents, wd.alpha, wd.beta)
    xstar = o["cd_argmax"].reshape(-1).contiguous()
    q = wd.q.reshape(R, w.V)
    # the greedy call's cd_lse (reported at T = 1) gives D_KL(pi_p || pi_CD) by the lemma
    got = dcd.dcd_row_diagnostics(wd.z_exp.reshape(R, w.V), wd.z_ama.reshape(R, w.V), w.B, w.N, q=q, xstar=xstar,
                                  cd_lse=o["cd_lse"].reshape(-1).contiguous(), alpha=wd.alpha, beta=wd.beta)
    torch.cuda.synchronize()
    alpha = np.repeat(w.alpha.numpy(), w.N)
    beta0 = np.repeat((w.beta.numpy() if w.beta is not None else np.zeros(w.B)) == 0, w.N)
    ref = _oracle_rows(w.z_exp.reshape(R, w.V), w.z_ama.reshape(R, w.V), w.q.reshape(R, w.V), xstar.cpu().numpy(),
                       range(R), "bf16", alpha=alpha, lemma=beta0)
    _compare(got.cpu().numpy(), ref)
    assert np.isfinite(got.cpu().numpy()[:, 6:]).all()
    # leaves have q = 0: E_q terms and the divergence vanish
    leaf = (w.q.reshape(R, w.V).sum(dim=1) == 0).numpy()
    assert leaf.any() and np.all(got.cpu().numpy()[leaf][:, 4:6] == 0)


def test_diagnostics_f32_out_of_range_xstar():
    w = _inputs(1, 10000, "f32", seed=21)
    R = w.B * w.N
    dev = torch.device("cuda")
    xs = np.random.default_rng(5).integers(0, w.V, size=R).astype(np.int32)
    xs[0], xs[1] = -1, w.V  # outside [0, V): NaN signal
    xstar = torch.from_numpy(xs).to(dev)
    got = dcd.dcd_row_diagnostics(w.z_exp.reshape(R, w.V).to(dev), w.z_ama.reshape(R, w.V).to(dev), w.B, w.N,
                                  q=w.q.reshape(R, w.V).to(dev), xstar=xstar)
    torch.cuda.synchronize()
    ref = _oracle_rows(w.z_exp.reshape(R, w.V), w.z_ama.reshape(R, w.V), w.q.reshape(R, w.V), xs, range(R), "f32")
    _compare(got.cpu().numpy(), ref)
    assert np.isnan(got[0, 2].item()) and np.isnan(got[1, 2].item())


def test_diagnostics_padded_rows_ragged_tail():
    # V = 20004 inside rows of 20008: 16-byte loads with a 4-token ragged tail; q with its own stride
    V, ld = 20004, 20008
    w = _inputs(1, V, "bf16", seed=22)
    R = w.B * w.N
    dev = torch.device("cuda")
    zp = torch.zeros((R, ld), dtype=torch.bfloat16, device=dev)
    zq = torch.zeros((R, ld), dtype=torch.bfloat16, device=dev)
    qq = torch.zeros((R, ld + 4), dtype=torch.float32, device=dev)
    zp[:, :V] = w.z_exp.reshape(R, V).to(dev)
    zq[:, :V] = w.z_ama.reshape(R, V).to(dev)
    qq[:, :V] = w.q.reshape(R, V).to(dev)
    zp[:, V:] = 1e4  # padding beyond V must not be read as tokens
    zq[:, V:] = 1e4
    xs = torch.arange(R, dtype=torch.int32, device=dev) * 331 % V
    got = dcd.dcd_row_diagnostics(zp[:, :V], zq[:, :V], w.B, w.N, q=qq[:, :V], xstar=xs)
    torch.cuda.synchronize()
    ref = _oracle_rows(w.z_exp.reshape(R, V), w.z_ama.reshape(R, V), w.q.reshape(R, V), xs.cpu().numpy(), range(R),
                       "bf16")
    _compare(got.cpu().numpy(), ref)


def test_diagnostics_unaligned_rows_without_q():
    # V = 5003 (rows not 16-byte aligned): the one-token path; no q and no x*: NaN columns
    w = _inputs(2, 5003, "bf16", seed=23)
    R = w.B * w.N
    dev = torch.device("cuda")
    got = dcd.dcd_row_diagnostics(w.z_exp.reshape(R, w.V).to(dev), w.z_ama.reshape(R, w.V).to(dev), w.B, w.N)
    torch.cuda.synchronize()
    ref = _oracle_rows(w.z_exp.reshape(R, w.V), w.z_ama.reshape(R, w.V), None, None, range(R), "bf16")
    _compare(got.cpu().numpy(), ref)
    assert np.isnan(got[:, [2, 4, 5, 7]].cpu().numpy()).all()


def test_diagnostics_single_token_and_tiny_vocab():
    # V = 1: every distribution is a point mass (lse = the logit, the rest 0); V = 7: one partial vector
    dev = torch.device("cuda")
    for V in (1, 7):
        g = torch.Generator().manual_seed(V)
        zp = (3 * torch.randn(5, V, generator=g)).to(torch.float32)
        zq = (3 * torch.randn(5, V, generator=g)).to(torch.float32)
        q = torch.softmax(torch.randn(5, V, generator=g), dim=1)
        xs = torch.zeros(5, dtype=torch.int32)
        got = dcd.dcd_row_diagnostics(zp.to(dev), zq.to(dev), 1, 5, q=q.to(dev), xstar=xs.to(dev))
        torch.cuda.synchronize()
        ref = _oracle_rows(zp.numpy(), zq.numpy(), q, xs.numpy(), range(5), "f32")
        _compare(got.cpu().numpy(), ref)


def test_diagnostics_full_size_batch_sampled_rows():
    # the 32 x 60-node batch at V = 128256 in one call; 96 rows checked against the oracle
    w = workloads.make_config_torch(3)
    R = w.B * w.N
    q = w.q.reshape(R, w.V)
    xs = torch.randint(0, w.V, (R,), dtype=torch.int32, generator=torch.Generator().manual_seed(3)).cuda()
    got = dcd.dcd_row_diagnostics(w.z_exp.reshape(R, w.V), w.z_ama.reshape(R, w.V), w.B, w.N, q=q, xstar=xs)
    torch.cuda.synchronize()
    rows = np.sort(np.random.default_rng(7).choice(R, size=96, replace=False))
    ridx = torch.from_numpy(rows).cuda()
    zp = w.z_exp.reshape(R, w.V)[ridx].cpu()
    zq = w.z_ama.reshape(R, w.V)[ridx].cpu()
    qs = q[ridx].cpu()
    ref = _oracle_rows(zp, zq, qs, xs[ridx].cpu().numpy(), range(len(rows)), "bf16")
    _compare(got[ridx].cpu().numpy(), ref)


def test_diagnostics_kl_decomposition_lemma_per_sequence():
    """D_KL(pi_p || pi_CD) from the cd_lse of a sampled call with per-sequence alpha, beta and
    temperature: sequences at T = 1 with beta = 0 match the oracle's direct sum; a sequence with
    beta > 0 or with T = 0.5 reports NaN (the lemma holds for the untruncated T = 1 target only)."""
    dev = torch.device("cuda")
    w = workloads.make_config(3, B=6, V=9001, seed=24)
    R = w.B * w.N
    alpha = torch.tensor([0.0, 0.1, 0.5, 0.2, 1.0, 0.1], dtype=torch.float32)
    beta = torch.tensor([0.0, 0.0, 0.0, 0.1, 0.0, 0.0], dtype=torch.float32)
    temp = torch.tensor([1.0, 1.0, 0.0, 1.0, 0.5, 1.0], dtype=torch.float32)
    wd = w.to(dev)
    o = dcd.dcd_verify_sample(wd.z_exp, wd.z_ama, wd.q, wd.tokens, wd.parents, alpha.to(dev), temp.to(dev), w.seed, 0,
                              beta.to(dev))
    got = dcd.dcd_row_diagnostics(wd.z_exp, wd.z_ama, w.B, w.N, cd_lse=o["cd_lse"].reshape(-1).contiguous(),
                                  alpha=alpha.to(dev), beta=beta.to(dev), temperature=temp.to(dev))
    torch.cuda.synchronize()
    valid = np.repeat(((beta == 0) & ((temp == 0) | (temp == 1))).numpy(), w.N)
    ref = _oracle_rows(w.z_exp, w.z_ama, None, None, range(R), "bf16", alpha=np.repeat(alpha.numpy(), w.N),
                       lemma=valid)
    _compare(got.cpu().numpy(), ref)
    g = got.cpu().numpy()
    assert np.isfinite(g[valid, 7]).all() and np.isnan(g[~valid, 7]).all()
    assert np.abs(g[:w.N, 7]).max() < 1e-4  # alpha = 0: pi_CD = pi_p
