"""GPU parity of the sampled rule for siblings drawn without replacement (DCD_SIBLINGS_DISTINCT)
against the oracle's literal rule (q less the earlier siblings' tokens, renormalised), and its
losslessness on the GPU.  Bars as in parity_util."""

import numpy as np
import pytest
import torch
from scipy import special, stats

import oracle
from paper_2608_12913_gb300 import dcd, workloads
from parity_util import compare, run_gpu

pytestmark = pytest.mark.gpu


def _oracle(w, residual=False, seqs=None):
    return oracle.verify_workload(w, nthreads=oracle.max_threads(), want_residual=residual, seqs=seqs,
                                  distinct=True)


def test_distinct_tree_sampled_with_residual():
    w = workloads.make_config(2, V=4099, B=6, seed=31, margin_fn=oracle.margin_fn)
    g = run_gpu(w, sampled=True, residual=True, distinct=True)
    compare(w, g, _oracle(w, residual=True), check_residual=True)


def test_distinct_full_vocabulary_sampled():
    w = workloads.make_config(2, margin_fn=oracle.margin_fn)
    g = run_gpu(w, sampled=True, residual=True, distinct=True)
    compare(w, g, _oracle(w, residual=True), check_residual=True)


@pytest.mark.parametrize("beta", [0.1, 0.5])
def test_distinct_with_plausibility_mask(beta):
    # the distinct rule on masked rows (rows read whole, a max pass first), residual output included
    w = workloads.make_config(2, V=4099, B=6, beta=beta, seed=33, margin_fn=oracle.margin_fn)
    g = run_gpu(w, sampled=True, residual=True, distinct=True)
    compare(w, g, _oracle(w, residual=True), check_residual=True)


def test_distinct_mixed_batch_and_split_steps():
    w = workloads.make_config(3, B=6, V=20000, margin_fn=oracle.margin_fn)
    ref = _oracle(w)
    compare(w, run_gpu(w, sampled=True, distinct=True), ref)
    compare(w, run_gpu(w, sampled=True, stages=3, distinct=True), ref)


def test_distinct_full_size_sampled_sequences():
    dev = torch.device("cuda")
    w = workloads.make_config_torch(3, device=dev)
    g = run_gpu(w, sampled=True, distinct=True)
    seqs = [1, 3, 5, 7, 9, 11, 13, 15]
    compare(w, g, _oracle(w, seqs=seqs), seqs=seqs)


def test_distinct_duplicates_and_zero_draft_probability():
    w = workloads.make_config(2, B=6, V=501, seed=17, margin_fn=oracle.margin_fn)
    tok = w.tokens.clone()
    q = w.q.clone()
    for b in range(w.B):
        kids = workloads.children_lists(w.parents[b].numpy())
        for n, ch in enumerate(kids):
            if len(ch) >= 2:
                tok[b, ch[1]] = tok[b, ch[0]]  # a duplicate: its proposal is 0 once the first is removed
            if len(ch) >= 3:
                q[b * w.N + n, int(tok[b, ch[2]])] = 0.0
    w.tokens, w.q = tok, q
    g = run_gpu(w, sampled=True, residual=True, distinct=True)
    compare(w, g, _oracle(w, residual=True), check_residual=True)


def test_distinct_more_than_32_children_is_reported():
    w = workloads.make_config(2, B=2, V=1000, seed=19, levels=(1, 40), max_children=40)
    g = run_gpu(w, sampled=True, distinct=True)
    assert g["error_bits"] & 0x20
    assert np.all(g["accept_len"] == 0)


def test_distinct_lossless_on_the_gpu_monte_carlo():
    """The GPU's first emitted token follows pi_CD when the siblings are m distinct tokens drawn
    without replacement from q."""
    rng = np.random.default_rng(6)
    V, B, m = 6, 60000, 3
    N = m + 1
    zp = rng.standard_normal(V)
    zq = 0.7 * zp + rng.standard_normal(V)
    qd = special.softmax(zp + 0.8 * rng.standard_normal(V)).astype(np.float32)
    alpha, T = 0.3, 1.0
    qn = qd.astype(np.float64) / qd.sum(dtype=np.float64)
    gk = np.log(qn)[None, :] - np.log(-np.log(rng.random((B, V))))
    tokens = np.zeros((B, N), dtype=np.int32)
    tokens[:, 1:] = np.argsort(-gk, axis=1)[:, :m]  # Gumbel top-m: drawn without replacement
    parents = np.tile(np.array([-1] + [0] * m, dtype=np.int32), (B, 1))
    dev = "cuda"
    Z = torch.tensor(np.tile(zp.astype(np.float32), (B * N, 1)), device=dev)
    Zq = torch.tensor(np.tile(zq.astype(np.float32), (B * N, 1)), device=dev)
    Q = torch.tensor(np.tile(qd, (B * N, 1)), device=dev)
    o = dcd.dcd_verify_sample(Z, Zq, Q, torch.tensor(tokens, device=dev), torch.tensor(parents, device=dev),
                              torch.full((B,), alpha, device=dev), torch.full((B,), T, device=dev), 12, 0,
                              distinct=True)
    torch.cuda.synchronize()
    assert dcd.dcd_get_device_error(o["workspace"]) == 0
    L = o["accept_len"].cpu().numpy()
    path = o["accept_path"].cpu().numpy()
    first = np.where(L > 0, tokens[np.arange(B), path[:, 1].clip(0)], o["bonus"].cpu().numpy())
    pi = np.exp(oracle.row_logpi(zp.astype(np.float32).astype(np.float64), zq.astype(np.float32).astype(np.float64),
                                 alpha, 0.0, T)["logpi"])
    counts = np.bincount(first, minlength=V)
    assert stats.chisquare(counts, B * pi).pvalue > 1e-4


def _unnormalised(w, kind):
    """q rows whose mass is not 1: a drafter's top-k truncation (the mass outside the top 64
    tokens dropped, not renormalised), or every row scaled by 0.93."""
    q = w.q.clone()
    if kind == "topk":
        keep = torch.topk(q, 64, dim=1).indices
        mask = torch.zeros_like(q, dtype=torch.bool)
        mask.scatter_(1, keep, True)
        q = torch.where(mask, q, torch.zeros_like(q))
    else:
        q = q * 0.93
    w.q = q
    return w


@pytest.mark.parametrize("kind", ["topk", "scaled"])
@pytest.mark.parametrize("distinct", [True, False])
def test_unnormalised_draft_rows(kind, distinct):
    # Both rules take q as given: the i.i.d. rule uses it as is, the distinct rule renormalises
    # by the mass that remains after a removal, q's own mass less the removed tokens' (a
    # top-k-truncated drafter sends rows that sum to less than 1).
    w = _unnormalised(workloads.make_config(2, V=4099, B=6, seed=37, margin_fn=oracle.margin_fn), kind)
    g = run_gpu(w, sampled=True, residual=True, distinct=distinct)
    r = oracle.verify_workload(w, nthreads=oracle.max_threads(), want_residual=True, distinct=distinct)
    compare(w, g, r, check_residual=True)
    mass = w.q.double().sum(dim=1)
    assert float((mass - 1.0).abs().max()) > 0.05  # the rows really are unnormalised
