"""GPU parity of the cluster-per-row kernel's own paths against the oracle: rows of sampled
sequences split over clusters of 2 and 4 CTAs (bf16 and fp32, with and without the
plausibility mask, whose expert maxima are exchanged first), the greedy rows' half-row units
(a row with beta > 0 there is taken whole), and a batch of more than 1024 sequences, which has no
sequence list: every row is taken whole and a sampled row's residual chain runs in one CTA.
Siblings drawn without replacement run on split rows (their removed tokens' masses corrected
across the slices) and on whole rows.  Bars as in parity_util."""

import pytest
import torch

import oracle
from paper_2608_12913_gb300 import workloads
from parity_util import compare, run_gpu

pytestmark = pytest.mark.gpu


def _oracle(w, residual=False):
    return oracle.verify_workload(w, nthreads=oracle.max_threads(), want_residual=residual)


@pytest.mark.parametrize("dtype,V", [("bf16", 40000), ("f32", 20000)])
@pytest.mark.parametrize("beta", [0.0, 0.1, 0.5])
def test_split_rows_with_chains_and_mask(dtype, V, beta):
    # 240 rows of sampled sequences: clusters of 2 CTAs (five statistics stages a row), each
    # row's slices exchanged; with beta > 0 the slices' expert maxima are exchanged first
    w = workloads.generate(name="split", B=4, V=V, dtype=dtype, spikes=(1, 6), alphas=(0.1, 0.5), beta=beta,
                           temperatures=(1.0, 0.7), seed=int(beta * 100) + V, margin_fn=oracle.margin_fn)
    g = run_gpu(w, sampled=True, residual=True)
    compare(w, g, _oracle(w, residual=True), check_residual=True)


def test_split_rows_four_ctas_and_an_empty_slice():
    # fp32 rows of 34176 tokens are nine 4096-token stages: clusters of 4 CTAs take three stages
    # each, and the fourth CTA's slice is empty
    w = workloads.generate(name="split4", B=3, V=34176, dtype="f32", spikes=(1, 6), alphas=(0.0, 0.5),
                           temperatures=(1.0,), levels=(1, 5, 8, 5, 3), seed=25, margin_fn=oracle.margin_fn)
    g = run_gpu(w, sampled=True, residual=True)
    compare(w, g, _oracle(w, residual=True), check_residual=True)


@pytest.mark.parametrize("beta", [0.0, 0.1])
def test_greedy_rows_in_half_row_units(beta):
    # 720 greedy rows (past the one-launch path): every CTA takes rows whole, the last wave in two
    # half-row units combined through the workspace; with beta > 0 those rows are taken whole
    w = workloads.generate(name="halves", B=12, V=20000, dtype="bf16", spikes=(1, 6), alphas=(0.05, 0.1, 0.2),
                           beta=beta, temperatures=(0.0,), seed=61 + int(beta * 10), margin_fn=oracle.margin_fn)
    g = run_gpu(w, sampled=False)
    compare(w, g, _oracle(w))


def test_mixed_batch_with_two_cta_clusters():
    # 1080 rows, half of them in sampled sequences: clusters of 2 CTAs for those, whole rows and
    # half-row units for the greedy ones
    w = workloads.make_config(3, B=18, V=40000, seed=71, margin_fn=oracle.margin_fn)
    g = run_gpu(w, sampled=True, residual=True)
    compare(w, g, _oracle(w, residual=True), check_residual=True)


def test_more_than_1024_sequences_rows_whole():
    # 1100 sequences of 4 nodes (a root with three children), every other one sampled: no
    # sequence list, so every row is taken whole and a sampled root's chain runs in one CTA
    w = workloads.generate(name="many", B=1100, V=1000, dtype="bf16", spikes=(1, 3), alphas=(0.1, 0.5),
                           temperatures=(0.0, 1.0), levels=(1, 3), seed=81, margin_fn=oracle.margin_fn)
    g = run_gpu(w, sampled=True, residual=True)
    compare(w, g, _oracle(w, residual=True), check_residual=True, max_amb_frac=0.05)
    assert int((w.temperature > 0).sum()) == 550


def _oracle_distinct(w):
    return oracle.verify_workload(w, nthreads=oracle.max_threads(), want_residual=True, distinct=True)


@pytest.mark.parametrize("dtype,V,beta", [("bf16", 40000, 0.0), ("bf16", 40000, 0.5), ("f32", 34176, 0.1)])
def test_distinct_siblings_on_split_rows(dtype, V, beta):
    # siblings drawn without replacement on rows split over clusters of 4 CTAs (bf16) and 8 CTAs
    # with three empty slices (fp32): q's own mass is summed over the slices in the first pass,
    # and the removed tokens' frozen masses correct the exchanged pass sums and the owning CTA's
    # race blocks; nodes of up to 10 children make long chains of removals
    w = workloads.generate(name="split_distinct", B=4, V=V, dtype=dtype, spikes=(1, 6), alphas=(0.1, 0.5),
                           beta=beta, temperatures=(1.0, 0.7), levels=(1, 10, 12, 8), max_children=10,
                           seed=90 + int(beta * 10) + V % 7, margin_fn=oracle.margin_fn)
    g = run_gpu(w, sampled=True, residual=True, distinct=True)
    compare(w, g, _oracle_distinct(w), check_residual=True)


def test_distinct_duplicates_and_zero_draft_probability_on_split_rows():
    # a duplicated sibling token (its proposal is 0 once the first copy is removed) and a sibling
    # token of zero draft probability, on rows split over clusters of 4 CTAs
    w = workloads.generate(name="split_dup", B=3, V=40000, dtype="bf16", spikes=(1, 6), alphas=(0.2,),
                           temperatures=(1.0,), levels=(1, 6, 9, 6), seed=97, margin_fn=oracle.margin_fn)
    tok = w.tokens.clone()
    q = w.q.clone()
    for b in range(w.B):
        kids = workloads.children_lists(w.parents[b].numpy())
        for n, ch in enumerate(kids):
            if len(ch) >= 2:
                tok[b, ch[1]] = tok[b, ch[0]]
            if len(ch) >= 3:
                q[b * w.N + n, int(tok[b, ch[2]])] = 0.0
    w.tokens, w.q = tok, q
    g = run_gpu(w, sampled=True, residual=True, distinct=True)
    compare(w, g, _oracle_distinct(w), check_residual=True)


def test_distinct_siblings_more_than_1024_sequences():
    # no sequence list: every row whole on one CTA, the removed-token bookkeeping in one CTA's
    # shared memory; a root with five children allows chains of removals
    w = workloads.generate(name="many_distinct", B=1030, V=1000, dtype="bf16", spikes=(1, 3), alphas=(0.1, 0.5),
                           temperatures=(1.0, 0.0), levels=(1, 5), seed=83, margin_fn=oracle.margin_fn)
    g = run_gpu(w, sampled=True, residual=True, distinct=True)
    compare(w, g, _oracle_distinct(w), check_residual=True, max_amb_frac=0.05)
