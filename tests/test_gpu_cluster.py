"""GPU parity of the cluster-per-row kernel's own paths against the oracle: rows of sampled
sequences split over clusters of 2 and 4 CTAs (bf16 and fp32, with and without the
plausibility mask, whose expert maxima are exchanged first), the greedy rows' half-row units
(a row with beta > 0 there is taken whole), and a batch of more than 1024 sequences, which has no
sequence list: every row is taken whole and a sampled row's residual chain runs in one CTA.
Bars as in parity_util."""

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
