"""A seeded sweep of random shapes against the oracle.  Each case draws, from its own fixed seed,
the batch size, the tree (random levels, a chain or a star), the vocabulary (ragged sizes from 8
to 40000), the logit dtype (every fifth case a batch of 40-64 sequences of 25 nodes, more than
two rows per resident CTA), alpha, beta, the temperatures and the sibling rule, so the sweep is
the same on every run.  Inputs obey the margin rule; the bars are parity_util's (integers
bit-exact, scores within 1e-4, residuals within 1e-5 total variation)."""

import numpy as np
import pytest

import oracle
from paper_2608_12913_gb300 import workloads
from parity_util import compare, run_gpu

pytestmark = pytest.mark.gpu

N_CASES = 64


def _case(i):
    rng = np.random.default_rng(7000 + i)
    kind = str(rng.choice(["levels", "chain", "star"]))
    if kind == "chain":
        shape = dict(chain_len=int(rng.integers(1, 40)))
    elif kind == "star":
        shape = dict(levels=(1, int(rng.integers(1, 9))))
    else:  # at most 8 nodes per node of the level above: every node finds a parent
        shape = dict(levels=tuple([1] + [int(rng.integers(1, 9)) for _ in range(int(rng.integers(1, 6)))]))
    V = int(rng.choice([8, 17, 255, 1024, 1025, 4097, int(rng.integers(8, 40001))]))
    B = int(rng.integers(1, 7))
    if i % 5 == 4:  # a batch of more than two rows per resident CTA: whole rows, large-batch pieces
        B = int(rng.integers(40, 65))
        shape = dict(levels=(1, 8, 8, 8))
        V = int(rng.integers(8, 5001))
    spec = dict(name=f"fuzz{i}", B=B, V=V, dtype=str(rng.choice(["bf16", "f32"])),
                spikes=(1, int(rng.integers(1, 7))),
                alphas=tuple(float(a) for a in rng.choice([0.0, 0.05, 0.1, 0.5, 1.0], size=2)),
                beta=float(rng.choice([0.0, 0.0, 1e-3, 0.1])),
                temperatures=tuple(float(t) for t in rng.choice([0.0, 0.5, 1.0, 1.5], size=2)),
                seed=9000 + i, offset=int(rng.integers(0, 1 << 20)), **shape)
    return spec, bool(rng.integers(0, 2))


@pytest.mark.parametrize("i", range(N_CASES))
def test_random_case_matches_oracle(i):
    spec, distinct = _case(i)
    w = workloads.generate(margin_fn=oracle.margin_fn, **spec)
    sampled = bool((w.temperature > 0).any())
    distinct = distinct and sampled
    g = run_gpu(w, sampled=sampled, residual=sampled, distinct=distinct)
    r = oracle.verify_workload(w, nthreads=oracle.max_threads(), want_residual=sampled, distinct=distinct)
    compare(w, g, r, check_residual=sampled, max_amb_frac=0.34)
