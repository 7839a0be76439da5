"""The one-launch greedy path of small calls (at most 512 rows and 256 nodes a sequence): parity
with the oracle and agreement with the persistent row kernel (dcd_score_rows + dcd_tree_walk)
on the same inputs.  Bars as in parity_util: integers bit-exact, cd_lse / cd_logprob within 1e-4
of the oracle; between the two GPU paths, which sum in different orders, within 1e-5."""

import numpy as np
import pytest
import torch

import oracle
from paper_2608_12913_gb300 import dcd, workloads
from parity_util import compare, run_gpu

pytestmark = pytest.mark.gpu


def _persistent(w):
    wd = w.to("cuda")
    o = dcd.dcd_score_rows(wd.z_exp, wd.z_ama, wd.tokens, wd.parents, wd.alpha, wd.beta)
    dcd.dcd_tree_walk(w.B, w.N, w.V, o, o["workspace"])
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in o.items() if k != "workspace"}


def _check(w):
    fast = run_gpu(w, sampled=False)  # dcd_verify_greedy: one launch for a small call
    ref = oracle.verify_workload(w, nthreads=oracle.max_threads())
    compare(w, fast, ref)
    slow = _persistent(w)
    for k in ("accept_len", "accept_path", "bonus", "cd_argmax"):
        assert np.array_equal(fast[k], slow[k]), k
    assert np.abs(fast["cd_lse"] - slow["cd_lse"]).max() <= 1e-5
    both = np.isneginf(fast["cd_logprob"]) & np.isneginf(slow["cd_logprob"])
    assert np.array_equal(np.isneginf(fast["cd_logprob"]), np.isneginf(slow["cd_logprob"]))
    with np.errstate(invalid="ignore"):
        diff = np.where(both, 0.0, np.abs(fast["cd_logprob"] - slow["cd_logprob"]))
    assert diff.max() <= 1e-5


def test_small_chain_fp32_and_tree_bf16():
    _check(workloads.make_config(0))                    # 6-node chain, fp32, V = 32000
    _check(workloads.make_config(1))                    # 60-node tree, bf16, V = 128256
    _check(workloads.make_config(1, B=8, V=4099, seed=31))  # 480 rows, ragged vocabulary


@pytest.mark.parametrize("beta", [1e-3, 0.1])
def test_small_plausibility_mask(beta):
    w = workloads.make_config(1, B=2, V=20000, beta=beta, seed=32)
    _check(w)


def test_small_tiny_vocabularies_and_unaligned_rows():
    for V in (1, 7, 9, 2049):
        _check(workloads.make_config(1, B=1, V=V, seed=33 + V))
    # rows at an odd element offset inside a padded buffer: not 16-byte aligned (one-token loads)
    w = workloads.make_config(1, B=2, V=3001, seed=34)
    wd = w.to("cuda")
    R, V = w.R, w.V
    zp = torch.zeros((R, V + 3), dtype=wd.z_exp.dtype, device="cuda")
    zq = torch.zeros_like(zp)
    zp[:, 1:V + 1] = wd.z_exp
    zq[:, 1:V + 1] = wd.z_ama
    o = dcd.dcd_verify_greedy(zp[:, 1:V + 1], zq[:, 1:V + 1], wd.tokens, wd.parents, wd.alpha, wd.beta)
    ref = run_gpu(w, sampled=False)
    torch.cuda.synchronize()
    for k in ("accept_len", "accept_path", "bonus", "cd_argmax"):
        assert np.array_equal(o[k].cpu().numpy(), ref[k]), k
    np.testing.assert_allclose(o["cd_lse"].cpu().numpy(), ref["cd_lse"], atol=1e-5)


def test_small_path_boundaries():
    # 2 x 256-node chains = 512 rows: the one-launch path; 257 nodes: the persistent kernel
    for n, b in ((256, 2), (257, 1)):
        w = workloads.make_config(0, V=2000, chain_len=n, B=b, dtype="bf16", seed=35)
        _check(w)
