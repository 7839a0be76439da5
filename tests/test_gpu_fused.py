"""GPU parity of the greedy step fused with the two LM heads (tcgen05 GEMMs with the CD epilogue)
against the oracle on the same bf16 hidden states and weights: the oracle forms the logits
h W^T in fp64 and runs its row definition (Eq. 1, beta = 0, greedy rule).  Bars as in
parity_util: integers bit-exact, cd_lse / cd_logprob within 1e-4."""

import numpy as np
import pytest
import torch

import oracle
from paper_2608_12913_gb300 import dcd, workloads
from parity_util import FUSED_AMB_MASK, FUSED_SCORE_TOL, compare, run_fused_gpu

pytestmark = pytest.mark.gpu


def _check(w, seqs=None):
    gpu = run_fused_gpu(w)
    ref = oracle.verify_fused_workload(w, nthreads=oracle.max_threads(), seqs=seqs)
    return compare(w, gpu, ref, seqs=seqs)


def test_fused_one_tile_ragged_vocab_and_k():
    # 120 rows (one row tile), V = 4099 (17 vocabulary tiles, the last ragged), K tails of 8 and 8
    w = workloads.make_fused_torch(B=2, V=4099, H_exp=520, H_ama=136, seed=11)
    _check(w)


def test_fused_several_row_tiles():
    # 180 rows: a full and a ragged row tile; V = 1000: four vocabulary tiles
    w = workloads.make_fused_torch(B=3, V=1000, H_exp=1024, H_ama=256, seed=12)
    _check(w)


def test_fused_wide_vocabulary():
    w = workloads.make_fused_torch(B=4, V=32000, H_exp=2048, H_ama=512, seed=13)
    _check(w)


def test_fused_full_size_sampled_sequences():
    # the fused LM-head workload at full size (3840 rows, V = 128256, H = 8192 / 2048); the
    # oracle recomputes two of its 64 sequences
    w = workloads.make_fused_torch()
    _check(w, seqs=[0, 37])


def test_fused_node_with_too_many_children_is_reported():
    w = workloads.make_fused_torch(B=2, V=1000, H_exp=256, H_ama=64, seed=14)
    par = w.parents.clone()
    par[1, 1:10] = 0  # nine children of the root of sequence 1 (parents stay ordered)
    par[1, 10:] = 1
    w.parents = par
    gpu = run_fused_gpu(w)
    assert gpu["error_bits"] & 0x20
    assert gpu["accept_len"][1] == 0 and gpu["bonus"][1] == -1
    # sequence 0 is unaffected
    ref = oracle.verify_fused_workload(w, seqs=[0])
    assert gpu["accept_len"][0] == ref["accept_len"][0]
    assert np.array_equal(gpu["accept_path"][0], ref["accept_path"][0])


def test_fused_equals_greedy_on_materialised_logits():
    # the same step on logits the caller computed: bf16 matmul in fp32 accumulation, rounded to
    # fp32 -- decisions agree and scores agree to fp32 rounding
    w = workloads.make_fused_torch(B=2, V=4099, H_exp=512, H_ama=128, seed=15)
    zp = (w.h_exp.float() @ w.w_exp.float().t()).contiguous()
    zq = (w.h_ama.float() @ w.w_ama.float().t()).contiguous()
    a = dcd.dcd_verify_greedy(zp, zq, w.tokens, w.parents, w.alpha, None)
    f = dcd.dcd_verify_fused_lmhead(w.h_exp, w.w_exp, w.h_ama, w.w_ama, w.tokens, w.parents, w.alpha)
    torch.cuda.synchronize()
    for k in ("accept_len", "accept_path", "bonus", "cd_argmax"):
        assert torch.equal(a[k], f[k]), k
    assert (a["cd_lse"] - f["cd_lse"]).abs().max().item() < 1e-4
    assert (a["cd_logprob"] - f["cd_logprob"]).abs().max().item() < 1e-4


# ---- the plausibility mask (beta > 0): a max sweep over the expert's logits, then the masked sweep


def _check_beta(w, seqs=None):
    # a row whose threshold lies within the GEMM's rounding of a token may mask it either way: its
    # sequence is checked for validity only, and at least half the sequences are compared exactly
    gpu = run_fused_gpu(w, beta=w.beta)
    ref = oracle.verify_fused_workload(w, nthreads=oracle.max_threads(), seqs=seqs)
    res = compare(w, gpu, ref, seqs=seqs, amb_mask=FUSED_AMB_MASK, max_amb_frac=0.5, score_tol=FUSED_SCORE_TOL)
    # the observed error of masked rows (shown with pytest -s), against the bar it is held to
    print(f"masked fused rows: max |cd_lse err| {res['max_lse_err']:.3g}, "
          f"max |cd_logprob err| {res['max_logprob_err']:.3g} (bar {FUSED_SCORE_TOL:g})")
    return res


@pytest.mark.parametrize("beta", [0.1, 0.5])
def test_fused_plausibility_mask_small(beta):
    # one ragged row tile (V = 4099, K tails), and several row tiles over four vocabulary tiles.
    # The weights are scaled so the logits spread like the full-size model's (std about 3): the
    # threshold then lies in the tail, where few tokens sit within the GEMM's rounding of it.
    _check_beta(workloads.make_fused_torch(B=8, V=4099, H_exp=520, H_ama=136, seed=41, beta=beta, w_std=0.15))
    _check_beta(workloads.make_fused_torch(B=6, V=1000, H_exp=1024, H_ama=256, seed=42, beta=beta, w_std=0.1))


def test_fused_plausibility_mask_mixed_and_zero():
    # per-sequence thresholds, one of them 0 (unmasked); a zero beta vector gives the unmasked
    # call's results bit for bit (the two sweeps see the same logits)
    w = workloads.make_fused_torch(B=4, V=32000, H_exp=2048, H_ama=512, seed=43, w_std=0.075)
    w.beta = torch.tensor([0.0, 0.2, 0.5, 0.9], dtype=torch.float32, device=w.h_exp.device)
    _check_beta(w)
    a = dcd.dcd_verify_fused_lmhead(w.h_exp, w.w_exp, w.h_ama, w.w_ama, w.tokens, w.parents, w.alpha)
    z = dcd.dcd_verify_fused_lmhead(w.h_exp, w.w_exp, w.h_ama, w.w_ama, w.tokens, w.parents, w.alpha,
                                    torch.zeros_like(w.beta))
    torch.cuda.synchronize()
    for k in ("accept_len", "accept_path", "bonus", "cd_argmax", "cd_lse", "cd_logprob"):
        assert torch.equal(a[k], z[k]), k


def test_fused_plausibility_mask_full_size():
    # the full fused workload with beta = 0.5; the oracle recomputes two sequences
    w = workloads.make_fused_torch(beta=0.5)
    _check_beta(w, seqs=[3, 50, 61])


def test_fused_bad_beta_is_reported():
    w = workloads.make_fused_torch(B=2, V=1000, H_exp=256, H_ama=64, seed=44)
    beta = torch.tensor([0.1, 1.5], dtype=torch.float32, device=w.h_exp.device)
    gpu = run_fused_gpu(w, beta=beta)
    assert gpu["error_bits"] & 0x10
    assert gpu["accept_len"][1] == 0 and gpu["bonus"][1] == -1
