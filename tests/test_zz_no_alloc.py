"""The allocation-free entry point against the workspace one.

dcd_verify_sample_noalloc serves callers that cannot allocate device memory (an engine
plugin whose memory is all reserved by the engine's allocator, or a hook that must not call
cudaMalloc/cudaFree).  It keeps its scratch in an array built into the library, so this test
runs it twice in a row, through the C ABI, and checks both calls against the ordinary
workspace entry point on the same inputs.  The file sorts last so that a run stopping at the
first failure has already run every other test; it also passes when run alone.
"""

import numpy as np
import pytest
import torch

from paper_2608_12913_gb300 import dcd, workloads

pytestmark = pytest.mark.gpu

SCORE_TOL = 1e-4


def _check_same(a, b):
    for k in ("accept_len", "accept_path", "bonus", "cd_argmax"):
        assert np.array_equal(a[k].cpu().numpy(), b[k].cpu().numpy()), k
    for k in ("cd_logprob", "cd_lse"):
        x, y = a[k].cpu().numpy(), b[k].cpu().numpy()
        assert np.array_equal(np.isneginf(x), np.isneginf(y)), k
        fin = np.isfinite(x)
        assert np.abs(x[fin] - y[fin]).max(initial=0.0) <= SCORE_TOL, k


def test_noalloc_matches_workspace_entry_point_on_two_calls():
    w = workloads.make_config(3, B=8, V=20011, seed=61).to("cuda")
    args = (w.z_exp, w.z_ama, w.q, w.tokens, w.parents, w.alpha, w.temperature, w.seed)
    for offset in (5, 6):  # two calls in a row on the shared scratch
        ref = dcd.dcd_verify_sample(*args, offset, w.beta)
        got = dcd.dcd_verify_sample_noalloc(*args, offset, w.beta)
        torch.cuda.synchronize()
        _check_same(got, ref)
    # a second workload of another shape reuses the same scratch
    w2 = workloads.make_config(1, B=3, V=5003, seed=62).to("cuda")
    q2 = torch.zeros_like(w2.z_exp, dtype=torch.float32)
    ref = dcd.dcd_verify_sample(w2.z_exp, w2.z_ama, q2, w2.tokens, w2.parents, w2.alpha, w2.temperature, 1, 0)
    got = dcd.dcd_verify_sample_noalloc(w2.z_exp, w2.z_ama, q2, w2.tokens, w2.parents, w2.alpha, w2.temperature,
                                        1, 0)
    torch.cuda.synchronize()
    _check_same(got, ref)


def _residual_tv(a, b):
    return 0.5 * np.abs(a["residual"].cpu().numpy() - b["residual"].cpu().numpy()).sum(axis=1).max(initial=0.0)


@pytest.mark.parametrize("distinct", [False, True])
def test_noalloc_residual_and_sibling_rules_match_workspace_entry_point(distinct):
    # the residual output (the distribution each bonus token was drawn from) and both sibling
    # rules, two calls in a row on the shared scratch
    w = workloads.make_config(3, B=6, V=12007, seed=63).to("cuda")
    args = (w.z_exp, w.z_ama, w.q, w.tokens, w.parents, w.alpha, w.temperature, w.seed)
    for offset in (11, 12):
        ref = dcd.dcd_verify_sample(*args, offset, w.beta, residual=True, distinct=distinct)
        got = dcd.dcd_verify_sample_noalloc(*args, offset, w.beta, residual=True, distinct=distinct)
        torch.cuda.synchronize()
        _check_same(got, ref)
        assert _residual_tv(got, ref) <= 1e-5


def test_noalloc_reports_device_input_errors_per_sequence():
    # a parent index that breaks the ordering rule and a token outside the vocabulary (both
    # built on the host; the kernel checks them and writes no out-of-range address): those
    # sequences report accept_len = 0 and bonus = -1, the others are unaffected
    w = workloads.make_config(3, B=4, V=9001, seed=64)
    parents = w.parents.clone()
    tokens = w.tokens.clone()
    parents[1, 5] = 7  # node 5 claims a later node as its parent
    tokens[2, 3] = w.V + 5
    wd = w.to("cuda")
    pd, td = parents.to("cuda"), tokens.to("cuda")
    args = (wd.z_exp, wd.z_ama, wd.q, td, pd, wd.alpha, wd.temperature, w.seed, 3, wd.beta)
    got = dcd.dcd_verify_sample_noalloc(*args)
    ref = dcd.dcd_verify_sample(*args)
    torch.cuda.synchronize()
    for b in (1, 2):
        assert int(got["accept_len"][b]) == 0 and int(got["bonus"][b]) == -1
    assert dcd.dcd_get_device_error(ref["workspace"]) & 0x3
    for k in ("accept_len", "accept_path", "bonus"):
        assert np.array_equal(got[k].cpu().numpy(), ref[k].cpu().numpy()), k
    # the next call on the same scratch is clean again
    good = dcd.dcd_verify_sample_noalloc(wd.z_exp, wd.z_ama, wd.q, wd.tokens, wd.parents, wd.alpha, wd.temperature,
                                         w.seed, 3, wd.beta)
    ref = dcd.dcd_verify_sample(wd.z_exp, wd.z_ama, wd.q, wd.tokens, wd.parents, wd.alpha, wd.temperature, w.seed, 3,
                                wd.beta)
    torch.cuda.synchronize()
    _check_same(good, ref)


def test_noalloc_rejects_shapes_beyond_its_capacity():
    import ctypes
    lib = dcd.load()
    P = ctypes.c_void_p(0x10000)
    big = dcd.make_shape(2000, 60, 128256, dcd.DCD_BF16)  # 120000 rows need far more than 4 MiB
    rc = lib.dcd_verify_sample_noalloc(ctypes.byref(big), P, P, P, P, P, P, None, P, 0, 0, P, P, P, None, None,
                                       None, None, None)
    assert rc == -3
