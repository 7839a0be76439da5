"""The device-side timeout path of the streaming kernel, exercised without a fault or a hang.

Every wait in the row kernel is bounded.  dcd_score_rows_ex takes a limit for the one wait that
has no copy in flight: a CTA whose rows are all claimed polls for residual passes that other CTAs
may still publish.  With a limit of one cycle that poll gives up at once.  The call must then
report DCD_DEVERR_TIMEOUT in its error word, the tree walk must fail every sequence (accept_len
0, bonus -1, a root-only path) rather than read records the call may not have rewritten, and the
same workspace must give correct results on the next call.
"""

import numpy as np
import pytest
import torch

import oracle
from paper_2608_12913_gb300 import dcd, workloads
from parity_util import compare, run_gpu

pytestmark = pytest.mark.gpu

DEVERR_TIMEOUT = 0x8


def _timed_out_call(wd, w, ws):
    o = dcd.dcd_score_rows(wd.z_exp, wd.z_ama, wd.tokens, wd.parents, wd.alpha, wd.beta, q=wd.q,
                           temperature=wd.temperature, seed=w.seed, offset=w.offset, workspace=ws,
                           poll_limit_cycles=1)
    dcd.dcd_tree_walk(w.B, w.N, w.V, o, ws)
    torch.cuda.synchronize()
    return o


def test_poll_timeout_is_reported_and_fails_every_sequence():
    w = workloads.make_config(3, B=6, V=20011, seed=71, margin_fn=oracle.margin_fn)
    wd = w.to(torch.device("cuda"))
    ws = dcd.alloc_workspace(w.B, w.N, w.V, wd.z_exp.device)
    # a correct call first, so the workspace holds valid-looking records of the same inputs
    good = run_gpu(w, sampled=True, workspace=ws)
    assert good["error_bits"] == 0
    assert (good["accept_len"] > 0).any()

    o = _timed_out_call(wd, w, ws)
    bits = dcd.dcd_get_device_error(ws)
    assert bits & DEVERR_TIMEOUT
    assert (o["accept_len"].cpu().numpy() == 0).all()
    assert (o["bonus"].cpu().numpy() == -1).all()
    path = o["accept_path"].cpu().numpy()
    assert (path[:, 0] == 0).all() and (path[:, 1:] == -1).all()

    # the context and the workspace stay usable: the next call is correct and clears the word
    again = run_gpu(w, sampled=True, workspace=ws)
    assert again["error_bits"] == 0
    compare(w, again, oracle.verify_workload(w, nthreads=oracle.max_threads()))
    for k in ("accept_len", "accept_path", "bonus", "cd_argmax"):
        assert np.array_equal(again[k], good[k]), k


def test_poll_timeout_on_a_greedy_call():
    # an all-greedy call has no residual passes, but a CTA that runs out of rows still polls
    # until every row is done; the one-cycle bound makes that poll give up too
    w = workloads.make_config(1, B=2, V=9001, seed=72, margin_fn=oracle.margin_fn)
    wd = w.to(torch.device("cuda"))
    ws = dcd.alloc_workspace(w.B, w.N, w.V, wd.z_exp.device)
    o = dcd.dcd_score_rows(wd.z_exp, wd.z_ama, wd.tokens, wd.parents, wd.alpha, wd.beta, workspace=ws,
                           poll_limit_cycles=1)
    dcd.dcd_tree_walk(w.B, w.N, w.V, o, ws)
    torch.cuda.synchronize()
    assert dcd.dcd_get_device_error(ws) & DEVERR_TIMEOUT
    assert (o["accept_len"].cpu().numpy() == 0).all()
    assert (o["bonus"].cpu().numpy() == -1).all()
    g = run_gpu(w, sampled=False, stages=2, workspace=ws)
    assert g["error_bits"] == 0
    compare(w, g, oracle.verify_workload(w, nthreads=oracle.max_threads()))
