"""The verification calls inside CUDA graphs: a captured greedy or sampled call (the row kernel's
cooperative launch, the workspace memset and the tree walk's programmatic dependent launch)
replays to the same results as the eager call; several small calls captured back to back in one
graph each give their own results."""

import numpy as np
import pytest
import torch

import oracle
from paper_2608_12913_gb300 import dcd, workloads

pytestmark = pytest.mark.gpu


def _inputs(cfg, **kw):
    w = workloads.make_config(cfg, margin_fn=oracle.margin_fn, **kw)
    return w.to(torch.device("cuda"))


def _eq(a, b):
    for k in ("accept_len", "accept_path", "bonus", "cd_argmax"):
        assert torch.equal(a[k], b[k]), k
    assert torch.equal(a["cd_lse"], b["cd_lse"])
    assert torch.equal(a["cd_logprob"], b["cd_logprob"])


@pytest.mark.parametrize("sampled", [False, True])
def test_captured_call_replays_to_the_eager_results(sampled):
    w = _inputs(2 if sampled else 1, V=4099, B=3)
    dev = torch.device("cuda")
    out_e = dcd.alloc_outputs(w.B, w.N, dev)
    out_g = dcd.alloc_outputs(w.B, w.N, dev)
    ws_e = dcd.alloc_workspace(w.B, w.N, w.V, dev)
    ws_g = dcd.alloc_workspace(w.B, w.N, w.V, dev)

    def call(out, ws, stream=None):
        if sampled:
            return dcd.dcd_verify_sample(w.z_exp, w.z_ama, w.q, w.tokens, w.parents, w.alpha, w.temperature, w.seed, 7,
                                         w.beta, out=out, workspace=ws, stream=stream)
        return dcd.dcd_verify_greedy(w.z_exp, w.z_ama, w.tokens, w.parents, w.alpha, w.beta, out=out, workspace=ws,
                                     stream=stream)

    call(out_e, ws_e)
    torch.cuda.synchronize()
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        call(out_g, ws_g, stream=s)  # warm-up outside capture
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    for k in out_g:
        out_g[k].fill_(-7)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        call(out_g, ws_g, stream=torch.cuda.current_stream())
    for _ in range(3):
        g.replay()
        torch.cuda.synchronize()
        _eq(out_e, out_g)
        assert dcd.dcd_get_device_error(ws_g) == 0


def test_many_small_calls_in_one_graph():
    # eight independent single-sequence chain verifications (the latency-bound shape) captured
    # back to back, each with its own workspace and outputs
    dev = torch.device("cuda")
    ws_list, calls, eager = [], [], []
    for i in range(8):
        w = _inputs(0, seed=40 + i)
        out = dcd.alloc_outputs(w.B, w.N, dev)
        ws = dcd.alloc_workspace(w.B, w.N, w.V, dev, dtype=dcd.DCD_F32)
        e = dcd.dcd_verify_greedy(w.z_exp, w.z_ama, w.tokens, w.parents, w.alpha, w.beta)
        torch.cuda.synchronize()
        eager.append({k: v.clone() for k, v in e.items() if k != "workspace"})
        calls.append((w, out, ws))
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        for w, out, ws in calls:
            dcd.dcd_verify_greedy(w.z_exp, w.z_ama, w.tokens, w.parents, w.alpha, w.beta, out=out, workspace=ws,
                                  stream=s)
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for w, out, ws in calls:
            dcd.dcd_verify_greedy(w.z_exp, w.z_ama, w.tokens, w.parents, w.alpha, w.beta, out=out, workspace=ws,
                                  stream=torch.cuda.current_stream())
    g.replay()
    torch.cuda.synchronize()
    for (w, out, ws), e in zip(calls, eager):
        _eq(e, out)
