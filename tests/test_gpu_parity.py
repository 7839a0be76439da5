"""GPU (libdcd.so through the C ABI) against the fp64 oracle on the same seeded inputs.

Covers the four streaming workloads (tiny fp32 chain; 60-node tree greedy; the same
tree sampled at T = 1; the 32-sequence mixed batch, reduced and at full size), the
plausibility mask, every ring depth and the plain-load path, ragged and tiny
vocabularies, degenerate trees, device-side input errors, determinism and offsets.
Bars and the ambiguity rule are in parity_util.
"""

import numpy as np
import pytest
import torch
from scipy import special, stats

import oracle
from paper_2608_12913_gb300 import dcd, workloads
from parity_util import AMB_MASK, compare, run_gpu

pytestmark = pytest.mark.gpu


def _oracle(w, residual=False, seqs=None):
    return oracle.verify_workload(w, nthreads=oracle.max_threads(), want_residual=residual, seqs=seqs)


def test_config0_tiny_chain_fp32_greedy():
    w = workloads.make_config(0, margin_fn=oracle.margin_fn)
    g = run_gpu(w, sampled=False)
    r = _oracle(w)
    compare(w, g, r)


def test_config1_tree_greedy_full_vocab():
    w = workloads.make_config(1, margin_fn=oracle.margin_fn)
    g = run_gpu(w, sampled=False)
    r = _oracle(w)
    st = compare(w, g, r)
    assert st["ambiguous_seqs"] == 0


def test_config2_tree_sampled_full_vocab_with_residual():
    w = workloads.make_config(2, margin_fn=oracle.margin_fn)
    g = run_gpu(w, sampled=True, residual=True)
    r = _oracle(w, residual=True)
    compare(w, g, r, check_residual=True)


def test_config3_reduced_mixed_batch():
    w = workloads.make_config(3, B=12, V=20011, margin_fn=oracle.margin_fn)
    g = run_gpu(w, sampled=True, residual=True)
    r = _oracle(w, residual=True)
    compare(w, g, r, check_residual=True)


def test_wide_vocabulary_mixed_batch():
    # a 262K vocabulary (ragged: not a multiple of a stage, a race block or a residual piece)
    w = workloads.make_config(3, B=2, V=262147, seed=43, margin_fn=oracle.margin_fn)
    g = run_gpu(w, sampled=True, residual=True)
    r = _oracle(w, residual=True)
    compare(w, g, r, check_residual=True)


def test_vocabulary_beyond_shared_memory_is_unsupported():
    # the row kernel keeps 8 bytes per 1024 vocabulary tokens of a row in shared memory; a
    # vocabulary past that returns DCD_ERR_UNSUPPORTED before any launch
    V = 1 << 25
    z = torch.zeros((2, V), dtype=torch.bfloat16, device="cuda")
    q = torch.full((2, V), 1.0 / V, dtype=torch.float32, device="cuda")
    tokens = torch.tensor([[0, 1]], dtype=torch.int32, device="cuda")
    parents = torch.tensor([[-1, 0]], dtype=torch.int32, device="cuda")
    one = torch.ones(1, dtype=torch.float32, device="cuda")
    with pytest.raises(dcd.DcdError) as e:
        dcd.dcd_verify_sample(z, z, q, tokens, parents, one * 0.1, one, 1, 0)
    assert e.value.status == -3


def test_config3_full_size_sampled_sequences():
    """The 32 x 60-node, V = 128256 batch in the launch configuration the benchmark times;
    the oracle recomputes 8 of its sequences (4 greedy, 4 sampled) one by one."""
    w = workloads.make_config_torch(3, device="cuda")
    g = run_gpu(w, sampled=True)
    seqs = [0, 2, 29, 30, 1, 3, 5, 31]
    r = _oracle(w, seqs=seqs)
    compare(w, g, r, seqs=seqs, max_amb_frac=0.25)


@pytest.mark.parametrize("beta", [1e-3, 0.1, 0.5, 1.0])
@pytest.mark.parametrize("sampled", [False, True])
def test_plausibility_mask(beta, sampled):
    # beta = 1 keeps only the expert's argmax set: pi_CD is a point mass there.  Its mask test,
    # z_p - max z_p >= log 1 = 0, is exact in fp32 and fp64 alike (0 for the max token, nonzero for
    # any other), so the max token's zero distance to the threshold is no ambiguity.
    cfg = 2 if sampled else 1
    w = workloads.make_config(cfg, B=3, V=9001, beta=beta, seed=40 + int(beta * 100), margin_fn=oracle.margin_fn)
    g = run_gpu(w, sampled=sampled, residual=sampled)
    r = _oracle(w, residual=sampled)
    compare(w, g, r, check_residual=sampled, amb_mask=0.0 if beta == 1.0 else AMB_MASK)


@pytest.mark.parametrize("stages", [2, 3, 4, 6])
@pytest.mark.parametrize("plain", [False, True])
def test_every_ring_depth(stages, plain):
    w = workloads.make_config(3, B=4, V=12347, seed=7, margin_fn=oracle.margin_fn)
    g = run_gpu(w, sampled=True, stages=stages, plain=plain)
    r = _oracle(w)
    compare(w, g, r)


@pytest.mark.parametrize("V", [1, 3, 7, 8, 9, 31, 1000, 1001, 4099])
def test_ragged_and_tiny_vocabularies(V):
    for temps in ((0.0,), (0.8,)):
        w = workloads.generate(name="ragged", B=3, V=V, dtype="bf16", spikes=(1, 1), alphas=(0.3,),
                               temperatures=temps, levels=(1, 3, 2, 1), seed=V, margin_fn=oracle.margin_fn)
        g = run_gpu(w, sampled=temps[0] > 0, residual=temps[0] > 0)
        r = _oracle(w, residual=temps[0] > 0)
        compare(w, g, r, check_residual=temps[0] > 0, max_amb_frac=0.34)


def test_root_only_and_star_trees():
    for levels in ((1,), (1, 20), (1, 1, 1, 1, 1, 1, 1, 1)):
        for temps in ((0.0,), (1.0,), (0.0, 1.3)):
            w = workloads.generate(name="shapes", B=4, V=777, dtype="f32", spikes=(2, 2), alphas=(0.1, 0.5),
                                   temperatures=temps, levels=levels, seed=len(levels), margin_fn=oracle.margin_fn,
                                   max_children=32)
            g = run_gpu(w, sampled=max(temps) > 0, residual=max(temps) > 0)
            r = _oracle(w, residual=max(temps) > 0)
            compare(w, g, r, check_residual=max(temps) > 0, max_amb_frac=0.25)
            if levels == (1,):
                assert np.all(g["accept_len"] == 0)


def test_unaligned_row_stride_uses_plain_loads():
    w = workloads.make_config(2, B=2, V=3001, seed=9, margin_fn=oracle.margin_fn)
    wd = w.to("cuda")
    R, V = w.R, w.V
    zp = torch.zeros((R, V + 3), dtype=wd.z_exp.dtype, device="cuda")
    zq = torch.zeros_like(zp)
    zp[:, 1:V + 1] = wd.z_exp
    zq[:, 1:V + 1] = wd.z_ama
    o = dcd.dcd_verify_sample(zp[:, 1:V + 1], zq[:, 1:V + 1], wd.q, wd.tokens, wd.parents, wd.alpha, wd.temperature,
                              w.seed, w.offset, wd.beta)
    ref = run_gpu(w, sampled=True)
    torch.cuda.synchronize()
    assert np.array_equal(o["accept_len"].cpu().numpy(), ref["accept_len"])
    assert np.array_equal(o["accept_path"].cpu().numpy(), ref["accept_path"])
    assert np.array_equal(o["bonus"].cpu().numpy(), ref["bonus"])
    np.testing.assert_allclose(o["cd_lse"].cpu().numpy(), ref["cd_lse"], atol=1e-5)


def test_duplicate_siblings_and_zero_draft_probability():
    w = workloads.make_config(2, B=6, V=501, seed=13, margin_fn=oracle.margin_fn)
    tok = w.tokens.clone()
    q = w.q.clone()
    for b in range(w.B):
        kids = workloads.children_lists(w.parents[b].numpy())
        for n, ch in enumerate(kids):
            if len(ch) >= 2:
                tok[b, ch[1]] = tok[b, ch[0]]  # duplicate sibling token
            if len(ch) >= 3:
                q[b * w.N + n, int(tok[b, ch[2]])] = 0.0  # drafter gave this token no mass
    w.tokens, w.q = tok, q
    for sampled in (False, True):
        g = run_gpu(w, sampled=sampled, residual=sampled)
        r = _oracle(w if sampled else _greedy(w), residual=sampled)
        compare(w, g, r, check_residual=sampled)


def _greedy(w):
    import dataclasses
    return dataclasses.replace(w, temperature=torch.zeros_like(w.temperature))


def test_split_steps_equal_verify_and_determinism():
    w = workloads.make_config(3, B=6, V=4001, seed=17)
    a = run_gpu(w, sampled=True)
    b = run_gpu(w, sampled=True, stages=0)
    wd = w.to("cuda")
    o = dcd.dcd_score_rows(wd.z_exp, wd.z_ama, wd.tokens, wd.parents, wd.alpha, wd.beta, q=wd.q,
                           temperature=wd.temperature, seed=w.seed, offset=w.offset)
    dcd.dcd_tree_walk(w.B, w.N, w.V, o, o["workspace"])
    torch.cuda.synchronize()
    for k in ("accept_len", "accept_path", "bonus", "cd_argmax"):
        assert np.array_equal(a[k], b[k])
        assert np.array_equal(a[k], o[k].cpu().numpy())
    assert np.array_equal(a["cd_lse"], b["cd_lse"])  # bitwise: same launch, same order


def test_offsets_change_the_draws():
    w = workloads.make_config(2, B=8, V=64, seed=3)
    outs = [run_gpu(w, sampled=True, offset=o) for o in range(6)]
    bon = np.stack([o["bonus"] for o in outs])
    assert len({tuple(x) for x in bon}) > 1
    again = run_gpu(w, sampled=True, offset=2)
    assert np.array_equal(again["bonus"], outs[2]["bonus"])
    for o in range(6):
        r = _oracle(__import__("dataclasses").replace(w, offset=o))
        compare(__import__("dataclasses").replace(w, offset=o), outs[o], r)


def test_lossless_on_the_gpu_monte_carlo():
    """The GPU's first emitted token follows pi_CD when siblings are drawn i.i.d. from q (App. B.3)."""
    rng = np.random.default_rng(5)
    V, B, m = 6, 60000, 3
    N = m + 1
    zp = rng.standard_normal(V)
    zq = 0.7 * zp + rng.standard_normal(V)
    qd = special.softmax(zp + 0.8 * rng.standard_normal(V)).astype(np.float32)
    alpha, T = 0.3, 1.0
    tokens = np.zeros((B, N), dtype=np.int32)
    qn = qd.astype(np.float64) / qd.sum(dtype=np.float64)
    tokens[:, 1:] = rng.choice(V, size=(B, m), p=qn)
    parents = np.tile(np.array([-1] + [0] * m, dtype=np.int32), (B, 1))
    dev = "cuda"
    Z = torch.tensor(np.tile(zp.astype(np.float32), (B * N, 1)), device=dev)
    Zq = torch.tensor(np.tile(zq.astype(np.float32), (B * N, 1)), device=dev)
    Q = torch.tensor(np.tile(qd, (B * N, 1)), device=dev)
    o = dcd.dcd_verify_sample(Z, Zq, Q, torch.tensor(tokens, device=dev), torch.tensor(parents, device=dev),
                              torch.full((B,), alpha, device=dev), torch.full((B,), T, device=dev), 11, 0)
    torch.cuda.synchronize()
    L = o["accept_len"].cpu().numpy()
    path = o["accept_path"].cpu().numpy()
    first = np.where(L > 0, tokens[np.arange(B), path[:, 1].clip(0)], o["bonus"].cpu().numpy())
    pi = np.exp(oracle.row_logpi(zp.astype(np.float32).astype(np.float64), zq.astype(np.float32).astype(np.float64),
                                 alpha, 0.0, T)["logpi"])
    counts = np.bincount(first, minlength=V)
    assert stats.chisquare(counts, B * pi).pvalue > 1e-4


def test_device_input_errors_are_reported_not_trapped():
    w = workloads.make_config(1, B=3, V=1000, seed=23)
    wd = w.to("cuda")
    good = run_gpu(w, sampled=False)
    assert good["error_bits"] == 0
    cases = []
    p = wd.parents.clone()
    p[1, 5] = 7  # parent after its child
    cases.append(("parents", p, 0x1))
    t = wd.tokens.clone()
    t[2, 3] = w.V  # out of range
    cases.append(("tokens", t, 0x2))
    for what, arr, bit in cases:
        kw = dict(parents=wd.parents, tokens=wd.tokens)
        kw[what] = arr
        o = dcd.dcd_verify_greedy(wd.z_exp, wd.z_ama, kw["tokens"], kw["parents"], wd.alpha, wd.beta)
        bits = dcd.dcd_get_device_error(o["workspace"])
        assert bits & bit
        bad_seq = 1 if what == "parents" else 2
        assert int(o["accept_len"][bad_seq]) == 0 and int(o["bonus"][bad_seq]) == -1
        assert int(o["bonus"][0]) == int(good["bonus"][0])
        # the next valid call on the same workspace reports a clean word
        o2 = dcd.dcd_verify_greedy(wd.z_exp, wd.z_ama, wd.tokens, wd.parents, wd.alpha, wd.beta,
                                   workspace=o["workspace"])
        assert dcd.dcd_get_device_error(o2["workspace"]) == 0
    z = wd.z_exp.clone()
    z[4, 17] = float("nan")
    o = dcd.dcd_verify_greedy(z, wd.z_ama, wd.tokens, wd.parents, wd.alpha, wd.beta)
    assert dcd.dcd_get_device_error(o["workspace"]) & 0x4
    a = wd.alpha.clone()
    a[0] = -1.0
    o = dcd.dcd_verify_greedy(wd.z_exp, wd.z_ama, wd.tokens, wd.parents, a, wd.beta)
    assert dcd.dcd_get_device_error(o["workspace"]) & 0x10


def test_largest_tree_chain_of_max_nodes():
    # N = 1024 (the largest tree the library accepts): a chain of depth 1023, greedy and sampled
    for temp in (0.0, 1.0):
        w = workloads.make_config(0, V=1000, chain_len=1024, B=1, temperatures=(temp,), dtype="f32", seed=21)
        gpu = run_gpu(w, sampled=temp > 0)
        ref = oracle.verify_workload(w, nthreads=oracle.max_threads())
        compare(w, gpu, ref)


def test_binding_rejects_outputs_and_vectors_it_cannot_write_or_read():
    # checked on the host, before any launch: a wrong output shape would let a kernel write past
    # the caller's tensor, a strided parameter vector would be read as dense
    w = workloads.make_config(1, B=2, V=1000, seed=51).to("cuda")
    out = dcd.alloc_outputs(w.B, w.N, "cuda")
    bad = dict(out, accept_path=torch.empty((w.B, w.N - 1), dtype=torch.int32, device="cuda"))
    with pytest.raises(ValueError):
        dcd.dcd_verify_greedy(w.z_exp, w.z_ama, w.tokens, w.parents, w.alpha, w.beta, out=bad)
    bad = dict(out, cd_lse=torch.empty((w.B, w.N), dtype=torch.float64, device="cuda"))
    with pytest.raises(TypeError):
        dcd.dcd_verify_greedy(w.z_exp, w.z_ama, w.tokens, w.parents, w.alpha, w.beta, out=bad)
    bad = {k: v for k, v in out.items() if k != "bonus"}
    with pytest.raises(ValueError):
        dcd.dcd_verify_greedy(w.z_exp, w.z_ama, w.tokens, w.parents, w.alpha, w.beta, out=bad)
    strided = torch.zeros(2 * w.B, dtype=torch.float32, device="cuda")[::2]
    with pytest.raises(ValueError):
        dcd.dcd_verify_greedy(w.z_exp, w.z_ama, w.tokens, w.parents, strided, w.beta, out=out)
    o = dcd.dcd_verify_greedy(w.z_exp, w.z_ama, w.tokens, w.parents, w.alpha, w.beta, out=out)
    torch.cuda.synchronize()
    assert o["accept_len"] is out["accept_len"]

