"""Property-based pins of the oracle (no GPU).  Hypothesis draws tiny vocabularies, logits and the
parameters, and the oracle must agree with definitions evaluated independently here:

* the row target: pi_CD = pi_p^(1+alpha) pi_q^(-alpha) over P_beta = {x : pi_p(x) >= beta max
  pi_p} (Eq. 1, Sec. 2.1), raised to 1/T and normalised, in product form -- and its argmax;
* the residual chain of Algorithm 1 for one sibling list: after k rejections the residual is
  normalise(max(0, r_{k-1} - q)), applied literally step by step from r_0 = pi_CD.

Cases whose decision lies within rounding of a threshold (the mask boundary, an argmax tie) are
discarded, as the parity bars do."""

import numpy as np
import pytest

hypothesis = pytest.importorskip("hypothesis")
from hypothesis import assume, given, settings  # noqa: E402
from hypothesis import strategies as st  # noqa: E402

import oracle  # noqa: E402

PARAMS = dict(
    V=st.integers(1, 48),
    seed=st.integers(0, 2**31 - 1),
    alpha=st.floats(0.0, 2.0),
    beta=st.one_of(st.just(0.0), st.floats(1e-4, 1.0)),
    T=st.floats(0.25, 2.0),
    scale=st.floats(0.1, 4.0),
)


def _rows(seed, V, scale):
    rng = np.random.default_rng(seed)
    zp = scale * rng.standard_normal(V)
    zq = 0.7 * zp + scale * rng.standard_normal(V)
    return zp, zq


def _product_form(zp, zq, alpha, beta, T):
    p = np.exp(zp - zp.max())
    p /= p.sum()
    qa = np.exp(zq - zq.max())
    qa /= qa.sum()
    keep = p >= beta * p.max()
    w = np.where(keep, (p ** (1.0 + alpha) * qa ** (-alpha)) ** (1.0 / T), 0.0)
    return p, keep, w / w.sum()


@settings(max_examples=300, deadline=None)
@given(**PARAMS)
def test_row_target_equals_the_product_form(V, seed, alpha, beta, T, scale):
    zp, zq = _rows(seed, V, scale)
    p, keep, pi = _product_form(zp, zq, alpha, beta, T)
    if beta > 0:  # no token within rounding of the mask threshold
        gap = np.abs(np.log(p) - np.log(beta * p.max()))
        assume(np.all(gap[p < p.max()] > 1e-9))
    r = oracle.row_logpi(zp, zq, alpha=alpha, beta=beta, T=T)
    np.testing.assert_allclose(np.exp(r["logpi"]), pi, rtol=1e-9, atol=1e-300)
    score = np.where(keep, (1.0 + alpha) * np.log(p) - alpha * np.log(np.exp(zq - zq.max()) /
                                                                        np.exp(zq - zq.max()).sum()), -np.inf)
    top = np.sort(score)[::-1]
    assume(V == 1 or not np.isfinite(top[1]) or top[0] - top[1] > 1e-9)
    assert r["argmax"] == int(np.argmax(score))


@settings(max_examples=200, deadline=None)
@given(m=st.integers(1, 4), **PARAMS)
def test_residual_chain_equals_literal_renormalisation(m, V, seed, alpha, beta, T, scale):
    zp, zq = _rows(seed, V, scale)
    p, _, pi = _product_form(zp, zq, alpha, beta, T)
    if beta > 0:  # no token within rounding of the mask threshold
        gap = np.abs(np.log(p) - np.log(beta * p.max()))
        assume(np.all(gap[p < p.max()] > 1e-9))
    rng = np.random.default_rng(seed ^ 0x5EED)
    q = rng.dirichlet(np.full(V, 0.7)).astype(np.float32).astype(np.float64)  # q is fp32 in the ABI
    kids = rng.integers(0, V, size=m).astype(np.int32)
    # Algorithm 1, literally: r_0 = pi; each rejection r <- normalise(max(0, r - q)); a step without
    # residual mass leaves r as it is (reading c6)
    r = pi.copy()
    ratios = []
    for t in kids:
        ratios.append(r[t] / q[t] if q[t] > 0 else (np.inf if r[t] > 0 else 0.0))
        nxt = np.maximum(r - q, 0.0)
        mass = nxt.sum()
        assume(mass == 0.0 or mass > 1e-6)  # a mass within rounding of zero decides nothing here
        if mass > 0.0:
            r = nxt / mass
    assume(np.all(np.isfinite(ratios)))
    got_ratios, got_r = oracle.row_chain(zp, zq, alpha, beta, T, q, kids)
    np.testing.assert_allclose(got_ratios, ratios, rtol=1e-8, atol=1e-12)
    np.testing.assert_allclose(got_r, r, rtol=1e-8, atol=1e-12)


@settings(max_examples=150, deadline=None)
@given(V=st.integers(2, 24), seed=st.integers(0, 2**31 - 1), alpha=st.floats(0.0, 2.0),
       beta=st.one_of(st.just(0.0), st.floats(1e-4, 1.0)), N=st.integers(1, 20), hit=st.floats(0.0, 1.0))
def test_greedy_walk_follows_the_row_argmaxes(V, seed, alpha, beta, N, hit):
    """The greedy rule on a random tree (Algorithm 1 in the T -> 0 limit, sibling lists): from the
    root, descend into the first child (lowest node id) whose token is its parent row's CD argmax;
    accept_len counts the descents and the bonus is the argmax of the row where the walk stops."""
    alpha, beta = float(np.float32(alpha)), float(np.float32(beta))  # the oracle's fp32 parameters
    rng = np.random.default_rng(seed)
    parents = np.array([-1] + [int(rng.integers(0, i)) for i in range(1, N)], dtype=np.int32)
    zp = 2.0 * rng.standard_normal((N, V))
    zq = 0.7 * zp + 1.5 * rng.standard_normal((N, V))
    arg = np.empty(N, dtype=np.int64)
    for n in range(N):
        p, keep, _ = _product_form(zp[n], zq[n], alpha, beta, 1.0)
        lq = zq[n] - zq[n].max() - np.log(np.exp(zq[n] - zq[n].max()).sum())
        score = np.where(keep, (1.0 + alpha) * np.log(p) - alpha * lq, -np.inf)
        top = np.sort(score)[::-1]
        assume(V == 1 or not np.isfinite(top[1]) or top[0] - top[1] > 1e-9)
        if beta > 0:
            gap = np.abs(np.log(p) - np.log(beta * p.max()))
            assume(np.all(gap[p < p.max()] > 1e-9))
        arg[n] = int(np.argmax(score))
    # drafts: each node's token is its parent row's argmax with probability `hit`, else random
    tokens = np.zeros(N, dtype=np.int32)
    for c in range(1, N):
        tokens[c] = arg[parents[c]] if rng.random() < hit else int(rng.integers(0, V))
    # the walk
    cur, path = 0, [0]
    while True:
        nxt = [c for c in range(cur + 1, N) if parents[c] == cur and tokens[c] == arg[cur]]
        if not nxt:
            break
        cur = nxt[0]
        path.append(cur)
    r = oracle.verify(B=1, N=N, V=V, dtype="f64", z_exp=zp.reshape(1 * N, V), z_ama=zq.reshape(N, V),
                      tokens=tokens.reshape(1, N), parents=parents.reshape(1, N),
                      alpha=np.array([alpha], np.float32), beta=np.array([beta], np.float32),
                      temperature=np.zeros(1, np.float32))
    assert r["accept_len"][0] == len(path) - 1
    assert list(r["accept_path"][0][: len(path)]) == path
    assert np.all(r["accept_path"][0][len(path):] == -1)
    assert r["bonus"][0] == arg[cur]
