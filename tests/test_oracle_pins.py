"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each test checks the oracle against something other than itself: published
known-answer vectors, a product-form brute force of Eq. 1, a library special
case, the KL-decomposition lemma (App. B), the lossless theorem (App. B.3) by
exact enumeration and by Monte Carlo, Algorithm 1 on chains, and tree paths
whose outcome is fixed by construction.
"""

import itertools
import os

import numpy as np
import pytest
from scipy import special, stats

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rows(rng, V, scale=2.0):
    zp = scale * rng.standard_normal(V)
    zq = 0.7 * zp + 1.5 * rng.standard_normal(V)
    return zp, zq


# ----------------------------------------------------------------------------- Philox

def test_philox_known_answers():
    """Random123 kat_vectors for Philox4x32-10 (Salmon et al., SC'11)."""
    rows = [l.split() for l in open(os.path.join(GOLDEN, "philox4x32_10_kat.txt")) if l.strip() and l[0] != "#"]
    assert len(rows) == 3
    for r in rows:
        v = [int(x, 16) for x in r]
        out = oracle.philox(v[0:4], v[4:6])
        assert [int(x) for x in out] == v[6:10]


def test_uniform_conversion_open_interval_and_fp32_exact():
    for w in (0, 1, 511, 512, 0x7FFFFFFF, 0xFFFFFFFF, 0x12345678):
        u = oracle.u01(w)
        assert 0.0 < u < 1.0
        assert float(np.float32(u)) == u  # fp32 holds every value exactly
    assert oracle.u01(0) == 0.5 * 2.0 ** -23
    assert oracle.u01(0xFFFFFFFF) == 1.0 - 0.5 * 2.0 ** -23


def test_uniform_streams_are_uniform_and_distinct():
    accept = np.array([oracle.accept_uniform(7, 3, g) for g in range(20000)])
    race = np.array([oracle.race_uniform(7, 3, 11, x) for x in range(20000)])
    for u in (accept, race):
        assert stats.kstest(u, "uniform").pvalue > 1e-4
    assert abs(np.corrcoef(accept, race)[0, 1]) < 0.05
    # another offset gives another stream
    other = np.array([oracle.accept_uniform(7, 4, g) for g in range(2000)])
    assert np.mean(other == accept[:2000]) < 0.01


# ----------------------------------------------------------------------------- Eq. 1 target

@pytest.mark.parametrize("V", [7, 64, 1000])
def test_alpha_zero_is_expert_log_softmax(V):
    """alpha = 0: CD reduces to the expert distribution (Sec. 3.3, alpha = 0 boundary)."""
    rng = np.random.default_rng(V)
    zp, zq = _rows(rng, V)
    r = oracle.row_logpi(zp, zq, alpha=0.0, beta=0.0, T=1.0)
    np.testing.assert_allclose(r["logpi"], special.log_softmax(zp), rtol=0, atol=1e-12)
    assert r["argmax"] == int(np.argmax(zp))


@pytest.mark.parametrize("alpha,beta,T", [(0.1, 0.0, 1.0), (0.5, 0.0, 1.0), (1.0, 0.0, 0.7),
                                          (0.2, 0.1, 1.0), (0.05, 0.5, 1.3), (0.3, 1e-3, 0.5)])
def test_product_form_brute_force(alpha, beta, T):
    """pi_CD = pi_p^(1+a) pi_q^(-a) / Z (Eq. 1), masked to P_beta (Sec. 2.1), evaluated as products."""
    rng = np.random.default_rng(int(alpha * 100 + beta * 1000 + T * 10))
    for V in (5, 17, 64):
        zp, zq = _rows(rng, V, scale=1.0)
        p = np.exp(zp) / np.exp(zp).sum()
        qa = np.exp(zq) / np.exp(zq).sum()
        w = (p ** (1.0 + alpha) * qa ** (-alpha)) ** (1.0 / T)
        w = np.where(p >= beta * p.max(), w, 0.0)
        pi = w / w.sum()
        r = oracle.row_logpi(zp, zq, alpha=alpha, beta=beta, T=T)
        np.testing.assert_allclose(np.exp(r["logpi"]), pi, rtol=1e-11, atol=1e-15)
        assert r["argmax"] == int(np.argmax(np.where(w > 0, np.log(p ** (1 + alpha) * qa ** (-alpha)), -np.inf)))


def test_kl_decomposition_lemma():
    """App. B, Lemma kl_decomposition, at beta = 0 and T = 1."""
    rng = np.random.default_rng(5)
    for V, alpha in [(50, 0.1), (500, 0.5), (3000, 1.0), (200, 0.0)]:
        zp, zq = _rows(rng, V)
        lp, lq = special.log_softmax(zp), special.log_softmax(zq)
        p, qa = np.exp(lp), np.exp(lq)
        r = oracle.row_logpi(zp, zq, alpha=alpha, beta=0.0, T=1.0)
        lpi = r["logpi"]
        logZ = r["log_zcd"]
        kl = lambda a, la, lb: float(np.sum(a * (la - lb)))  # noqa: E731
        assert abs(kl(p, lp, lpi) - (logZ - alpha * kl(p, lp, lq))) < 1e-10
        assert abs(kl(qa, lq, lpi) - (logZ + (1 + alpha) * kl(qa, lq, lp))) < 1e-10
        # Z_CD = sum pi_p^(1+a) pi_q^(-a) (App. B.3)
        assert abs(logZ - np.log(np.sum(p ** (1 + alpha) * qa ** (-alpha)))) < 1e-10
        # the raw-logit normaliser differs from log Z_CD by (1+a) lse_p - a lse_q
        assert abs(r["cd_lse"] - (logZ + (1 + alpha) * r["lse_p"] - alpha * r["lse_q"])) < 1e-9


def test_plausibility_mask_invariants():
    """P_beta (Sec. 2.1): nested in beta, always holds argmax pi_p, pi_CD = 0 outside (App. B.3 remark)."""
    rng = np.random.default_rng(9)
    V = 400
    zp, zq = _rows(rng, V)
    p = special.softmax(zp)
    prev = None
    for alpha in (0.0, 0.05, 0.1, 0.2, 0.5, 1.0):
        prev = None
        for beta in (0.0, 1e-3, 0.1, 0.5, 1.0):
            r = oracle.row_logpi(zp, zq, alpha=alpha, beta=beta, T=1.0)
            inside = np.isfinite(r["logpi"])
            assert inside.sum() == int(np.sum(p >= beta * p.max()))
            assert inside[np.argmax(zp)]
            assert inside[r["argmax"]]
            assert abs(np.exp(r["logpi"][inside]).sum() - 1.0) < 1e-12
            if prev is not None:
                assert not np.any(inside & ~prev)  # nested: growing beta only removes tokens
            prev = inside
            if beta == 1.0:
                assert r["argmax"] == int(np.argmax(zp))
                assert inside.sum() == 1


# ----------------------------------------------------------------------------- lossless theorem

def _dyadic_distribution(p, zero_last=False, bits=12):
    """A float32 distribution with entries k / 2^bits summing to exactly one."""
    p = np.array(p, dtype=np.float64)
    if zero_last:
        p[-1] = 0.0
    k = np.floor(p / p.sum() * 2 ** bits)
    k[np.argmax(k)] += 2 ** bits - k.sum()
    return (k / 2 ** bits).astype(np.float32)


def _emission_from_chain(zp, zq, alpha, beta, T, q, tokens):
    ratios, rm = oracle.row_chain(zp, zq, alpha, beta, T, q, tokens)
    V = len(zp)
    emit = np.zeros(V)
    reach = 1.0
    for t, rho in zip(tokens, ratios):
        a = min(1.0, rho)
        emit[t] += reach * a
        reach *= 1.0 - a
    emit += reach * rm
    return emit


@pytest.mark.parametrize("m", [1, 2, 3])
@pytest.mark.parametrize("alpha,beta,T", [(0.1, 0.0, 1.0), (0.5, 0.2, 1.0), (1.0, 0.0, 0.6)])
def test_lossless_exact_enumeration(m, alpha, beta, T):
    """App. B.3: with m siblings drawn i.i.d. from q, the first emitted token is distributed as pi_CD.

    Every sibling tuple is enumerated and the acceptance uniforms are integrated analytically
    (accept with probability min(1, ratio)); only the oracle's ratios and residuals are used.
    """
    rng = np.random.default_rng(m * 31 + int(alpha * 10))
    V = 5
    zp, zq = _rows(rng, V, scale=1.0)
    qd = _dyadic_distribution(special.softmax(zp + rng.standard_normal(V)), zero_last=True)
    q64 = qd.astype(np.float64)
    assert q64.sum() == 1.0
    total = np.zeros(V)
    for tup in itertools.product(range(V), repeat=m):
        w = np.prod([q64[t] for t in tup])
        if w == 0.0:
            continue
        total += w * _emission_from_chain(zp, zq, alpha, beta, T, qd, list(tup))
    total /= np.prod([q64.sum()] * m)
    pi = np.exp(oracle.row_logpi(zp, zq, alpha, beta, T)["logpi"])
    np.testing.assert_allclose(total, pi, rtol=0, atol=1e-12)


def _first_emitted(res, tokens):
    B = len(res["accept_len"])
    out = np.where(res["accept_len"] > 0, tokens[np.arange(B), res["accept_path"][:, 1].clip(0)], res["bonus"])
    return out


@pytest.mark.parametrize("beta", [0.0, 0.15])
def test_lossless_monte_carlo_full_verify(beta):
    """Full sampled verification (Philox, ratio test, residuals, exponential race) emits pi_CD."""
    rng = np.random.default_rng(123)
    V, B, m = 6, 120000, 3
    zp, zq = _rows(rng, V, scale=1.0)
    alpha, T = 0.3, 1.0
    qd = special.softmax(zp + 0.8 * rng.standard_normal(V)).astype(np.float32)
    qd = (qd / qd.sum(dtype=np.float64)).astype(np.float32)
    N = 1 + m
    parents = np.tile(np.array([-1, 0, 0, 0], dtype=np.int32), (B, 1))
    tokens = np.zeros((B, N), dtype=np.int32)
    tokens[:, 1:] = rng.choice(V, size=(B, m), p=qd.astype(np.float64) / qd.sum(dtype=np.float64))
    res = oracle.verify(B=B, N=N, V=V, dtype="f64", z_exp=zp, z_ama=zq, ld=0, tokens=tokens,
                        parents=parents, alpha=np.full(B, alpha), beta=np.full(B, beta),
                        temperature=np.full(B, T), q=qd, ldq=0, seed=99, offset=5, nthreads=4)
    first = _first_emitted(res, tokens)
    counts = np.bincount(first, minlength=V)
    pi = np.exp(oracle.row_logpi(zp, zq, alpha, beta, T)["logpi"])
    tv = 0.5 * np.abs(counts / B - pi).sum()
    assert tv < 3.0 * np.sqrt(V / B)
    nz = pi > 0
    assert counts[~nz].sum() == 0  # never emits outside the plausibility set
    chi = stats.chisquare(counts[nz], B * pi[nz])
    assert chi.pvalue > 1e-4


def test_exponential_race_samples_target():
    """A leaf row's bonus is drawn from pi_CD by the race (Algorithm 1, final sample)."""
    rng = np.random.default_rng(77)
    V, B = 8, 100000
    zp, zq = _rows(rng, V, scale=1.0)
    res = oracle.verify(B=B, N=1, V=V, dtype="f64", z_exp=zp, z_ama=zq, ld=0,
                        tokens=np.zeros((B, 1), np.int32), parents=np.full((B, 1), -1, np.int32),
                        alpha=np.full(B, 0.2), temperature=np.full(B, 0.8), q=np.zeros(V, np.float32), ldq=0,
                        seed=1, offset=0, nthreads=4)
    pi = np.exp(oracle.row_logpi(zp, zq, 0.2, 0.0, 0.8)["logpi"])
    counts = np.bincount(res["bonus"], minlength=V)
    assert stats.chisquare(counts, B * pi).pvalue > 1e-4
    assert np.all(res["accept_len"] == 0)


@pytest.mark.parametrize("T", [1.0, 0.7])
def test_two_level_race_samples_target_across_blocks(T):
    """V spans several 1024-token blocks (the last one ragged): the bonus is still drawn from pi_CD."""
    rng = np.random.default_rng(78)
    V, B = 2500, 200000
    zp = 0.6 * rng.standard_normal(V)
    zp[[5, 1100, 2499]] += 2.5  # mass in every block
    zq = 0.7 * zp + 0.5 * rng.standard_normal(V)
    res = oracle.verify(B=B, N=1, V=V, dtype="f64", z_exp=zp, z_ama=zq, ld=0,
                        tokens=np.zeros((B, 1), np.int32), parents=np.full((B, 1), -1, np.int32),
                        alpha=np.full(B, 0.3), temperature=np.full(B, T), q=np.zeros(V, np.float32), ldq=0,
                        seed=4, offset=2, nthreads=4)
    pi = np.exp(oracle.row_logpi(zp, zq, 0.3, 0.0, T)["logpi"])
    counts = np.bincount(res["bonus"], minlength=V)
    # block marginals and the token-level fit
    for lo, hi in ((0, 1024), (1024, 2048), (2048, 2500)):
        p = pi[lo:hi].sum()
        assert abs(counts[lo:hi].sum() / B - p) < 4 * np.sqrt(p * (1 - p) / B)
    assert stats.chisquare(counts, B * pi).pvalue > 1e-4


def test_race_returns_a_point_mass_wherever_it_sits():
    """A row whose whole mass is on one token (first, last or interior of a block, or in the ragged
    last block) always yields that token, whatever the uniforms."""
    V, B = 2100, 300
    for hot in (0, 1023, 1024, 2047, 2048, 2070, 2099):
        zp = np.zeros(V)
        zp[hot] = 200.0  # exp(-200) leaves every other token without representable mass
        res = oracle.verify(B=B, N=1, V=V, dtype="f64", z_exp=zp, z_ama=zp, ld=0,
                            tokens=np.zeros((B, 1), np.int32), parents=np.full((B, 1), -1, np.int32),
                            alpha=np.full(B, 0.2), temperature=np.full(B, 1.0), q=np.zeros(V, np.float32), ldq=0,
                            seed=hot, offset=1)
        assert np.all(res["bonus"] == hot)


# ----------------------------------------------------------------------------- Algorithm 1 on chains

def _algorithm1_chain(zp_rows, zq_rows, q_rows, drafts, alpha, T, seed, offset, b, N):
    """Algorithm 1 (one DCD round) for a chain of gamma drafts, from the pinned row target."""
    gamma = len(drafts)
    V = zp_rows.shape[1]
    pis = [np.exp(oracle.row_logpi(zp_rows[i], zq_rows[i], alpha, 0.0, T)["logpi"]) for i in range(gamma + 1)]
    k = gamma + 1
    for i in range(1, gamma + 1):
        r_i = oracle.accept_uniform(seed, offset, b * N + i)
        # row i-1 holds the logits after draft i-1, i.e. the distribution of draft i
        pi_i, q_i = pis[i - 1], q_rows[i - 1].astype(np.float64)
        ratio = pi_i[drafts[i - 1]] / q_i[drafts[i - 1]] if q_i[drafts[i - 1]] > 0 else np.inf
        if r_i > ratio:
            k = i
            break
    if k <= gamma:
        P = np.maximum(0.0, pis[k - 1] - q_rows[k - 1].astype(np.float64))
        P = P / P.sum()
        row = k - 1
    else:
        P = pis[gamma]
        row = gamma
    return k - 1, _two_level_race(P, seed, offset, b * N + row)


def _two_level_race(P, seed, offset, G, block=1024):
    """Sample from P with the library's two-level exponential race (block, then token)."""
    V = len(P)
    nb = (V + block - 1) // block
    mass = np.array([P[k * block:(k + 1) * block].sum() for k in range(nb)])
    kk = [np.log(mass[k]) - np.log(-np.log(oracle.block_uniform(seed, offset, G, k))) if mass[k] > 0 else -np.inf
          for k in range(nb)]
    kb = int(np.argmax(kk))
    xs = range(kb * block, min(V, (kb + 1) * block))
    keys = [np.log(P[x]) - np.log(-np.log(oracle.race_uniform(seed, offset, G, x))) if P[x] > 0 else -np.inf
            for x in xs]
    return kb * block + int(np.argmax(keys))


def test_chain_reduces_to_algorithm1():
    rng = np.random.default_rng(2024)
    V, gamma, B = 12, 5, 300
    N = gamma + 1
    alpha, T = 0.4, 1.0
    zp = rng.standard_normal((B * N, V))
    zq = 0.7 * zp + 0.8 * rng.standard_normal((B * N, V))
    q = special.softmax(zp + 0.5 * rng.standard_normal((B * N, V)), axis=1).astype(np.float32)
    tokens = np.zeros((B, N), dtype=np.int32)
    for b in range(B):
        for i in range(1, N):
            qq = q[b * N + i - 1].astype(np.float64)
            tokens[b, i] = rng.choice(V, p=qq / qq.sum())
    parents = np.tile(np.arange(-1, N - 1, dtype=np.int32), (B, 1))
    res = oracle.verify(B=B, N=N, V=V, dtype="f64", z_exp=zp, z_ama=zq, tokens=tokens, parents=parents,
                        alpha=np.full(B, alpha), temperature=np.full(B, T), q=q, seed=3, offset=8)
    for b in range(B):
        acc, y = _algorithm1_chain(zp[b * N:(b + 1) * N], zq[b * N:(b + 1) * N], q[b * N:(b + 1) * N],
                                   tokens[b, 1:], alpha, T, 3, 8, b, N)
        assert res["accept_len"][b] == acc
        assert res["bonus"][b] == y
        assert list(res["accept_path"][b, :acc + 1]) == list(range(acc + 1))


# ----------------------------------------------------------------------------- greedy walk

def _spiked_rows(rng, R, V, winners, alpha):
    """Rows whose CD argmax is `winners[g]` by construction: a +30 spike dominates every score."""
    zp = rng.standard_normal((R, V))
    zp[np.arange(R), winners] += 30.0
    zq = 0.7 * zp + 0.5 * rng.standard_normal((R, V))
    return zp, zq


def test_greedy_paths_fixed_by_construction():
    rng = np.random.default_rng(11)
    V, B = 50, 40
    from paper_2608_12913_gb300 import workloads
    for b_trial in range(3):
        parents = np.stack([workloads.tree_parents(np.random.default_rng(100 * b_trial + b)) for b in range(B)])
        N = parents.shape[1]
        winners = rng.integers(0, V, size=B * N)
        zp, zq = _spiked_rows(rng, B * N, V, winners, 0.1)
        tokens = rng.integers(0, V, size=(B, N)).astype(np.int32)
        expect_len, expect_bonus, expect_path = [], [], []
        for b in range(B):
            kids = workloads.children_lists(parents[b])
            cur, path = 0, [0]
            # choose a target path: descend through a random child while there is one
            while kids[cur] and rng.random() < 0.85:
                c = kids[cur][rng.integers(len(kids[cur]))]
                path.append(c)
                cur = c
            # tokens: the path's children carry their parent's winner, every other sibling
            # (and the path's last node's children) carry something else
            for n in range(N):
                for c in kids[n]:
                    w = winners[b * N + n]
                    if n in path[:-1] and c == path[path.index(n) + 1]:
                        tokens[b, c] = w
                    elif tokens[b, c] == w:
                        tokens[b, c] = (w + 1) % V
            expect_len.append(len(path) - 1)
            expect_bonus.append(winners[b * N + cur])
            expect_path.append(path)
        res = oracle.verify(B=B, N=N, V=V, dtype="f64", z_exp=zp, z_ama=zq, tokens=tokens, parents=parents,
                            alpha=np.full(B, 0.1))
        assert list(res["accept_len"]) == expect_len
        assert list(res["bonus"]) == expect_bonus
        for b in range(B):
            p = expect_path[b]
            assert list(res["accept_path"][b, :len(p)]) == p
            assert np.all(res["accept_path"][b, len(p):] == -1)


def test_greedy_duplicate_siblings_take_lowest_node():
    rng = np.random.default_rng(3)
    V = 20
    parents = np.array([[-1, 0, 0, 0, 2, 3]], dtype=np.int32)
    winners = np.array([7, 1, 2, 3, 4, 5])
    zp, zq = _spiked_rows(rng, 6, V, winners, 0.1)
    tokens = np.array([[0, 9, 7, 7, 2, 3]], dtype=np.int32)
    res = oracle.verify(B=1, N=6, V=V, dtype="f64", z_exp=zp, z_ama=zq, tokens=tokens, parents=parents,
                        alpha=np.full(1, 0.1))
    # nodes 2 and 3 both carry the root's winner 7: node 2 is taken; its child 4 carries
    # row 2's winner 2, so the path is 0 -> 2 -> 4 and the bonus is row 4's winner
    assert res["accept_len"][0] == 2
    assert list(res["accept_path"][0]) == [0, 2, 4, -1, -1, -1]
    assert res["bonus"][0] == 4


def test_full_acceptance_chain():
    rng = np.random.default_rng(8)
    V, N = 30, 9
    winners = rng.integers(0, V, size=N)
    zp, zq = _spiked_rows(rng, N, V, winners, 0.2)
    tokens = np.concatenate([[0], winners[:-1]]).astype(np.int32)[None, :]
    res = oracle.verify(B=1, N=N, V=V, dtype="f64", z_exp=zp, z_ama=zq, tokens=tokens,
                        parents=np.arange(-1, N - 1, dtype=np.int32)[None, :], alpha=np.full(1, 0.2))
    assert res["accept_len"][0] == N - 1
    assert res["bonus"][0] == winners[-1]


def test_sampled_rule_tends_to_greedy_as_T_vanishes():
    """T -> 0 with a uniform drafter: the sampled rule accepts exactly the greedy matches."""
    from paper_2608_12913_gb300 import workloads
    w = workloads.make_config(1, V=300, B=4, seed=21, margin_fn=oracle.margin_fn)
    B, N, V = w.B, w.N, w.V
    zp = w.z_exp.float().double().numpy()
    zq = w.z_ama.float().double().numpy()
    g = oracle.verify(B=B, N=N, V=V, dtype="f64", z_exp=zp, z_ama=zq, tokens=w.tokens, parents=w.parents,
                      alpha=w.alpha)
    # make the drafts hit the argmax often: every first child takes its parent's argmax
    tokens = w.tokens.numpy().copy()
    rows = g["rows"]
    for b in range(B):
        kids = workloads.children_lists(w.parents[b].numpy())
        for n in range(N):
            if kids[n]:
                tokens[b, kids[n][-1]] = rows[b, n]["argmax"]
    g = oracle.verify(B=B, N=N, V=V, dtype="f64", z_exp=zp, z_ama=zq, tokens=tokens, parents=w.parents,
                      alpha=w.alpha)
    qu = np.full((B * N, V), 1.0 / V, dtype=np.float32)
    s = oracle.verify(B=B, N=N, V=V, dtype="f64", z_exp=zp, z_ama=zq, tokens=tokens, parents=w.parents,
                      alpha=w.alpha, temperature=np.full(B, 1e-6, np.float32), q=qu, seed=4, offset=1)
    assert np.array_equal(g["accept_len"], s["accept_len"])
    assert np.array_equal(g["accept_path"], s["accept_path"])
    assert np.array_equal(g["bonus"], s["bonus"])
    assert g["accept_len"].max() >= 1


def test_residual_output_matches_chain():
    """The residual a sequence's bonus was drawn from equals the row chain's final residual."""
    from paper_2608_12913_gb300 import workloads
    w = workloads.make_config(2, V=200, B=6, seed=5)
    res = oracle.verify_workload(w, want_residual=True)
    zp = w.z_exp.float().double().numpy()
    zq = w.z_ama.float().double().numpy()
    for b in range(w.B):
        cur = res["accept_path"][b, res["accept_len"][b]]
        kids = workloads.children_lists(w.parents[b].numpy())[cur]
        g = b * w.N + cur
        _, rm = oracle.row_chain(zp[g], zq[g], float(w.alpha[b]), 0.0, float(w.temperature[b]), w.q[g].numpy(),
                                 [int(w.tokens[b, c]) for c in kids])
        np.testing.assert_allclose(res["residual"][b], rm, atol=1e-15)
        assert rm[res["bonus"][b]] > 0


def test_invalid_trees_rejected():
    V = 10
    z = np.zeros((3, V))
    base = dict(B=1, N=3, V=V, dtype="f64", z_exp=z, z_ama=z, alpha=np.zeros(1))
    with pytest.raises(ValueError):
        oracle.verify(tokens=np.zeros((1, 3), np.int32), parents=np.array([[-1, 0, 2]], np.int32), **base)
    with pytest.raises(ValueError):
        oracle.verify(tokens=np.array([[0, 0, V]], np.int32), parents=np.array([[-1, 0, 1]], np.int32), **base)
    with pytest.raises(ValueError):
        oracle.verify(tokens=np.zeros((1, 3), np.int32), parents=np.array([[0, 0, 1]], np.int32), **base)


def test_subset_of_a_batch_draws_the_batch_uniforms():
    """Verifying a subset of sequences (with their batch indices) reproduces the batch's results."""
    from paper_2608_12913_gb300 import workloads
    w = workloads.make_config(3, B=6, V=300, seed=31)
    full = oracle.verify_workload(w)
    sub = oracle.verify_workload(w, seqs=[4, 1])
    for i, b in enumerate([4, 1]):
        assert full["accept_len"][b] == sub["accept_len"][i]
        assert full["bonus"][b] == sub["bonus"][i]
        assert np.array_equal(full["rows"][b]["acc_child"], sub["rows"][i]["acc_child"])
        assert np.array_equal(full["rows"][b]["term_token"], sub["rows"][i]["term_token"])


def test_residual_chain_closed_form():
    """The iterated residual r_j = normalise(max(0, r_{j-1} - q)) of Algorithm 1 equals
    max(0, pi - c_j q) / D_j with c_0 = 0, D_0 = 1, c_{j+1} = c_j + D_j, D_j = sum max(0, pi - c_j q)
    (proof by induction on j); the GPU library evaluates the chain in this form."""
    rng = np.random.default_rng(0)
    for trial in range(8):
        V = 300
        zp = rng.standard_normal(V) * 2
        zq = 0.7 * zp + rng.standard_normal(V)
        q = np.exp(zp + rng.standard_normal(V))
        q = (q / q.sum()).astype(np.float32)
        toks = rng.integers(0, V, size=6)
        alpha, beta = 0.2, (0.0 if trial % 2 else 0.05)
        ratios, rm = oracle.row_chain(zp, zq, alpha, beta, 1.0, q, toks)
        pi = np.exp(oracle.row_logpi(zp, zq, alpha, beta, 1.0)["logpi"])
        qd = q.astype(np.float64)
        c, D = 0.0, 1.0
        closed = []
        for t in toks:
            closed.append(max(0.0, pi[t] - c * qd[t]) / D / qd[t])
            c, D = c + D, None
            D = np.maximum(0.0, pi - c * qd).sum()
        np.testing.assert_allclose(closed, ratios, rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(np.maximum(0.0, pi - c * qd) / D, rm, rtol=0, atol=1e-14)


def test_fused_logits_are_h_times_w_transposed():
    """The fused variant's logits z[r, v] = sum_k h[r, k] w[v, k] (w in the nn.Linear layout
    [V, H]), checked element by element against the sum written out, in blocks of the vocabulary
    smaller than V so that the blocking is exercised."""
    import torch
    g = torch.Generator().manual_seed(5)
    h = torch.randn((3, 11), generator=g).to(torch.bfloat16)
    w = (torch.randn((13, 11), generator=g) * 0.5).to(torch.bfloat16)
    z = oracle.fused_logits(h, w, chunk=4)
    hd, wd = h.double().numpy(), w.double().numpy()
    for r in range(3):
        for v in range(13):
            s = 0.0
            for k in range(11):
                s += hd[r, k] * wd[v, k]
            assert abs(z[r, v] - s) < 1e-12


def _emission_from_chain_distinct(zp, zq, alpha, beta, T, q, tokens):
    ratios, rm = oracle.row_chain(zp, zq, alpha, beta, T, q, tokens, distinct=True)
    V = len(zp)
    emit = np.zeros(V)
    reach = 1.0
    for t, rho in zip(tokens, ratios):
        a = min(1.0, rho)
        emit[t] += reach * a
        reach *= 1.0 - a
    emit += reach * rm
    return emit


def _wor_tuples(q64, m):
    """Every ordered tuple of m distinct draftable tokens with its probability under drawing
    without replacement from q."""
    V = len(q64)
    for tup in itertools.permutations([x for x in range(V) if q64[x] > 0], m):
        w, rest = 1.0, 1.0
        for t in tup:
            w *= q64[t] / rest
            rest -= q64[t]
        yield tup, w


@pytest.mark.parametrize("m", [1, 2, 3])
@pytest.mark.parametrize("alpha,beta,T", [(0.1, 0.0, 1.0), (0.5, 0.2, 1.0), (1.0, 0.0, 0.6)])
def test_lossless_exact_enumeration_siblings_without_replacement(m, alpha, beta, T):
    """Siblings drawn without replacement from q (distinct tokens): with each sibling tested
    against q less the earlier siblings' tokens, renormalised, the first emitted token is
    distributed as pi_CD, to 1e-12, over every ordered tuple of distinct tokens."""
    rng = np.random.default_rng(m * 37 + int(alpha * 10))
    V = 5
    zp, zq = _rows(rng, V, scale=1.0)
    qd = _dyadic_distribution(special.softmax(zp + rng.standard_normal(V)), zero_last=True)
    q64 = qd.astype(np.float64)
    total = np.zeros(V)
    wsum = 0.0
    for tup, w in _wor_tuples(q64, m):
        total += w * _emission_from_chain_distinct(zp, zq, alpha, beta, T, qd, list(tup))
        wsum += w
    assert abs(wsum - 1.0) < 1e-12
    pi = np.exp(oracle.row_logpi(zp, zq, alpha, beta, T)["logpi"])
    np.testing.assert_allclose(total, pi, rtol=0, atol=1e-12)


def test_iid_rule_is_not_lossless_for_distinct_siblings():
    """The plausible mistake of keeping q unchanged for distinct siblings: the i.i.d. rule on
    tuples drawn without replacement does not emit pi_CD (so the pin above separates the two)."""
    rng = np.random.default_rng(7)
    V = 5
    zp, zq = _rows(rng, V, scale=1.0)
    qd = _dyadic_distribution(special.softmax(zp + rng.standard_normal(V)), zero_last=True)
    q64 = qd.astype(np.float64)
    total = np.zeros(V)
    for tup, w in _wor_tuples(q64, 2):
        total += w * _emission_from_chain(zp, zq, 0.3, 0.0, 1.0, qd, list(tup))
    pi = np.exp(oracle.row_logpi(zp, zq, 0.3, 0.0, 1.0)["logpi"])
    assert np.abs(total - pi).max() > 1e-4


def test_distinct_rule_equals_iid_rule_for_one_sibling():
    rng = np.random.default_rng(8)
    V = 40
    zp, zq = _rows(rng, V, scale=2.0)
    q = special.softmax(zp + rng.standard_normal(V)).astype(np.float32)
    r1, m1 = oracle.row_chain(zp, zq, 0.2, 0.0, 1.0, q, [int(np.argmax(q))])
    r2, m2 = oracle.row_chain(zp, zq, 0.2, 0.0, 1.0, q, [int(np.argmax(q))], distinct=True)
    np.testing.assert_array_equal(r1, r2)
    np.testing.assert_array_equal(m1, m2)


def test_lossless_monte_carlo_full_verify_siblings_without_replacement():
    """Full sampled verification with the distinct-sibling rule (Philox, ratio test, residuals,
    race) on siblings drawn without replacement from q emits pi_CD."""
    rng = np.random.default_rng(321)
    V, B, m = 6, 120000, 3
    zp, zq = _rows(rng, V, scale=1.0)
    alpha, T = 0.3, 1.0
    qd = special.softmax(zp + 0.8 * rng.standard_normal(V)).astype(np.float32)
    qd = (qd / qd.sum(dtype=np.float64)).astype(np.float32)
    p64 = qd.astype(np.float64) / qd.sum(dtype=np.float64)
    N = 1 + m
    parents = np.tile(np.array([-1, 0, 0, 0], dtype=np.int32), (B, 1))
    tokens = np.zeros((B, N), dtype=np.int32)
    # m distinct tokens per sequence, in draw order: Gumbel top-m is sampling without replacement
    gk = np.log(p64)[None, :] - np.log(-np.log(rng.random((B, V))))
    tokens[:, 1:] = np.argsort(-gk, axis=1)[:, :m]
    res = oracle.verify(B=B, N=N, V=V, dtype="f64", z_exp=zp, z_ama=zq, ld=0, tokens=tokens,
                        parents=parents, alpha=np.full(B, alpha), beta=np.zeros(B),
                        temperature=np.full(B, T), q=qd, ldq=0, seed=77, offset=3, nthreads=4, distinct=True)
    first = _first_emitted(res, tokens)
    counts = np.bincount(first, minlength=V)
    pi = np.exp(oracle.row_logpi(zp, zq, alpha, 0.0, T)["logpi"])
    tv = 0.5 * np.abs(counts / B - pi).sum()
    assert tv < 3.0 * np.sqrt(V / B)
    chi = stats.chisquare(counts[pi > 0], B * pi[pi > 0])
    assert chi.pvalue > 1e-4


def test_row_diagnostics_closed_forms():
    """The diagnostics against closed forms: lse against scipy's logsumexp; E_{pi_q}[log pi_p -
    log pi_q] = -KL(pi_q || pi_p) and D_KL(pi_e || pi_p) from scipy's relative entropy; the signal
    from the log-softmax difference at x*; E_{pi_e} with pi_e = pi_q equals E_{pi_q}; the KL of
    pi_p from itself is zero."""
    rng = np.random.default_rng(41)
    V = 97
    zp, zq = _rows(rng, V, scale=2.0)
    lp, lq = special.log_softmax(zp), special.log_softmax(zq)
    pe = special.softmax(zp + rng.standard_normal(V))
    x = int(np.argmax(zp))
    d = oracle.row_diagnostics(zp, zq, x, q=pe.astype(np.float32))
    assert abs(d["lse_p"] - special.logsumexp(zp)) < 1e-12
    assert abs(d["lse_q"] - special.logsumexp(zq)) < 1e-12
    assert abs(d["signal"] - abs(lp[x] - lq[x])) < 1e-12
    assert abs(d["e_q"] + special.rel_entr(np.exp(lq), np.exp(lp)).sum()) < 1e-12
    pe32 = pe.astype(np.float32).astype(np.float64)
    assert abs(d["kl_e_p"] - special.rel_entr(pe32, np.exp(lp)).sum()) < 1e-9
    assert abs(d["e_e"] - (pe32 * (lp - lq)).sum()) < 1e-12
    same = oracle.row_diagnostics(zp, zq, x, q=np.exp(lq).astype(np.float32))
    assert abs(same["e_e"] - d["e_q"]) < 1e-6  # pi_e = pi_q (up to fp32 rounding of q)
    self_kl = oracle.row_diagnostics(zp, zq, x, q=np.exp(lp).astype(np.float32))["kl_e_p"]
    assert abs(self_kl) < 1e-6
    assert np.isnan(oracle.row_diagnostics(zp, zq, x)["e_e"])
    assert np.isnan(oracle.row_diagnostics(zp, zq, x)["kl_p_cd"])


@pytest.mark.parametrize("alpha", [0.0, 0.1, 0.5, 1.5])
def test_row_diagnostics_kl_columns(alpha):
    """D_KL(pi_p || pi_q) against scipy's relative entropy; D_KL(pi_p || pi_CD), which the oracle
    sums term by term from Eq. 1's definition, against scipy's relative entropy of pi_CD =
    softmax((1 + alpha) log pi_p - alpha log pi_q) and against the decomposition lemma of App. B,
    D_KL(pi_p || pi_CD) = log Z_CD - alpha D_KL(pi_p || pi_q) with Z_CD = sum pi_p^(1+alpha)
    pi_q^(-alpha); at alpha = 0 the target is pi_p and the divergence vanishes."""
    rng = np.random.default_rng(int(alpha * 100) + 5)
    V = 211
    zp, zq = _rows(rng, V, scale=2.0)
    lp, lq = special.log_softmax(zp), special.log_softmax(zq)
    d = oracle.row_diagnostics(zp, zq, 0, alpha=alpha)
    pp, pq = np.exp(lp), np.exp(lq)
    assert abs(d["kl_p_q"] - special.rel_entr(pp, pq).sum()) < 1e-12
    pcd = special.softmax((1 + alpha) * lp - alpha * lq)
    assert abs(d["kl_p_cd"] - special.rel_entr(pp, pcd).sum()) < 1e-12
    log_z = special.logsumexp((1 + alpha) * lp - alpha * lq)
    assert abs(d["kl_p_cd"] - (log_z - alpha * d["kl_p_q"])) < 1e-12
    if alpha == 0.0:
        assert abs(d["kl_p_cd"]) < 1e-14
    assert d["kl_p_cd"] >= -1e-15 and d["kl_p_q"] >= -1e-15
