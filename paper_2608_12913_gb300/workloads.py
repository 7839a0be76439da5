"""Seeded synthetic inputs for the contrastive-decoding (CD) verification step.

This module only draws random numbers and lays them out; it holds none of the
method's arithmetic (no log-softmax, no CD score, no acceptance rule). It
serves both the CUDA path and the CPU oracle, which never import each other.

Recipe (the paper's datasets and checkpoints are not available; these shapes
stand in for them):

* vocabulary V = 128256 (the Llama-3 tokenizer of the paper's main model pair,
  Table model_details) or V = 32000 for the tiny chain case;
* expert logits  z_p = N(0, 2^2) with +10 "spikes" on k distinct random tokens
  of each row (k fixed or uniform in a range);
* amateur logits z_q = 0.7 * z_p + N(0, 1.5^2), from the pre-rounding z_p;
* logits are drawn in fp64 and rounded to bf16 (round-to-nearest-even) or to
  fp32;
* draft trees: level sizes (1, 8, 16, 16, 10, 5, 3, 1) give 60 nodes of depth
  7; each depth-d node picks its parent uniformly among the depth-(d-1) nodes
  that still have fewer than 8 children; node ids are in BFS order, so
  parents[i] < i; a chain is parents = (-1, 0, 1, ...);
* a parent's children carry the top-m tokens of (z_p[parent] + N(0, 1)) in
  descending order (an EAGLE-style top-k expansion of a noisy expert);
* sampled sequences get the draft distribution q[parent] = softmax(z_p[parent]
  + the same N(0, 1) noise) in fp32, the distribution their drafts came from.

Two generators follow the recipe: ``backend="numpy"`` (PCG64, one
``SeedSequence([seed, stream, row, attempt])`` per row, identical on every
platform; used for parity cases and stored expected values) and
``backend="torch"`` (a seeded torch generator on the target device, for the
full-size benchmark workloads, where drawing 0.5 G normals on the host would
dominate the run).

A margin callback (supplied by the tests, which compute it with the oracle)
lets the numpy generator redraw any row whose top-2 CD-score gap, or whose
distance to the plausibility threshold, is below a bound: decisions taken in
fp32 on the GPU and in fp64 on the CPU then agree.
"""

from __future__ import annotations

import dataclasses
from typing import Callable, Optional, Sequence

import numpy as np
import torch

TREE_LEVELS_60 = (1, 8, 16, 16, 10, 5, 3, 1)
MAX_CHILDREN = 8

# Stream ids of the per-row seed sequences.
_S_TREE, _S_LOGITS, _S_DRAFT, _S_HIDDEN, _S_WEIGHT = 0, 1, 2, 3, 4


@dataclasses.dataclass
class Workload:
    """One verification call's inputs.

    Rows are numbered g = b * N + n; row g holds the next-token logits after
    node n of sequence b (the distribution its children were drafted from).
    """

    name: str
    B: int
    N: int
    V: int
    dtype: str  # "f32" or "bf16" for the logits
    z_exp: torch.Tensor  # [B*N, V]
    z_ama: torch.Tensor  # [B*N, V]
    tokens: torch.Tensor  # int32 [B, N]; tokens[:, 0] is the root (not verified)
    parents: torch.Tensor  # int32 [B, N]; parents[:, 0] = -1, parents[i] < i
    alpha: torch.Tensor  # float32 [B]
    beta: torch.Tensor  # float32 [B]
    temperature: torch.Tensor  # float32 [B]; 0 selects the greedy rule
    q: Optional[torch.Tensor]  # float32 [B*N, V] or None when every sequence is greedy
    seed: int = 0
    offset: int = 0
    # fused LM-head variant only
    h_exp: Optional[torch.Tensor] = None  # bf16 [B*N, H_exp]
    w_exp: Optional[torch.Tensor] = None  # bf16 [V, H_exp]
    h_ama: Optional[torch.Tensor] = None  # bf16 [B*N, H_ama]
    w_ama: Optional[torch.Tensor] = None  # bf16 [V, H_ama]

    @property
    def R(self) -> int:
        return self.B * self.N

    def sampled_rows_with_children(self) -> int:
        """Rows whose q the sampled rule reads: non-leaf rows of T > 0 sequences."""
        par = self.parents.cpu().numpy()
        temp = self.temperature.cpu().numpy()
        count = 0
        for b in range(self.B):
            if temp[b] > 0:
                count += len(set(int(p) for p in par[b, 1:] if p >= 0))
        return count

    def to(self, device) -> "Workload":
        out = dataclasses.replace(self)
        for f in dataclasses.fields(self):
            v = getattr(self, f.name)
            if isinstance(v, torch.Tensor):
                setattr(out, f.name, v.to(device))
        return out


def _rng(seed: int, stream: int, row: int, attempt: int = 0) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, stream, row, attempt])))


def tree_parents(rng: np.random.Generator, levels: Sequence[int] = TREE_LEVELS_60,
                 max_children: int = MAX_CHILDREN) -> np.ndarray:
    """Parent array of a random top-k style draft tree, in BFS order."""
    assert levels[0] == 1
    parents = [-1]
    depth_nodes = [[0]]
    n_children = {0: 0}
    for d in range(1, len(levels)):
        prev = depth_nodes[-1]
        picks = []
        for _ in range(levels[d]):
            free = [p for p in prev if n_children[p] < max_children]
            if not free:
                raise ValueError("tree level sizes exceed the child budget")
            p = free[int(rng.integers(len(free)))]
            n_children[p] += 1
            picks.append(p)
        picks.sort()  # BFS: children of earlier parents first
        ids = []
        for p in picks:
            nid = len(parents)
            parents.append(p)
            n_children[nid] = 0
            ids.append(nid)
        depth_nodes.append(ids)
    return np.asarray(parents, dtype=np.int32)


def chain_parents(n: int) -> np.ndarray:
    return np.arange(-1, n - 1, dtype=np.int32)


def children_lists(parents: np.ndarray) -> list:
    ch = [[] for _ in range(len(parents))]
    for i, p in enumerate(parents):
        if i > 0:
            ch[int(p)].append(i)
    return ch


def _to_dtype(x: np.ndarray, dtype: str) -> torch.Tensor:
    t = torch.from_numpy(np.ascontiguousarray(x))
    return t.to(torch.bfloat16) if dtype == "bf16" else t.to(torch.float32)


def _row_logits(seed, g, attempt, V, spikes):
    rng = _rng(seed, _S_LOGITS, g, attempt)
    zp = 2.0 * rng.standard_normal(V)
    k = int(spikes[0]) if spikes[0] == spikes[1] else int(rng.integers(spikes[0], spikes[1] + 1))
    k = min(k, V)
    idx = rng.choice(V, size=k, replace=False)
    zp[idx] += 10.0
    za = 0.7 * zp + 1.5 * rng.standard_normal(V)
    return zp, za


def _topm(v: np.ndarray, m: int) -> np.ndarray:
    """Indices of the m largest entries, descending, ties to the lower index."""
    if m <= 0:
        return np.zeros(0, dtype=np.int64)
    m = min(m, v.shape[0])
    part = np.argpartition(-v, m - 1)[:m] if m < v.shape[0] else np.arange(v.shape[0])
    order = np.lexsort((part, -v[part]))
    return part[order]


def generate(*, name: str, B: int, V: int, dtype: str, spikes=(1, 6),
             alphas: Sequence[float] = (0.1,), beta: float = 0.0,
             temperatures: Sequence[float] = (0.0,), levels: Optional[Sequence[int]] = None,
             chain_len: Optional[int] = None, seed: int = 0, offset: int = 0,
             margin_fn: Optional[Callable] = None, margin: float = 1e-3,
             max_attempts: int = 100, max_children: int = MAX_CHILDREN) -> Workload:
    """Numpy generator (CPU tensors). Per-sequence alpha/T cycle through the given lists.

    ``margin_fn(zp_row, za_row, alpha, beta) -> float`` receives the rounded logits
    (as float64 arrays) and returns the row's decision margin; rows below ``margin``
    are redrawn with the next attempt number (at most ``max_attempts`` times).
    """
    if chain_len is not None:
        tree = [chain_parents(chain_len) for _ in range(B)]
    else:
        lv = tuple(levels) if levels is not None else TREE_LEVELS_60
        tree = [tree_parents(_rng(seed, _S_TREE, b), lv, max_children) for b in range(B)]
    N = len(tree[0])
    assert all(len(t) == N for t in tree)
    R = B * N
    alpha = np.array([alphas[b % len(alphas)] for b in range(B)], dtype=np.float32)
    temp = np.array([temperatures[b % len(temperatures)] for b in range(B)], dtype=np.float32)
    beta_a = np.full(B, beta, dtype=np.float32)
    sampled_any = bool((temp > 0).any())

    np_dtype = np.float32
    zp_all = np.empty((R, V), dtype=np.float64)
    za_all = np.empty((R, V), dtype=np.float64)
    zp_out = torch.empty((R, V), dtype=torch.bfloat16 if dtype == "bf16" else torch.float32)
    za_out = torch.empty_like(zp_out)
    for g in range(R):
        b = g // N
        attempt = 0
        while True:
            zp, za = _row_logits(seed, g, attempt, V, spikes)
            tp, ta = _to_dtype(zp, dtype), _to_dtype(za, dtype)
            if margin_fn is None or attempt >= max_attempts:
                break
            if margin_fn(tp.double().numpy(), ta.double().numpy(), float(alpha[b]), float(beta_a[b])) >= margin:
                break
            attempt += 1
        zp_all[g], za_all[g] = zp, za
        zp_out[g], za_out[g] = tp, ta

    tokens = np.zeros((B, N), dtype=np.int32)
    q = np.zeros((R, V), dtype=np_dtype) if sampled_any else None
    for b in range(B):
        ch = children_lists(tree[b])
        for n in range(N):
            if not ch[n]:
                continue
            g = b * N + n
            eps = _rng(seed, _S_DRAFT, g).standard_normal(V)
            noisy = zp_all[g] + eps
            top = _topm(noisy, len(ch[n]))
            for c, t in zip(ch[n], top):
                tokens[b, c] = int(t)
            if temp[b] > 0:
                e = np.exp(noisy - noisy.max())
                q[g] = (e / e.sum()).astype(np_dtype)
    return Workload(
        name=name, B=B, N=N, V=V, dtype=dtype, z_exp=zp_out, z_ama=za_out,
        tokens=torch.from_numpy(tokens), parents=torch.from_numpy(np.stack(tree).astype(np.int32)),
        alpha=torch.from_numpy(alpha), beta=torch.from_numpy(beta_a), temperature=torch.from_numpy(temp),
        q=None if q is None else torch.from_numpy(q), seed=seed, offset=offset)


# The five workloads of the verification benchmark (sizes stated in the module docstring).
CONFIGS = {
    0: dict(name="tiny_chain_B1_N6_V32000_f32_greedy", B=1, V=32000, dtype="f32", spikes=(3, 3),
            alphas=(0.1,), temperatures=(0.0,), chain_len=6, seed=0),
    1: dict(name="tree60_B1_V128256_bf16_greedy", B=1, V=128256, dtype="bf16", spikes=(1, 6),
            alphas=(0.1,), temperatures=(0.0,), seed=1),
    2: dict(name="tree60_B1_V128256_bf16_sampled_T1", B=1, V=128256, dtype="bf16", spikes=(1, 6),
            alphas=(0.1,), temperatures=(1.0,), seed=2),
    # sequence s: alpha = (0.05, 0.1, 0.2)[s % 3]; even s greedy, odd s sampled at T = 1
    3: dict(name="batched_B32_tree60_V128256_bf16_mixed", B=32, V=128256, dtype="bf16", spikes=(1, 6),
            alphas=(0.05, 0.1, 0.2), temperatures=(0.0, 1.0), seed=3),
}

FUSED_CONFIG = dict(name="fused_lmhead_B64_tree60_V128256_Hexp8192_Hama2048_bf16_greedy",
                    B=64, V=128256, H_exp=8192, H_ama=2048, alpha=0.1, seed=4, w_std=0.02)


def make_config(cfg: int, **overrides) -> Workload:
    """Numpy-backend workload for config ``cfg`` (any field may be overridden, e.g. V or B)."""
    spec = dict(CONFIGS[cfg])
    spec.update(overrides)
    return generate(**spec)


def generate_torch(*, name: str, B: int, V: int, dtype: str, spikes=(1, 6),
                   alphas: Sequence[float] = (0.1,), beta: float = 0.0,
                   temperatures: Sequence[float] = (0.0,), levels: Optional[Sequence[int]] = None,
                   chain_len: Optional[int] = None, seed: int = 0, offset: int = 0,
                   device="cuda", row_block: int = 256) -> Workload:
    """Same recipe drawn with a seeded torch generator on ``device`` (fast, full size).

    Tree shapes still come from the numpy PCG64 streams, so they match ``generate``;
    the logits and draft noise are a different (but equally seeded) random stream.
    """
    dev = torch.device(device)
    if chain_len is not None:
        tree = [chain_parents(chain_len) for _ in range(B)]
    else:
        lv = tuple(levels) if levels is not None else TREE_LEVELS_60
        tree = [tree_parents(_rng(seed, _S_TREE, b), lv) for b in range(B)]
    N = len(tree[0])
    R = B * N
    alpha = torch.tensor([alphas[b % len(alphas)] for b in range(B)], dtype=torch.float32)
    temp = torch.tensor([temperatures[b % len(temperatures)] for b in range(B)], dtype=torch.float32)
    beta_a = torch.full((B,), float(beta), dtype=torch.float32)
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    gen = torch.Generator(device=dev)
    gen.manual_seed(1_000_003 * seed + 17)
    z_exp = torch.empty((R, V), dtype=tdt, device=dev)
    z_ama = torch.empty((R, V), dtype=tdt, device=dev)
    parents = np.stack(tree).astype(np.int32)
    kids = [children_lists(t) for t in tree]
    sampled = (temp > 0).numpy()
    q = torch.zeros((R, V), dtype=torch.float32, device=dev) if sampled.any() else None
    tokens = np.zeros((B, N), dtype=np.int32)
    kmax = max(1, min(int(spikes[1]), V))
    for r0 in range(0, R, row_block):
        r1 = min(R, r0 + row_block)
        n = r1 - r0
        zp = torch.randn((n, V), generator=gen, device=dev, dtype=torch.float32) * 2.0
        k = torch.randint(int(spikes[0]), int(spikes[1]) + 1, (n, 1), generator=gen, device=dev)
        pick = torch.rand((n, V), generator=gen, device=dev).topk(kmax, dim=1).indices
        keep = (torch.arange(kmax, device=dev)[None, :] < k).to(torch.float32)
        zp.scatter_add_(1, pick, 10.0 * keep)
        za = 0.7 * zp + 1.5 * torch.randn((n, V), generator=gen, device=dev, dtype=torch.float32)
        z_exp[r0:r1] = zp.to(tdt)
        z_ama[r0:r1] = za.to(tdt)
        eps = torch.randn((n, V), generator=gen, device=dev, dtype=torch.float32)
        noisy = zp + eps
        top = noisy.topk(MAX_CHILDREN, dim=1).indices.cpu().numpy()
        for i in range(n):
            g = r0 + i
            b, node = divmod(g, N)
            ch = kids[b][node]
            for c, t in zip(ch, top[i]):
                tokens[b, c] = int(t)
        if q is not None:
            rows = [i for i in range(n) if sampled[(r0 + i) // N] and kids[(r0 + i) // N][(r0 + i) % N]]
            if rows:
                idx = torch.tensor(rows, device=dev)
                q[r0 + idx] = torch.softmax(noisy[idx].double(), dim=1).float()
        del zp, za, eps, noisy, pick
    return Workload(
        name=name, B=B, N=N, V=V, dtype=dtype, z_exp=z_exp, z_ama=z_ama,
        tokens=torch.from_numpy(tokens).to(dev), parents=torch.from_numpy(parents).to(dev),
        alpha=alpha.to(dev), beta=beta_a.to(dev), temperature=temp.to(dev), q=q,
        seed=seed, offset=offset)


def make_config_torch(cfg: int, device="cuda", **overrides) -> Workload:
    spec = dict(CONFIGS[cfg])
    spec.update(overrides)
    return generate_torch(device=device, **spec)


def make_fused_torch(device="cuda", B: Optional[int] = None, V: Optional[int] = None,
                     H_exp: Optional[int] = None, H_ama: Optional[int] = None,
                     seed: Optional[int] = None, levels: Optional[Sequence[int]] = None,
                     beta: float = 0.0, w_std: Optional[float] = None) -> Workload:
    """Fused LM-head workload: hidden states ~ N(0,1), weights ~ N(0, w_std^2) (0.02 unless
    given), all bf16.

    Weights use the nn.Linear layout [V, H] (row v holds the output-embedding of token v).
    Draft tokens are the top-m of (z_p[parent] + N(0,1)) with z_p = h_exp @ w_exp^T taken
    from a bf16 torch matmul (input generation only).
    """
    c = dict(FUSED_CONFIG)
    B = B or c["B"]
    V = V or c["V"]
    H_exp = H_exp or c["H_exp"]
    H_ama = H_ama or c["H_ama"]
    seed = c["seed"] if seed is None else seed
    dev = torch.device(device)
    lv = tuple(levels) if levels is not None else TREE_LEVELS_60
    tree = [tree_parents(_rng(seed, _S_TREE, b), lv) for b in range(B)]
    N = len(tree[0])
    R = B * N
    gen = torch.Generator(device=dev)
    gen.manual_seed(1_000_003 * seed + 29)
    h_exp = torch.randn((R, H_exp), generator=gen, device=dev).to(torch.bfloat16)
    h_ama = torch.randn((R, H_ama), generator=gen, device=dev).to(torch.bfloat16)
    ws = c["w_std"] if w_std is None else w_std
    w_exp = (torch.randn((V, H_exp), generator=gen, device=dev) * ws).to(torch.bfloat16)
    w_ama = (torch.randn((V, H_ama), generator=gen, device=dev) * ws).to(torch.bfloat16)
    tokens = np.zeros((B, N), dtype=np.int32)
    kids = [children_lists(t) for t in tree]
    blk = 512
    for r0 in range(0, R, blk):
        r1 = min(R, r0 + blk)
        zp = (h_exp[r0:r1] @ w_exp.t()).float()
        noisy = zp + torch.randn(zp.shape, generator=gen, device=dev)
        top = noisy.topk(MAX_CHILDREN, dim=1).indices.cpu().numpy()
        for i in range(r1 - r0):
            b, node = divmod(r0 + i, N)
            for cid, t in zip(kids[b][node], top[i]):
                tokens[b, cid] = int(t)
        del zp, noisy
    return Workload(
        name=c["name"], B=B, N=N, V=V, dtype="bf16", z_exp=torch.empty(0), z_ama=torch.empty(0),
        tokens=torch.from_numpy(tokens).to(dev), parents=torch.from_numpy(np.stack(tree)).to(dev),
        alpha=torch.full((B,), c["alpha"], dtype=torch.float32, device=dev),
        beta=torch.full((B,), beta, dtype=torch.float32, device=dev),
        temperature=torch.zeros(B, dtype=torch.float32, device=dev), q=None, seed=seed,
        h_exp=h_exp, w_exp=w_exp, h_ama=h_ama, w_ama=w_ama)
