"""Seeded synthetic planner instances.

This module only synthesises inputs (trees, chunk weights, demand, cost
tables, start orders).  It holds none of the planner's arithmetic: no
objective, marginal, DP or refinement step lives here.  The CUDA path and the
CPU oracle both read its arrays, so generator floating point can never affect
parity: every array it returns is integer.

Cost model (Section II-B):
  * a chunk of w slots holds w * 512 tokens, KV footprint
    w * 512 * 36,864 B = w * 18,874,368 B (the 3B FP16 profile of Table I;
    "18.9 MB" per 512-token chunk in Fig. 1);
  * fetch cost f = Z / r (Eq. 1) in integer microseconds,
    t = (Z * 8 * 10^6 + g // 2) // g for an integer goodput g in bit/s;
  * recomputation w_r(v) = weight(v) * (beta_r + alpha_r * p(v)), p(v) the
    existing-prefix length in tokens, linear as in the RQ1 fits
    (170.2 + 0.0100p ms on L4-7B, 48.1 + 0.0050p ms on A100-7B).  Three
    hardware classes with alpha ratio 1:3:8.
  * demand: requests land on leaves (Zipf-ranked popularity, Poisson counts);
    a request contributes to every chunk on its prefix path (Section III-A).
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

CHUNK_TOKENS = 512
KV_BYTES_PER_TOKEN = 36_864                   # Table I, 3B FP16 profiles
CHUNK_BYTES = CHUNK_TOKENS * KV_BYTES_PER_TOKEN   # 18,874,368 B per unit-weight chunk
GOODPUT_BPS = 1.5e9                            # common effective KV goodput of Fig. 1
ALPHA_US_PER_TOKEN = (4, 12, 32)               # recompute slope per class, ratio 1:3:8
BETA_US = (40_000, 55_000, 110_000)            # recompute intercept per class
REQUESTS_PER_EPOCH = 30_000                    # epoch size of the replay study


def fetch_us(nbytes, goodput_bps):
    """Eq. 1 in integer microseconds: round(Z * 8 / r * 1e6), integer division."""
    nbytes = np.asarray(nbytes, dtype=np.int64)
    g = np.asarray(goodput_bps, dtype=np.int64)
    return (nbytes * 8 * 1_000_000 + g // 2) // g


@dataclass
class Instance:
    name: str
    n: int
    W: int
    parent: np.ndarray          # [n] int32, -1 = top level
    weight: np.ndarray          # [n] int32 slots
    demand: np.ndarray          # [W][n] int64
    recompute: np.ndarray       # [W][n] int64 us
    transfer: np.ndarray        # mode 0: [W][n]; mode 1: [W][W][n] int64 us, [src][req][v]
    mode: int                   # 0 requester-side, 1 source-dependent
    budget: np.ndarray          # [W] int32
    starts: int
    rounds: int
    seed: int = 0
    profile: dict = field(default_factory=dict)


# ----------------------------------------------------------------------------
# trees
# ----------------------------------------------------------------------------

def _grow_random(rng, n, n_roots, max_depth, quota):
    """Grow a forest by attaching each new node under a uniformly random open node.

    A node is open while its depth is below max_depth and it has fewer children
    than its quota (drawn by `quota(rng)` when the node is created)."""
    parent = np.full(n, -1, np.int32)
    depth = np.zeros(n, np.int32)
    nchild = np.zeros(n, np.int32)
    q = np.zeros(n, np.int32)
    open_ = []
    cnt = 0
    for _ in range(min(n_roots, n)):
        depth[cnt] = 1
        q[cnt] = quota(rng)
        if max_depth > 1:
            open_.append(cnt)
        cnt += 1
    while cnt < n:
        if not open_:
            depth[cnt] = 1
            q[cnt] = quota(rng)
            if max_depth > 1:
                open_.append(cnt)
            cnt += 1
            continue
        k = int(rng.integers(len(open_)))
        u = open_[k]
        v = cnt
        cnt += 1
        parent[v] = u
        depth[v] = depth[u] + 1
        q[v] = quota(rng)
        nchild[u] += 1
        if nchild[u] >= q[u]:
            open_[k] = open_[-1]
            open_.pop()
        if depth[v] < max_depth:
            open_.append(v)
    return parent


def _add_chain(parent_list, under, length):
    ids = []
    p = under
    for _ in range(length):
        v = len(parent_list)
        parent_list.append(p)
        ids.append(v)
        p = v
    return ids


def _zipf_weights(m, s):
    r = np.arange(1, m + 1, dtype=np.float64)
    w = r ** (-float(s))
    return w / w.sum()


def _rag_tree(rng, n, n_sys=16, n_docs=2000, doc_frac=0.6, doc_zipf=1.0):
    """System-prompt chains, Zipf-drawn document chains under them, query chains."""
    parent = []
    sys_end = []
    for _ in range(n_sys):
        ids = _add_chain(parent, -1, int(rng.integers(2, 5)))          # depth 2..4
        sys_end.append(ids[-1])
    doc_len = rng.integers(4, 17, size=n_docs)                         # depth 4..16
    doc_p = _zipf_weights(n_docs, doc_zipf)
    doc_rank = rng.permutation(n_docs)
    seen = set()
    doc_ends, doc_pop = [], []
    target = int(doc_frac * n)
    while len(parent) < target:
        r = int(rng.integers(n_sys))
        d = int(doc_rank[rng.choice(n_docs, p=doc_p)])
        if (r, d) in seen:
            continue
        seen.add((r, d))
        ln = min(int(doc_len[d]), n - len(parent))
        ids = _add_chain(parent, sys_end[r], ln)
        doc_ends.append(ids[-1])
        doc_pop.append(doc_p[np.where(doc_rank == d)[0][0]])
    doc_pop = np.asarray(doc_pop, np.float64)
    doc_pop /= doc_pop.sum()
    while len(parent) < n:
        e = doc_ends[int(rng.choice(len(doc_ends), p=doc_pop))]
        ln = min(int(rng.integers(1, 4)), n - len(parent))             # query chain 1..3
        _add_chain(parent, e, ln)
    return np.asarray(parent, np.int32)


def _mixed_tree(rng, n, prefix_frac=0.3, prefix_depth=8, chain_depth=64, n_roots=32):
    """Bushy shared system / few-shot prefixes, then conversation chains under them."""
    n_pre = int(prefix_frac * n)
    pre = _grow_random(rng, n_pre, n_roots, prefix_depth, lambda r: int(r.geometric(0.35)) + 1)
    parent = list(pre.tolist())
    while len(parent) < n:
        u = int(rng.integers(n_pre))
        ln = min(int(rng.integers(2, chain_depth + 1)), n - len(parent))
        _add_chain(parent, u, ln)
    return np.asarray(parent, np.int32)


def _stress_tree(rng, n, n_docs=20_000, deep=256):
    """Deep chains (to depth 256) mixed with bushy Zipf document fan-out."""
    parent = []
    roots = []
    for _ in range(64):                                              # shared roots, depth 1..3
        ids = _add_chain(parent, -1, int(rng.integers(1, 4)))
        roots.append(ids[-1])
    doc_p = _zipf_weights(n_docs, 1.0)
    doc_len = rng.integers(2, 9, size=n_docs)
    doc_end = {}
    while len(parent) < n:
        if rng.random() < 0.25:                                       # deep conversation chain
            u = roots[int(rng.integers(len(roots)))]
            ln = min(int(rng.integers(deep // 4, deep + 1)), n - len(parent))
            _add_chain(parent, u, ln)
        else:                                                         # document fan-out
            d = int(rng.choice(n_docs, p=doc_p))
            if d not in doc_end:
                u = roots[d % len(roots)]
                ln = min(int(doc_len[d]), n - len(parent))
                doc_end[d] = _add_chain(parent, u, ln)[-1]
            else:
                ln = min(int(rng.integers(1, 4)), n - len(parent))
                _add_chain(parent, doc_end[d], ln)
    return np.asarray(parent, np.int32)


# ----------------------------------------------------------------------------
# demand and costs
# ----------------------------------------------------------------------------

def _depth_order(parent):
    """Node ids grouped by depth (parents strictly before children)."""
    n = parent.shape[0]
    depth = np.zeros(n, np.int64)
    # parents precede children in every generator above, so one pass suffices
    for v in range(n):
        p = parent[v]
        depth[v] = 1 if p < 0 else depth[p] + 1
    return depth


def _prefix_tokens(parent, weight, depth):
    """Existing-prefix length in tokens: 512 * sum of strict ancestors' weights."""
    n = parent.shape[0]
    anc_w = np.zeros(n, np.int64)
    order = np.argsort(depth, kind="stable")
    for v in order:
        p = parent[v]
        if p >= 0:
            anc_w[v] = anc_w[p] + weight[p]
    return anc_w * CHUNK_TOKENS


def _leaf_demand(rng, parent, W, zipf_s, per_worker_perm):
    n = parent.shape[0]
    is_leaf = np.ones(n, bool)
    is_leaf[parent[parent >= 0]] = False
    leaves = np.nonzero(is_leaf)[0]
    L = leaves.shape[0]
    zw = _zipf_weights(L, zipf_s)
    per_worker = REQUESTS_PER_EPOCH / W
    counts = np.zeros((W, n), np.int64)
    shared_rank = rng.permutation(L)
    for m in range(W):
        rank = rng.permutation(L) if per_worker_perm else shared_rank
        lam = per_worker * zw[rank]
        counts[m, leaves] = rng.poisson(lam)
    return counts


def _propagate_up(parent, counts, depth):
    """Every chunk on a request's prefix path carries that request's demand."""
    dem = counts.copy()
    maxd = int(depth.max()) if depth.size else 0
    for d in range(maxd, 1, -1):
        nodes = np.nonzero(depth == d)[0]
        np.add.at(dem, (slice(None), parent[nodes]), dem[:, nodes])
    return dem


def _recompute(weight, ptok, classes):
    W = len(classes)
    out = np.zeros((W, weight.shape[0]), np.int64)
    for m, c in enumerate(classes):
        out[m] = weight.astype(np.int64) * (BETA_US[c] + ALPHA_US_PER_TOKEN[c] * ptok)
    return out


def _transfer_requester(rng, weight, W, sigma):
    g = np.rint(rng.lognormal(np.log(GOODPUT_BPS), sigma, size=W)).astype(np.int64)
    nbytes = weight.astype(np.int64) * CHUNK_BYTES
    return np.stack([fetch_us(nbytes, g[m]) for m in range(W)]).astype(np.int64)


def _transfer_source(rng, weight, W, sigma, near=4, near_factor=4.0):
    g = rng.lognormal(np.log(GOODPUT_BPS), sigma, size=(W, W))
    g = np.triu(g, 1)
    g = g + g.T                                                    # symmetric
    near = min(near, W)
    g[:near, :near] *= near_factor                                 # a fast local cluster
    np.fill_diagonal(g, GOODPUT_BPS)                               # diagonal is never read
    gi = np.rint(g).astype(np.int64)
    wmax = int(weight.max())
    table = np.zeros((W, W, wmax + 1), np.int64)
    for w in range(1, wmax + 1):
        table[:, :, w] = fetch_us(w * CHUNK_BYTES, gi)
    return table[:, :, weight]                                      # [src][req][v]


# ----------------------------------------------------------------------------
# the five workloads
# ----------------------------------------------------------------------------

CONFIGS = {
    0: dict(name="tiny-n2000-W4-k256", n=2000, W=4, k=256, mode=0, starts=1, rounds=3),
    1: dict(name="rag-n10000-W8-k1024", n=10_000, W=8, k=1024, mode=0, starts=4, rounds=5),
    2: dict(name="srcdep-n20000-W16-k2048", n=20_000, W=16, k=2048, mode=1, starts=8, rounds=5),
    3: dict(name="paper-n50000-W16-k4096", n=50_000, W=16, k=4096, mode=1, starts=16, rounds=6),
    4: dict(name="stress-n200000-W32-k8192", n=200_000, W=32, k=8192, mode=1, starts=32, rounds=4),
}


def make(cfg: int, seed: int = 0) -> Instance:
    c = CONFIGS[cfg]
    rng = np.random.default_rng(seed * 1000 + cfg)
    n, W = c["n"], c["W"]
    if cfg == 0:
        parent = _grow_random(rng, n, 8, 24, lambda r: int(r.geometric(0.5)))
        weight = np.ones(n, np.int32)
        classes = [m % 3 for m in range(W)]
        zipf_s, perm = 1.1, False
    elif cfg in (1, 2):
        parent = _rag_tree(rng, n)
        weight = np.ones(n, np.int32) if cfg == 1 else rng.integers(1, 3, size=n).astype(np.int32)
        classes = [0, 0, 0, 1, 1, 1, 2, 2] if cfg == 1 else [m % 3 for m in range(W)]
        zipf_s, perm = 0.9, False
    elif cfg == 3:
        parent = _mixed_tree(rng, n)
        weight = np.ones(n, np.int32)
        classes = [m % 3 for m in range(W)]
        zipf_s, perm = 1.0, True
    elif cfg == 4:
        parent = _stress_tree(rng, n)
        weight = rng.integers(1, 5, size=n).astype(np.int32)
        classes = [m % 3 for m in range(W)]
        zipf_s, perm = 1.0, True
    else:
        raise KeyError(cfg)
    depth = _depth_order(parent)
    counts = _leaf_demand(rng, parent, W, zipf_s, perm)
    demand = _propagate_up(parent, counts, depth)
    recompute = _recompute(weight, _prefix_tokens(parent, weight, depth), classes)
    if c["mode"] == 0:
        transfer = _transfer_requester(rng, weight, W, 0.3)
    else:
        transfer = _transfer_source(rng, weight, W, 0.5)
    budget = np.full(W, c["k"], np.int32)
    prof = dict(max_depth=int(depth.max()), leaves=int((np.bincount(parent[parent >= 0],
                minlength=n) == 0).sum()), classes=classes)
    return Instance(c["name"], n, W, parent, weight, demand, recompute,
                    np.ascontiguousarray(transfer), c["mode"], budget, c["starts"], c["rounds"],
                    seed, prof)


def random_small(rng, n, W, mode, k_max=4, w_max=1, demand_max=5, relabel=True) -> Instance:
    """A small random instance for brute-force checks (arbitrary node-id order)."""
    parent = np.full(n, -1, np.int32)
    for v in range(1, n):
        parent[v] = -1 if rng.random() < 0.2 else int(rng.integers(v))
    if relabel:
        perm = rng.permutation(n)           # new id of old node
        newp = np.full(n, -1, np.int32)
        for v in range(n):
            if parent[v] >= 0:
                newp[perm[v]] = perm[parent[v]]
        parent = newp
    weight = rng.integers(1, w_max + 1, size=n).astype(np.int32)
    demand = rng.integers(0, demand_max + 1, size=(W, n)).astype(np.int64)
    recompute = rng.integers(0, 50, size=(W, n)).astype(np.int64)
    if mode == 0:
        transfer = rng.integers(0, 50, size=(W, n)).astype(np.int64)
    else:
        transfer = rng.integers(0, 50, size=(W, W, n)).astype(np.int64)
    budget = rng.integers(0, k_max + 1, size=W).astype(np.int32)
    return Instance(f"random-n{n}-W{W}", n, W, parent, weight, demand, recompute, transfer, mode,
                    budget, 1, 3)


def random_orders(W: int, S: int, seed: int = 0) -> np.ndarray:
    """Explicit start orders: numpy permutations (an ABI input, so parity never
    depends on either side's own permutation generator)."""
    rng = np.random.default_rng(seed)
    return np.stack([rng.permutation(W) for _ in range(S)]).astype(np.int32)
