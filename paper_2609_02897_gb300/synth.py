"""Seeded synthetic verify-step workloads.

This module only draws inputs: random tensors, draft-tree shapes, context
lengths, page tables and the drafted-token mixture.  It contains none of the
verification arithmetic (no attention, no LM head, no margin rule, no walk).
The drafted-token mixture needs the target model's top-5 tokens of each parent
row; that ranking is computed by the caller and handed in (`attach_tokens`).

Workload shapes follow the paper's 8B-class targets (Sec. 4.1 "Models":
Llama-3.1-8B, DeepSeek-R1-Distill-Llama-8B, Qwen3-8B) and its draft-tree
triplets (Sec. 3.3, Table 4).  All dense values are drawn in float32 and, for
bf16 workloads, rounded to the nearest bfloat16 before use, so every consumer
sees bit-identical inputs.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Callable, Optional

import numpy as np

# --------------------------------------------------------------------------
# Configurations.  Names describe the workload; sizes are the full ones.
# --------------------------------------------------------------------------

WORKLOADS = {
    1: dict(name="tiny-fp32", dtype="f32", B=1, ctx=(256, 256), Hq=4, Hkv=4, D=64,
            hidden=256, vocab=4096, tree="c1", tau=(1.0, 0.3), page_size=0),
    2: dict(name="llama3.1-8b-b1-ctx2048-eagle60", dtype="bf16", B=1, ctx=(2048, 2048),
            Hq=32, Hkv=8, D=128, hidden=4096, vocab=128256,
            tree=("eagle", 8, 10, 60), tau=(0.3,), page_size=0),
    3: dict(name="llama3.1-8b-ragged-b16", dtype="bf16", B=16, ctx=(512, 4096),
            Hq=32, Hkv=8, D=128, hidden=4096, vocab=128256,
            tree=("ragged", (16, 96), (3, 10), (1, 12)), tau=(0.5,), page_size=0),
    4: dict(name="qwen3-8b-b8-ctx16384-tree64", dtype="bf16", B=8, ctx=(16384, 16384),
            Hq=32, Hkv=8, D=128, hidden=4096, vocab=151936,
            tree=("grown", 64, 10, 10), tau=(0.3,), page_size=0, decay=(0.8, 0.1)),
    5: dict(name="llama3.1-8b-paged-b64-ctx8192-tree128", dtype="bf16", B=64,
            ctx=(8192, 8192), Hq=32, Hkv=8, D=128, hidden=4096, vocab=128256,
            tree=("grown", 128, 12, 16), tau=(1.0, 0.5, 0.3, 0.1), page_size=16),
    # The draft trees the paper itself verifies (Sec. 3.3, Sec. 4.1 and its
    # configuration table), as (n_steps, top-k, ndt) with ndt counting the
    # root: the deep chain (7,1,8), the wide end of the dynamic range (3,4,4),
    # and EAGLE-3's static (3,1,4); margin threshold kappa = 0.2 as in the
    # paper's main results, and 1.0 (strict verification).
    6: dict(name="llama3.1-8b-b1-ctx2048-chain-7-1-8", dtype="bf16", B=1, ctx=(2048, 2048),
            Hq=32, Hkv=8, D=128, hidden=4096, vocab=128256,
            tree=("eagle", 7, 1, 8), tau=(0.2, 1.0), page_size=0),
    7: dict(name="llama3.1-8b-b1-ctx2048-tree-3-4-4", dtype="bf16", B=1, ctx=(2048, 2048),
            Hq=32, Hkv=8, D=128, hidden=4096, vocab=128256,
            tree=("eagle", 3, 4, 4), tau=(0.2, 1.0), page_size=0),
    8: dict(name="llama3.1-8b-b1-ctx2048-chain-3-1-4", dtype="bf16", B=1, ctx=(2048, 2048),
            Hq=32, Hkv=8, D=128, hidden=4096, vocab=128256,
            tree=("eagle", 3, 1, 4), tau=(0.2, 1.0), page_size=0),
}

# Reduced variants with the same structure (tree recipe, GQA group, paging,
# ragged lengths) but sizes an fp64 CPU oracle finishes in seconds.  Every
# dimension still spans several kernel tiles and ends in a ragged tail.
SMALL = {
    1: dict(),
    2: dict(ctx=(300, 300), Hq=8, Hkv=2, hidden=512, vocab=5000),
    3: dict(B=5, ctx=(40, 333), Hq=8, Hkv=2, hidden=384, vocab=3001),
    4: dict(B=2, ctx=(1100, 1100), Hq=8, Hkv=2, hidden=512, vocab=4999),
    5: dict(B=6, ctx=(200, 200), Hq=8, Hkv=2, hidden=512, vocab=5000),
    6: dict(ctx=(300, 300), Hq=8, Hkv=2, hidden=512, vocab=5000),
    7: dict(ctx=(300, 300), Hq=8, Hkv=2, hidden=512, vocab=5000),
    8: dict(ctx=(300, 300), Hq=8, Hkv=2, hidden=512, vocab=5000),
}

P_TOP1 = 0.5      # drafted token = the target's top-1 of the parent row
P_RANK2TO5 = 0.3  # drafted token = one of the parent row's rank-2..5 tokens
# remainder (0.2): uniform over the vocabulary


_ROUND_CHUNK = 1 << 16


def _round_bf16_inplace(x: np.ndarray) -> np.ndarray:
    """Rounds a contiguous float32 array to bfloat16 values in place, in
    cache-sized chunks of 32-bit integer arithmetic (the sum wraps modulo 2^32
    only for NaN patterns, which then end as the wider computation's would)."""
    u = x.reshape(-1).view(np.uint32)
    for i in range(0, u.size, _ROUND_CHUNK):
        c = u[i:i + _ROUND_CHUNK]
        t = c >> 16
        t &= 1
        t += 0x7FFF
        c += t
        c &= np.uint32(0xFFFF0000)
    return x


def round_bf16(x: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bfloat16 (ties to even); float32 out."""
    return _round_bf16_inplace(np.array(x, dtype=np.float32, order="C", copy=True))


def _normal(rng: np.random.Generator, shape, std: float, bf16: bool) -> np.ndarray:
    x = rng.standard_normal(shape, dtype=np.float32)
    if std != 1.0:
        x *= np.float32(std)
    return _round_bf16_inplace(x) if bf16 else x


# --------------------------------------------------------------------------
# Draft-tree shapes.  A tree is a parent array with parent[0] = -1 and
# 0 <= parent[i] < i (topological numbering).
# --------------------------------------------------------------------------

def depths(parent: np.ndarray) -> np.ndarray:
    d = np.zeros(len(parent), dtype=np.int64)
    for i in range(1, len(parent)):
        d[i] = d[parent[i]] + 1
    return d


def bfs_renumber(parent: list[int], key: Optional[list] = None) -> np.ndarray:
    """Renumber nodes by (depth, key, old index); returns a topological parent array."""
    n = len(parent)
    d = [0] * n
    for i in range(n):  # parents may have larger old ids here; resolve iteratively
        j, k = i, 0
        while parent[j] >= 0:
            j, k = parent[j], k + 1
        d[i] = k
    key = key if key is not None else [0] * n
    order = sorted(range(n), key=lambda i: (d[i], key[i], i))
    new_id = {old: new for new, old in enumerate(order)}
    out = np.full(n, -1, dtype=np.int32)
    for old in range(n):
        if parent[old] >= 0:
            out[new_id[old]] = new_id[parent[old]]
    return out


def tree_fixed_c1() -> np.ndarray:
    """Root chain of depth 4 (0-1-2-3-4) plus side leaves 5, 6, 7 under 0, 1, 2."""
    return np.array([-1, 0, 1, 2, 3, 0, 1, 2], dtype=np.int32)


def tree_chain(n: int) -> np.ndarray:
    return np.arange(-1, n - 1, dtype=np.int32)


def tree_eagle(rng: np.random.Generator, depth: int, topk: int, n_nodes: int) -> np.ndarray:
    """EAGLE-2-style tree: expand the top-k frontier per depth with Dirichlet(1)
    branch probabilities, keep the top-(n_nodes-1) candidates by path score
    (ancestor-closed) plus the root, and number them by (depth, -score)."""
    scores, parents, cdepth = [], [], []
    frontier = [(1.0, -1)]
    for d in range(1, depth + 1):
        new = []
        for s, cid in frontier:
            w = rng.dirichlet(np.ones(topk))
            for j in range(topk):
                scores.append(s * float(w[j]))
                parents.append(cid)
                cdepth.append(d)
                new.append((scores[-1], len(scores) - 1))
        new.sort(key=lambda t: (-t[0], t[1]))
        frontier = new[:topk]
    order = sorted(range(len(scores)), key=lambda i: (-scores[i], i))
    chosen: list[int] = []
    chosen_set = set()
    for i in order:
        if len(chosen) == n_nodes - 1:
            break
        if parents[i] == -1 or parents[i] in chosen_set:
            chosen.append(i)
            chosen_set.add(i)
    # local list: node 0 = root, then chosen candidates
    loc = {cid: k + 1 for k, cid in enumerate(chosen)}
    par = [-1] + [0 if parents[c] == -1 else loc[parents[c]] for c in chosen]
    key = [0.0] + [-scores[c] for c in chosen]
    return bfs_renumber(par, key)


def tree_grown(rng: np.random.Generator, n: int, depth: int, width: int) -> np.ndarray:
    """A spine of the given depth, then random growth: each new node hangs off a
    uniformly chosen node with depth < `depth` and fewer than `width` children.
    Stops early when no node is eligible (capacity smaller than n)."""
    parent, d, nch = [-1], [0], [0]
    for k in range(1, min(depth, n - 1) + 1):
        parent.append(k - 1)
        d.append(k)
        nch[k - 1] += 1
        nch.append(0)
    while len(parent) < n:
        elig = [u for u in range(len(parent)) if d[u] < depth and nch[u] < width]
        if not elig:
            break
        u = elig[int(rng.integers(len(elig)))]
        parent.append(u)
        d.append(d[u] + 1)
        nch[u] += 1
        nch.append(0)
    return bfs_renumber(parent)


def random_topological_relabel(parent: np.ndarray, rng: np.random.Generator) -> np.ndarray:
    """Random relabelling that keeps node 0 the root and parent[i] < i."""
    n = len(parent)
    children = [[] for _ in range(n)]
    for i in range(1, n):
        children[parent[i]].append(i)
    ready, order = [0], []
    while ready:
        j = int(rng.integers(len(ready)))
        u = ready.pop(j)
        order.append(u)
        ready.extend(children[u])
    new_id = {old: new for new, old in enumerate(order)}
    out = np.full(n, -1, dtype=np.int32)
    for old in range(1, n):
        out[new_id[old]] = new_id[parent[old]]
    return out


# --------------------------------------------------------------------------
# Workloads
# --------------------------------------------------------------------------

@dataclasses.dataclass
class Workload:
    config: int
    name: str
    dtype: str                 # "f32" | "bf16"
    B: int
    Hq: int
    Hkv: int
    D: int
    hidden_dim: int
    vocab: int
    page_size: int             # 0 = contiguous cache
    taus: tuple
    ctx_len: np.ndarray        # [B] int32
    ctx_max: int               # cache slots per sequence (contiguous) / per page-table row
    parent: np.ndarray         # [T] int32, local parent ids, -1 at each root
    cu_nodes: np.ndarray       # [B+1] int32
    q: np.ndarray              # [T, Hq, D]
    tree_k: np.ndarray         # [T, Hkv, D]
    tree_v: np.ndarray         # [T, Hkv, D]
    k_cache: np.ndarray        # [B, Hkv, ctx_max, D] or [P, Hkv, page, D]
    v_cache: np.ndarray
    page_table: Optional[np.ndarray]  # [B, ctx_max // page] int32 or None
    hidden: np.ndarray         # [T, hidden]
    w: np.ndarray              # [V, hidden]
    p_top1: np.ndarray         # [T] per-node top-1 probability of the mixture
    max_path: int
    tokens: Optional[np.ndarray] = None   # [T] int32, set by attach_tokens
    seed: int = 0

    @property
    def T(self) -> int:
        return int(self.cu_nodes[-1])

    @property
    def num_pages(self) -> int:
        return 0 if self.page_size == 0 else int(self.k_cache.shape[0])

    def nodes_of(self, b: int) -> range:
        return range(int(self.cu_nodes[b]), int(self.cu_nodes[b + 1]))

    def global_parent(self) -> np.ndarray:
        gp = self.parent.astype(np.int64).copy()
        for b in range(self.B):
            s = int(self.cu_nodes[b])
            seg = gp[s:int(self.cu_nodes[b + 1])]
            seg[seg >= 0] += s
        return gp

    def parents_needed(self) -> np.ndarray:
        """Global ids of the rows whose ranking the token mixture needs."""
        gp = self.global_parent()
        return np.unique(gp[gp >= 0])


def _spec(config: int, small: bool, overrides: Optional[dict] = None) -> dict:
    s = dict(WORKLOADS[config])
    if small:
        s.update(SMALL[config])
    if overrides:
        s.update(overrides)
    return s


def make_workload(config: int, rep: int = 0, small: bool = False,
                  tree_override: Optional[list] = None,
                  overrides: Optional[dict] = None) -> Workload:
    """Draw every input of one verify step except the drafted tokens.

    Seeds: numpy PCG64 with seed 1000*config + rep (+ 500 for the reduced
    variant).  Weights ~ N(0, 0.02); hidden states, queries, keys and values
    ~ N(0, 1).
    """
    s = _spec(config, small, overrides)
    seed = 1000 * config + rep + (500 if small else 0)
    rng = np.random.Generator(np.random.PCG64(seed))
    bf16 = s["dtype"] == "bf16"
    B = s["B"]

    # trees
    trees = []
    p1 = []
    for b in range(B):
        t = s["tree"]
        if tree_override is not None:
            par = np.asarray(tree_override[b % len(tree_override)], dtype=np.int32)
        elif t == "c1":
            par = tree_fixed_c1()
        elif t[0] == "eagle":
            par = tree_eagle(rng, t[1], t[2], t[3])
        elif t[0] == "ragged":
            n = int(rng.integers(t[1][0], t[1][1] + 1))
            dep = int(rng.integers(t[2][0], t[2][1] + 1))
            wid = int(rng.integers(t[3][0], t[3][1] + 1))
            par = tree_grown(rng, n, dep, wid)
        elif t[0] == "grown":
            par = tree_grown(rng, t[1], t[2], t[3])
        else:
            raise ValueError(t)
        trees.append(par)
        dep = depths(par)
        if "decay" in s:
            hi, lo = s["decay"]
            maxd = max(1, s["tree"][2])
            pv = hi - (hi - lo) * (np.maximum(dep, 1) - 1) / max(1, maxd - 1)
        else:
            pv = np.full(len(par), P_TOP1)
        p1.append(pv)
    sizes = [len(p) for p in trees]
    cu = np.zeros(B + 1, dtype=np.int32)
    cu[1:] = np.cumsum(sizes)
    T = int(cu[-1])
    parent = np.concatenate(trees).astype(np.int32)
    max_depth = max(int(depths(p).max()) for p in trees)
    max_path = max_depth + 1

    lo, hi = s["ctx"]
    ctx_len = rng.integers(lo, hi + 1, size=B).astype(np.int32) if hi > lo \
        else np.full(B, lo, dtype=np.int32)

    Hq, Hkv, D = s["Hq"], s["Hkv"], s["D"]
    q = _normal(rng, (T, Hq, D), 1.0, bf16)
    tree_k = _normal(rng, (T, Hkv, D), 1.0, bf16)
    tree_v = _normal(rng, (T, Hkv, D), 1.0, bf16)

    ps = s["page_size"]
    need = int(ctx_len.max()) + max_path
    if ps == 0:
        ctx_max = int(math.ceil(need / 64.0) * 64)
        k_cache = _normal(rng, (B, Hkv, ctx_max, D), 1.0, bf16)
        v_cache = _normal(rng, (B, Hkv, ctx_max, D), 1.0, bf16)
        page_table = None
    else:
        pages_per_seq = int(math.ceil(need / ps))
        ctx_max = pages_per_seq * ps
        P = B * pages_per_seq + 7          # a few spare pages nobody maps
        perm = rng.permutation(P).astype(np.int32)
        page_table = perm[:B * pages_per_seq].reshape(B, pages_per_seq).copy()
        k_cache = _normal(rng, (P, Hkv, ps, D), 1.0, bf16)
        v_cache = _normal(rng, (P, Hkv, ps, D), 1.0, bf16)

    hidden = _normal(rng, (T, s["hidden"]), 1.0, bf16)
    w = _normal(rng, (s["vocab"], s["hidden"]), 0.02, bf16)

    return Workload(config=config, name=s["name"] + ("-small" if small else ""),
                    dtype=s["dtype"], B=B, Hq=Hq, Hkv=Hkv, D=D,
                    hidden_dim=s["hidden"], vocab=s["vocab"], page_size=ps,
                    taus=tuple(s["tau"]), ctx_len=ctx_len, ctx_max=ctx_max,
                    parent=parent, cu_nodes=cu, q=q, tree_k=tree_k, tree_v=tree_v,
                    k_cache=k_cache, v_cache=v_cache, page_table=page_table,
                    hidden=hidden, w=w, p_top1=np.concatenate(p1), max_path=max_path,
                    seed=seed)


def attach_tokens(wl: Workload, ranks: dict | Callable[[int], np.ndarray]) -> np.ndarray:
    """Draw the drafted token of every non-root node.

    ranks[p] (global row id p) lists the target model's top-5 tokens of row p in
    rank order; it is needed for every row that has children.  Mixture per
    child: the parent row's top-1 with probability p_top1 (per node), one of the
    rank-2..5 tokens (uniformly) with probability 0.6*(1-p_top1) (0.3 when
    p_top1 = 0.5), else a uniform token.  Sibling tokens are kept distinct, as
    in top-k drafting.  Root tokens (the last committed token) are uniform.
    """
    rng = np.random.Generator(np.random.PCG64([wl.seed, 7]))
    get = ranks if callable(ranks) else (lambda p: ranks[p])
    gp = wl.global_parent()
    tokens = np.zeros(wl.T, dtype=np.int32)
    V = wl.vocab
    used: dict[int, set] = {}
    for t in range(wl.T):
        p = int(gp[t])
        if p < 0:
            tokens[t] = int(rng.integers(V))
            continue
        sib = used.setdefault(p, set())
        r = np.asarray(get(p))
        p1 = float(wl.p_top1[t])
        pr = (1.0 - p1) * (P_RANK2TO5 / (1.0 - P_TOP1))
        tok = None
        for _ in range(64):
            u = float(rng.random())
            if u < p1:
                cand = int(r[0])
            elif u < p1 + pr:
                cand = int(r[int(rng.integers(1, 5))])
            else:
                cand = int(rng.integers(V))
            if cand not in sib:
                tok = cand
                break
        while tok is None:
            cand = int(rng.integers(V))
            if cand not in sib:
                tok = cand
        sib.add(tok)
        tokens[t] = tok
    wl.tokens = tokens
    return tokens


def subtree_sizes(parent: np.ndarray) -> np.ndarray:
    n = len(parent)
    sz = np.ones(n, dtype=np.int64)
    for i in range(n - 1, 0, -1):
        sz[parent[i]] += sz[i]
    return sz
