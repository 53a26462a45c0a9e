"""Oracle for tree attention (the verify forward of Sec. 2 "Verify" and
Sec. 3.1: the target scores every drafted node in one pass).

For node i of sequence b and query head h (KV head g = h // (Hq / Hkv)) the
key set is the sequence's committed context, positions 0 .. ctx_len[b]-1,
followed by the tree ancestors of i from the root down to i itself.  Scores are
q . k / sqrt(D); the output is the softmax-weighted sum of the values.  The
ancestor set is found by walking the parent array (no bitmask).
"""
import math

import numpy as np


def ancestors_of(parent_local, i):
    """Local node ids on the root-to-i path, root first (i included)."""
    path = []
    u = int(i)
    while u >= 0:
        path.append(u)
        u = int(parent_local[u])
    return path[::-1]


def _context_kv(k_cache, v_cache, b, g, ctx, page_table, page_size):
    """Context keys/values of sequence b, KV head g, positions 0..ctx-1."""
    if page_size == 0:
        return k_cache[b, g, :ctx], v_cache[b, g, :ctx]
    pos = np.arange(ctx)
    pages = page_table[b, pos // page_size]
    off = pos % page_size
    return k_cache[pages, g, off], v_cache[pages, g, off]


def tree_attention(q, k_cache, v_cache, ctx_len, tree_k, tree_v, parent, cu_nodes,
                   page_table=None, page_size=0, nodes=None):
    """Returns O [T, Hq, D] in float64 (rows not in `nodes` are left as NaN).

    q [T,Hq,D]; tree_k/tree_v [T,Hkv,D]; contiguous cache [B,Hkv,ctx_max,D]
    or paged pool [P,Hkv,page_size,D] with page_table [B, pages]; parent holds
    local ids (-1 at each root); cu_nodes [B+1] delimits the sequences.
    """
    q = np.asarray(q, dtype=np.float64)
    T, Hq, D = q.shape
    Hkv = tree_k.shape[1]
    G = Hq // Hkv
    out = np.full((T, Hq, D), np.nan)
    B = len(cu_nodes) - 1
    want = None if nodes is None else set(int(t) for t in nodes)
    scale = 1.0 / math.sqrt(D)
    for b in range(B):
        s, e = int(cu_nodes[b]), int(cu_nodes[b + 1])
        par = parent[s:e]
        ctx = int(ctx_len[b])
        for g in range(Hkv):
            kc, vc = _context_kv(k_cache, v_cache, b, g, ctx, page_table, page_size)
            kc = np.asarray(kc, dtype=np.float64)
            vc = np.asarray(vc, dtype=np.float64)
            for i in range(e - s):
                t = s + i
                if want is not None and t not in want:
                    continue
                anc = [s + a for a in ancestors_of(par, i)]
                keys = np.concatenate([kc, np.asarray(tree_k[anc, g], dtype=np.float64)])
                vals = np.concatenate([vc, np.asarray(tree_v[anc, g], dtype=np.float64)])
                # the G query heads that share KV head g, one softmax row each
                sc = q[t, g * G:(g + 1) * G] @ keys.T * scale
                p = np.exp(sc - sc.max(axis=1, keepdims=True))
                p /= p.sum(axis=1, keepdims=True)
                out[t, g * G:(g + 1) * G] = p @ vals
    return out
