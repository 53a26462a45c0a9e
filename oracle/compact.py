"""Oracle for committing the accepted nodes' K/V (Sec. 2: accepted draft tokens
are committed per target forward pass).

For k = 0 .. path_len[b]-1 the K and V rows of tree node path[b][k] (all KV
heads) are copied to cache slot ctx_len[b] + k of sequence b: directly in a
contiguous cache [B, Hkv, ctx_max, D], or through the page table (slot s lives
in page page_table[b, s // page_size] at offset s % page_size) in a paged pool
[P, Hkv, page_size, D].  New context lengths are ctx_len + path_len.
"""
import numpy as np


def kv_compact(k_cache, v_cache, tree_k, tree_v, cu_nodes, paths, ctx_len,
               page_table=None, page_size=0):
    """Returns (k_cache', v_cache', ctx_len_out) on copies of the caches."""
    kc = np.array(k_cache, copy=True)
    vc = np.array(v_cache, copy=True)
    out_len = np.array(ctx_len, dtype=np.int64).copy()
    for b, path in enumerate(paths):
        s = int(cu_nodes[b])
        for k, u in enumerate(path):
            slot = int(ctx_len[b]) + k
            if page_size == 0:
                kc[b, :, slot] = tree_k[s + u]
                vc[b, :, slot] = tree_v[s + u]
            else:
                page = int(page_table[b, slot // page_size])
                kc[page, :, slot % page_size] = tree_k[s + u]
                vc[page, :, slot % page_size] = tree_v[s + u]
        out_len[b] = int(ctx_len[b]) + len(path)
    return kc, vc, out_len
