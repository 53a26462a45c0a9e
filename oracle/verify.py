"""Oracle for one verify step: tree attention, LM head with the margin rule
(Eq. 1 and the kappa rule), the accepted-path choice and the K/V commit."""
from .attention import tree_attention
from .lmhead import lmhead_margin
from .accept import accept_path
from .compact import kv_compact


def verify_step(wl_arrays, tau, rule=0):
    """wl_arrays: mapping with q, k_cache, v_cache, ctx_len, tree_k, tree_v,
    parent, cu_nodes, page_table, page_size, hidden, w, tokens.  `rule`: the
    accepted-path reading (oracle.accept)."""
    a = wl_arrays
    out = tree_attention(a["q"], a["k_cache"], a["v_cache"], a["ctx_len"], a["tree_k"],
                         a["tree_v"], a["parent"], a["cu_nodes"], a.get("page_table"),
                         a.get("page_size", 0))
    lm = lmhead_margin(a["hidden"], a["w"], a["tokens"], a["parent"], a["cu_nodes"], tau)
    paths, plen, bonus, npro = accept_path(a["parent"], lm["accept"], lm["row_argmax"],
                                           a["tokens"], a["cu_nodes"], rule=rule,
                                           ratio=lm["ratio"])
    kc, vc, ctx_out = kv_compact(a["k_cache"], a["v_cache"], a["tree_k"], a["tree_v"],
                                 a["cu_nodes"], paths, a["ctx_len"], a.get("page_table"),
                                 a.get("page_size", 0))
    return dict(attn=out, paths=paths, path_len=plen, bonus=bonus, n_promoted=npro,
                k_cache=kc, v_cache=vc, ctx_len_out=ctx_out, **lm)
