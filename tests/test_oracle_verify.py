"""The oracle's verify step on reduced synthetic workloads: the chained call
agrees with the individual steps, and its outputs satisfy the invariants of
each step."""
import numpy as np
import pytest

import oracle
from paper_2609_02897_gb300 import synth


def _arrays(wl):
    return dict(q=wl.q, k_cache=wl.k_cache, v_cache=wl.v_cache, ctx_len=wl.ctx_len,
                tree_k=wl.tree_k, tree_v=wl.tree_v, parent=wl.parent, cu_nodes=wl.cu_nodes,
                page_table=wl.page_table, page_size=wl.page_size, hidden=wl.hidden, w=wl.w,
                tokens=wl.tokens)


def _with_tokens(wl):
    rows = wl.parents_needed()
    top = oracle.topk_tokens(wl.hidden, wl.w, rows, 5)
    synth.attach_tokens(wl, {int(r): top[j] for j, r in enumerate(rows)})
    return wl


@pytest.mark.parametrize("cfg", [1, 5])
def test_verify_step_chain(cfg):
    wl = _with_tokens(synth.make_workload(cfg, small=True))
    tau = wl.taus[-1]
    out = oracle.verify_step(_arrays(wl), tau)
    lm = oracle.lmhead_margin(wl.hidden, wl.w, wl.tokens, wl.parent, wl.cu_nodes, tau)
    np.testing.assert_array_equal(out["accept"], lm["accept"])
    gp = wl.global_parent()
    for b in range(wl.B):
        s = int(wl.cu_nodes[b])
        path = out["paths"][b]
        assert path[0] == 0
        for x, y in zip(path[:-1], path[1:]):
            assert wl.parent[s + y] == x and out["accept"][s + y] == 1
        assert out["ctx_len_out"][b] == wl.ctx_len[b] + len(path)
        assert out["bonus"][b] == out["row_argmax"][s + path[-1]]
    # the mixture makes roughly half of the drafted tokens strict matches
    strict = [wl.tokens[c] == out["row_argmax"][gp[c]] for c in range(wl.T) if gp[c] >= 0]
    assert 0.25 < np.mean(strict) < 0.75
