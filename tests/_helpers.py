"""Shared test helpers: workloads with drafted tokens, device copies, and the
comparison of library outputs with the oracle.

Tolerances: floating-point outputs of bf16 workloads within 2e-2 absolute
plus 1e-2 relative, of fp32 workloads within 1e-4 + 1e-4 relative.  Integer
outputs (argmax, accept, paths, cache bytes) are compared exactly, except
that non-strict nodes whose oracle margin lies within 1e-3 of tau, and rows
whose oracle top-2 logits are within 1e-4 (with their children), are
reported instead of counted (fp32
accumulation cannot decide them the same way as fp64); a sequence touching
such a node is checked for validity instead of equality.
"""
from __future__ import annotations

import numpy as np

import oracle
from paper_2609_02897_gb300 import synth

BAND = 1e-3
TIE = 1e-4


def tol(wl):
    return (2e-2, 1e-2) if wl.dtype == "bf16" else (1e-4, 1e-4)


def ranks_via_oracle(wl, rows=None):
    rows = wl.parents_needed() if rows is None else rows
    out = {}
    rows = np.asarray(rows)
    for i in range(0, len(rows), 256):
        chunk = rows[i:i + 256]
        top = oracle.topk_tokens(wl.hidden, wl.w, chunk, 5)
        for j, r in enumerate(chunk):
            out[int(r)] = top[j]
    return out


def prepared(cfg, small=True, rep=0, tree_override=None, overrides=None):
    wl = synth.make_workload(cfg, rep=rep, small=small, tree_override=tree_override,
                             overrides=overrides)
    synth.attach_tokens(wl, ranks_via_oracle(wl))
    return wl


def assert_close(got, ref, atol, rtol, what):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    err = np.abs(got - ref)
    lim = atol + rtol * np.abs(ref)
    bad = ~(err <= lim)
    if bad.any():
        idx = np.argwhere(bad)[:5]
        raise AssertionError(f"{what}: {int(bad.sum())} of {bad.size} outside tolerance "
                             f"(max err {np.nanmax(err):.3e}); first at {idx.tolist()}")
    return float(np.max(err)) if err.size else 0.0


def oracle_arrays(wl):
    return dict(q=wl.q, k_cache=wl.k_cache, v_cache=wl.v_cache, ctx_len=wl.ctx_len,
                tree_k=wl.tree_k, tree_v=wl.tree_v, parent=wl.parent, cu_nodes=wl.cu_nodes,
                page_table=wl.page_table, page_size=wl.page_size, hidden=wl.hidden, w=wl.w,
                tokens=wl.tokens)


def oracle_top2_gap(wl, rows):
    gaps = {}
    rows = np.asarray(rows)
    for i in range(0, len(rows), 256):
        chunk = rows[i:i + 256]
        lg = oracle.logits_rows(wl.hidden, wl.w, chunk)
        part = np.partition(lg, -2, axis=1)[:, -2:]
        for j, r in enumerate(chunk):
            gaps[int(r)] = float(part[j, 1] - part[j, 0])
    return gaps


class Report:
    def __init__(self):
        self.band_nodes = 0
        self.tie_rows = 0
        self.excluded_seqs = 0
        self.checked_seqs = 0
        self.max_err = {}

    def __repr__(self):
        return (f"band_nodes={self.band_nodes} tie_rows={self.tie_rows} "
                f"excluded_seqs={self.excluded_seqs} checked_seqs={self.checked_seqs} "
                f"max_err={self.max_err}")


def valid_path(parent_local, accept_local, path):
    """The path starts at the root, follows parent links, every non-root node is
    accepted, and no accepted path is longer."""
    if not path or path[0] != 0:
        return False
    for x, y in zip(path[:-1], path[1:]):
        if parent_local[y] != x or not accept_local[y]:
            return False
    n = len(parent_local)
    depth_ok = [False] * n
    best = 1
    for u in range(n):
        if u == 0:
            depth_ok[u] = True
        else:
            depth_ok[u] = depth_ok[parent_local[u]] and bool(accept_local[u])
    d = [0] * n
    for u in range(1, n):
        d[u] = d[parent_local[u]] + 1
        if depth_ok[u]:
            best = max(best, d[u] + 1)
    return len(path) == best


def reached_rows(wl, accept):
    """Roots, and every node whose parent is reached and which is accepted: the
    rows whose verdicts the accepted-path walk can need (a node is judged by its
    parent's row, and every walk moves from the root through accepted nodes)."""
    r = np.zeros(wl.T, bool)
    for b in range(wl.B):
        s, e = int(wl.cu_nodes[b]), int(wl.cu_nodes[b + 1])
        r[s] = True
        for i in range(s + 1, e):
            r[i] = r[s + int(wl.parent[i])] and int(accept[i]) == 1
    return r


def compare_verify(wl, tau, out, seqs=None, check_attn_nodes=None, rule=0, lazy=False):
    """Compares one verify step's outputs (numpy copies in `out`) with the
    oracle on the sequences `seqs` (all by default), the committed path under
    accepted-path reading `rule`.  Returns a Report.

    lazy: the step ran the lazy LM-head schedule, which computes only the rows
    of the roots and of the nodes reached through accepted nodes.  The rows it
    computed must be exactly that set under its own verdicts; the oracle then
    evaluates the same rows (Eq. 1 and the kappa rule on their children) and
    every computed statistic and every judged verdict is compared as for the
    every-row schedule.  Outside the reported band the verdicts agree, so the
    reached sets agree too; the rest keeps the documented fills."""
    rep = Report()
    atol, rtol = tol(wl)
    B = wl.B
    seqs = list(range(B)) if seqs is None else list(seqs)
    nodes = np.concatenate([np.arange(wl.cu_nodes[b], wl.cu_nodes[b + 1]) for b in seqs])
    gp = wl.global_parent()
    all_nodes = nodes
    if lazy:
        reach = ~np.isnan(out["row_max"])
        np.testing.assert_array_equal(reach, reached_rows(wl, out["accept"]),
                                      err_msg="lazy schedule: rows computed")
        nodes = nodes[reach[nodes]]

    # step 1: attention
    att_nodes = all_nodes if check_attn_nodes is None else np.asarray(check_attn_nodes)
    ref_attn = oracle.tree_attention(wl.q, wl.k_cache, wl.v_cache, wl.ctx_len, wl.tree_k,
                                     wl.tree_v, wl.parent, wl.cu_nodes, wl.page_table,
                                     wl.page_size, nodes=att_nodes)
    rep.max_err["attn"] = assert_close(out["attn_out"][att_nodes], ref_attn[att_nodes], atol, rtol,
                                       "attention output")

    # step 2: LM head + margin rule
    lm = oracle.lmhead_margin(wl.hidden, wl.w, wl.tokens, wl.parent, wl.cu_nodes, tau, rows=nodes)
    rep.max_err["row_max"] = assert_close(out["row_max"][nodes], lm["row_max"][nodes], atol, rtol,
                                          "row_max")
    rep.max_err["row_lse"] = assert_close(out["row_lse"][nodes], lm["row_lse"][nodes], atol, rtol,
                                          "row_lse")
    gaps = oracle_top2_gap(wl, nodes)
    tie = {r for r, g in gaps.items() if g < TIE}
    rep.tie_rows = len(tie)
    for r in nodes:
        if int(r) not in tie:
            assert out["row_argmax"][r] == lm["row_argmax"][r], f"argmax row {r}"
    if lazy:
        # judged nodes: those whose parent row was computed
        judged = set(int(c) for c in all_nodes if gp[c] >= 0 and reach[gp[c]])
        kids = np.array(sorted(judged), dtype=np.int64)
        rest = np.array([c for c in all_nodes if gp[c] >= 0 and int(c) not in judged],
                        dtype=np.int64)
        if len(rest):
            assert np.all(out["accept"][rest] == 0)
            assert np.all(np.isnan(out["ratio"][rest])) and np.all(np.isnan(out["l_draft"][rest]))
        unreached = all_nodes[~reach[all_nodes]]
        assert np.all(np.isnan(out["row_lse"][unreached]))
        assert np.all(out["row_argmax"][unreached] == -1)
    else:
        kids = np.array([c for c in nodes if gp[c] >= 0], dtype=np.int64)
    if len(kids):
        rep.max_err["l_draft"] = assert_close(out["l_draft"][kids], lm["l_draft"][kids], atol, rtol,
                                              "l_draft")
        rep.max_err["ratio"] = assert_close(out["ratio"][kids], lm["ratio"][kids], 1e-6, 5e-2,
                                            "ratio")
        assert np.all(out["ratio"][kids] <= 1.0) and np.all(out["ratio"][kids] >= 0.0)
    roots = np.array([c for c in all_nodes if gp[c] < 0])
    assert np.all(out["accept"][roots] == 1)
    band = set()
    for c in kids:
        # the threshold decides only non-strict nodes; strict ones hinge on the argmax
        strict = int(wl.tokens[c]) == int(lm["row_argmax"][gp[c]])
        if (abs(lm["ratio"][c] - tau) < BAND and not strict) or int(gp[c]) in tie:
            band.add(int(c))
            continue
        assert out["accept"][c] == lm["accept"][c], \
            f"accept node {c}: gpu {out['accept'][c]} oracle {lm['accept'][c]} ratio {lm['ratio'][c]}"
    if rule >= 2:
        # the greedy walks order promoted siblings by ratio: near-equal ratios
        # cannot be ordered alike in fp32 and fp64
        for u in nodes:
            sib = sorted((float(lm["ratio"][c]) for c in kids if gp[c] == u and lm["accept"][c] == 1
                          and int(wl.tokens[c]) != int(lm["row_argmax"][u])), reverse=True)
            if len(sib) > 1 and sib[0] - sib[1] < 1e-3:
                band.update(int(c) for c in kids if gp[c] == u)
    rep.band_nodes = len(band)

    # steps 3-4: path and commit
    for b in seqs:
        s, e = int(wl.cu_nodes[b]), int(wl.cu_nodes[b + 1])
        plen = int(out["path_len"][b])
        path = [int(x) for x in out["path"][b][:plen]]
        assert all(int(x) == -1 for x in out["path"][b][plen:])
        acc_gpu = out["accept"][s:e]
        if rule == 0:
            assert valid_path(list(wl.parent[s:e]), list(acc_gpu), path), f"seq {b} path {path}"
        # the walk itself, on the GPU's own verdicts, is exact
        own = oracle.accept_path(wl.parent[s:e], acc_gpu, out["row_argmax"][s:e], wl.tokens[s:e],
                                 [0, e - s], rule=rule, ratio=out["ratio"][s:e])
        assert path == own[0][0], f"seq {b} rule {rule}: gpu {path} walk on its verdicts {own[0][0]}"
        if band.intersection(range(s, e)):
            rep.excluded_seqs += 1
        else:
            rep.checked_seqs += 1
            paths, plens, bonus, npro = oracle.accept_path(
                wl.parent[s:e], lm["accept"][s:e], lm["row_argmax"][s:e], wl.tokens[s:e], [0, e - s],
                rule=rule, ratio=lm["ratio"][s:e])
            assert path == paths[0], f"seq {b}: gpu {path} oracle {paths[0]}"
            assert int(out["bonus"][b]) == int(bonus[0])
            assert int(out["n_promoted"][b]) == int(npro[0])
        assert int(out["ctx_len_out"][b]) == int(wl.ctx_len[b]) + plen
        # committed rows are the path's tree K/V, bit for bit
        for k, u in enumerate(path):
            slot = int(wl.ctx_len[b]) + k
            if wl.page_size == 0:
                kc = out["k_cache"][b, :, slot]
                vc = out["v_cache"][b, :, slot]
            else:
                page = wl.page_table[b, slot // wl.page_size]
                kc = out["k_cache"][page, :, slot % wl.page_size]
                vc = out["v_cache"][page, :, slot % wl.page_size]
            np.testing.assert_array_equal(kc, wl.tree_k[s + u])
            np.testing.assert_array_equal(vc, wl.tree_v[s + u])
    return rep


def untouched_cache_equal(wl, out, written_slots):
    """Every cache slot outside `written_slots` (list of (b, slot)) keeps its bytes."""
    kc, vc = out["k_cache"], out["v_cache"]
    if wl.page_size == 0:
        mask = np.ones((wl.B, wl.ctx_max), dtype=bool)
        for b, s in written_slots:
            mask[b, s] = False
        np.testing.assert_array_equal(kc.transpose(0, 2, 1, 3)[mask],
                                      wl.k_cache.transpose(0, 2, 1, 3)[mask])
        np.testing.assert_array_equal(vc.transpose(0, 2, 1, 3)[mask],
                                      wl.v_cache.transpose(0, 2, 1, 3)[mask])
    else:
        P = wl.k_cache.shape[0]
        mask = np.ones((P, wl.page_size), dtype=bool)
        for b, s in written_slots:
            mask[wl.page_table[b, s // wl.page_size], s % wl.page_size] = False
        np.testing.assert_array_equal(kc.transpose(0, 2, 1, 3)[mask],
                                      wl.k_cache.transpose(0, 2, 1, 3)[mask])
        np.testing.assert_array_equal(vc.transpose(0, 2, 1, 3)[mask],
                                      wl.v_cache.transpose(0, 2, 1, 3)[mask])
