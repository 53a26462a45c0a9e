"""bench.py's algorithmic-work helpers: the tree keys a step's attention sees
(against the oracle's ancestor lists) and the lazy schedule's computed rows and
weight passes (against a hand-worked tree)."""
import os
import sys

import numpy as np

import oracle
from paper_2609_02897_gb300 import synth

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
import bench  # noqa: E402


def test_tree_keys_match_the_oracle_ancestors():
    for cfg in sorted(synth.WORKLOADS):
        wl = synth.make_workload(cfg, small=True)
        for b in range(wl.B):
            s, e = int(wl.cu_nodes[b]), int(wl.cu_nodes[b + 1])
            par = wl.parent[s:e]
            assert bench.tree_keys(par) == sum(len(oracle.ancestors_of(par, i))
                                               for i in range(e - s)), (cfg, b)


def test_tree_keys_closed_forms():
    assert bench.tree_keys(np.array([-1])) == 1
    chain = np.arange(-1, 7)                       # 8-node chain: 1 + 2 + ... + 8
    assert bench.tree_keys(chain) == 36
    star = np.array([-1] + [0] * 9)                # root + 9 leaves: 1 + 9 * 2
    assert bench.tree_keys(star) == 19


def test_lazy_work_counts_rows_and_levels():
    class W:
        pass
    wl = W()
    # two sequences: 0-1-2-3 chain with 4 -> 0; 5 root with 6, 7 children
    wl.parent = np.array([-1, 0, 1, 2, 0, -1, 0, 0], np.int32)
    wl.cu_nodes = np.array([0, 5, 8], np.int32)
    wl.B, wl.T = 2, 8
    nan = float("nan")
    # computed: 0, 1, 2 (depths 0..2) and 5, 7 (depths 0..1)
    row_max = np.array([1, 1, 1, nan, nan, 1, nan, 1], np.float32)
    assert bench.lazy_work(wl, row_max) == (5, 3)
    assert bench.lazy_work(wl, np.full(8, nan, np.float32)) == (0, 0)


def _oracle_as_outputs(wl, tau):
    """The oracle's verify step laid out like the library's outputs (its
    committed cache included), for exercising the bench's parity check."""
    r = oracle.verify_step(bench.oracle_arrays(wl), tau)
    out = {k: np.asarray(r[k]) for k in ("row_max", "row_argmax", "row_lse", "l_draft", "ratio",
                                         "accept", "path_len", "bonus", "n_promoted",
                                         "ctx_len_out")}
    out["attn_out"] = r["attn"]
    path = np.full((wl.B, wl.max_path), -1)
    for b, p in enumerate(r["paths"]):
        path[b, :len(p)] = p
    out["path"] = path
    kc, vc = r["k_cache"], r["v_cache"]

    def rows(b, slot):
        if wl.page_size == 0:
            return kc[b, :, slot], vc[b, :, slot]
        page = int(wl.page_table[b, slot // wl.page_size])
        return kc[page, :, slot % wl.page_size], vc[page, :, slot % wl.page_size]
    return out, r, rows


def _prepared(cfg):
    wl = synth.make_workload(cfg, small=True)
    rows = wl.parents_needed()
    top = oracle.topk_tokens(wl.hidden, wl.w, rows, 5)
    synth.attach_tokens(wl, {int(r): top[j] for j, r in enumerate(rows)})
    return wl


def test_parity_check_accepts_the_oracle_and_catches_planted_mistakes():
    wl = _prepared(2)
    tau = 0.3
    out, full, rows = _oracle_as_outputs(wl, tau)
    rep = bench.parity_check(wl, tau, out, rows, full=full)
    assert rep["ok"], rep
    rep2 = bench.parity_check(wl, tau, out, rows)          # recomputed by the oracle itself
    assert rep2["ok"] and rep2["checked_seqs"] + rep2["excluded_seqs"] == wl.B, rep2
    plen = int(out["path_len"][0])
    for plant in ("attn", "argmax", "accept", "path", "commit"):
        bad = {k: np.array(v, copy=True) for k, v in out.items()}
        bad_rows = rows
        if plant == "attn":
            bad["attn_out"][3, 1, 5] += 0.5
        elif plant == "argmax":
            bad["row_argmax"][0] += 1
        elif plant == "accept":
            c = 1 + int(np.argmax(np.abs(full["ratio"][1:] - tau) > 0.01))
            bad["accept"][c] ^= 1
        elif plant == "path":
            bad["bonus"][0] += 1
        else:
            def bad_rows(b, slot):
                k, v = rows(b, slot)
                if slot == int(wl.ctx_len[b]) + plen - 1:
                    k = np.array(k, copy=True)
                    k[0, 0] += 1.0
                return k, v
        rep = bench.parity_check(wl, tau, bad, bad_rows, full=full)
        assert not rep["ok"], plant


def test_parity_check_on_sampled_sequences():
    wl = _prepared(3)
    tau = 0.5
    out, _, rows = _oracle_as_outputs(wl, tau)
    rep = bench.parity_check(wl, tau, out, rows, seqs=[0, 2])
    assert rep["ok"] and rep["checked_seqs"] + rep["excluded_seqs"] == 2, rep
    bad = {k: np.array(v, copy=True) for k, v in out.items()}
    s = int(wl.cu_nodes[2])
    bad["row_lse"][s + 1] += 0.5
    assert not bench.parity_check(wl, tau, bad, rows, seqs=[0, 2])["ok"]


def test_lmhead_traffic_is_null_for_other_sources(monkeypatch):
    monkeypatch.setattr(bench, "LMHEAD_TRAFFIC_SOURCE", "0" * 16)
    assert bench.lmhead_traffic(2) is None
    monkeypatch.setattr(bench, "LMHEAD_TRAFFIC_SOURCE", bench.lmhead_source_hash())
    assert bench.lmhead_traffic(2) == bench.LMHEAD_TRAFFIC_BY_CONFIG[2]
