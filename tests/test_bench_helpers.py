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
