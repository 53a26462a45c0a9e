"""Pins for the accepted-path oracle: exhaustive comparison with two other
formulations on every small tree, hand-worked cases, and the reductions the
paper implies (strict greedy verification at kappa = 1, chains)."""
import itertools
import json
import os

import numpy as np
import pytest

import oracle
from paper_2609_02897_gb300 import synth

GOLDEN = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_settings.json")))


def _dfs_best(parent, accept):
    """Bottom-up recursion: the best path below u is u followed by the best of
    its accepted children's best paths (longest, then lexicographically smallest)."""
    n = len(parent)
    children = [[] for _ in range(n)]
    for i in range(1, n):
        children[parent[i]].append(i)

    def best(u):
        cand = [best(c) for c in children[u] if accept[c]]
        if not cand:
            return [u]
        L = max(len(c) for c in cand)
        return [u] + min(c for c in cand if len(c) == L)
    return best(0)


def _height_walk(parent, accept):
    """Heights of accepted subtrees, then a root-down walk to the lowest-index
    child of maximal height."""
    n = len(parent)
    h = [1] * n
    for i in range(n - 1, 0, -1):
        if accept[i]:
            h[parent[i]] = max(h[parent[i]], h[i] + 1)
    path = [0]
    u = 0
    while True:
        nxt = [c for c in range(1, n) if parent[c] == u and accept[c] and h[c] == h[u] - 1]
        if not nxt:
            return path
        u = min(nxt)
        path.append(u)


def _all_trees(n):
    for ps in itertools.product(*[range(i) for i in range(1, n)]):
        yield [-1] + list(ps)


@pytest.mark.parametrize("n", [1, 2, 3, 4, 5, 6])
def test_exhaustive_small_trees(n):
    for parent in _all_trees(n):
        for bits in itertools.product([0, 1], repeat=n - 1):
            acc = [1] + list(bits)
            paths, plen, _, _ = oracle.accept_path(np.array(parent), np.array(acc),
                                                   np.zeros(n, dtype=int), np.zeros(n, dtype=int),
                                                   [0, n])
            ref = _dfs_best(parent, acc)
            assert paths[0] == ref, (parent, acc)
            assert plen[0] == len(ref)
            assert _height_walk(parent, acc) == ref


def test_random_larger_trees_random_numbering():
    rng = np.random.default_rng(0)
    for trial in range(200):
        par = synth.tree_grown(rng, int(rng.integers(2, 60)), int(rng.integers(1, 9)),
                               int(rng.integers(1, 6)))
        par = synth.random_topological_relabel(par, rng)
        acc = (rng.random(len(par)) < 0.7).astype(int)
        acc[0] = 1
        paths, _, _, _ = oracle.accept_path(par, acc, np.zeros(len(par), int),
                                            np.zeros(len(par), int), [0, len(par)])
        assert paths[0] == _dfs_best(list(par), list(acc)) == _height_walk(list(par), list(acc))


def test_hand_worked_cases():
    # Tree:        0
    #            /   \
    #           1     2
    #          / \     \
    #         3   4     5
    #                    \
    #                     6
    parent = np.array([-1, 0, 0, 1, 1, 2, 5])
    tokens = np.array([9, 10, 11, 12, 13, 14, 15])
    # row_argmax chosen so that strict matches are: 1 (under 0), 4 (under 1), 6 (under 5)
    row_argmax = np.array([10, 13, 99, 99, 99, 15, 77])
    cu = [0, 7]
    # (a) everything accepted: longest is 0-2-5-6 (length 4)
    p, L, bonus, npro = oracle.accept_path(parent, np.ones(7, int), row_argmax, tokens, cu)
    assert p[0] == [0, 2, 5, 6] and L[0] == 4
    assert bonus[0] == row_argmax[6]
    # nodes 2 (tok 11 vs argmax 10) and 5 (tok 14 vs 99) promoted; 6 strict
    assert npro[0] == 2
    # (b) node 6 rejected: 0-1-3, 0-1-4 and 0-2-5 all have length 3 -> lexicographic 0-1-3
    acc = np.array([1, 1, 1, 1, 1, 1, 0])
    p, L, bonus, npro = oracle.accept_path(parent, acc, row_argmax, tokens, cu)
    assert p[0] == [0, 1, 3] and L[0] == 3 and bonus[0] == row_argmax[3]
    assert npro[0] == 1   # node 3 (tok 12 vs argmax of node 1 = 13) promoted; node 1 strict
    # (c) nodes 1 and 2 rejected: only the root
    acc = np.array([1, 0, 0, 1, 1, 1, 1])
    p, L, bonus, npro = oracle.accept_path(parent, acc, row_argmax, tokens, cu)
    assert p[0] == [0] and L[0] == 1 and bonus[0] == row_argmax[0] and npro[0] == 0


def test_kappa_one_matches_classic_greedy_verification():
    """With kappa = 1 and distinct sibling tokens the accepted path is the
    textbook greedy one: from the root, follow the child whose token equals the
    target's argmax until none does."""
    rng = np.random.default_rng(1)
    V, K = 6, 3
    for trial in range(100):
        par = synth.tree_grown(rng, int(rng.integers(2, 25)), 5, 4)
        n = len(par)
        hidden = rng.standard_normal((n, K))
        W = rng.standard_normal((V, K))
        children = [[] for _ in range(n)]
        for i in range(1, n):
            children[par[i]].append(i)
        tokens = np.zeros(n, dtype=int)
        for u in range(n):
            toks = rng.permutation(V)[:len(children[u])]
            for c, t in zip(children[u], toks):
                tokens[c] = t
        lm = oracle.lmhead_margin(hidden, W, tokens, par, [0, n], tau=1.0)
        paths, _, bonus, npro = oracle.accept_path(par, lm["accept"], lm["row_argmax"], tokens, [0, n])
        lg = hidden @ W.T
        greedy, u = [0], 0
        while True:
            top = int(np.argmax(lg[u]))
            nxt = [c for c in children[u] if tokens[c] == top]
            if not nxt:
                break
            u = nxt[0]
            greedy.append(u)
        assert paths[0] == greedy
        assert npro[0] == 0
        assert bonus[0] == int(np.argmax(lg[greedy[-1]]))


@pytest.mark.parametrize("triplet", ["triplet_deep_narrow", "triplet_eagle3_static"])
def test_paper_chain_shapes_stop_at_first_rejection(triplet):
    """Chains of the paper's (nsteps, 1, ndt) configurations: the committed
    prefix ends right before the first rejected node."""
    nsteps, topk, ndt = GOLDEN[triplet]["value"]
    assert topk == 1 and ndt == nsteps + 1
    parent = synth.tree_chain(ndt)
    for first_rej in range(1, ndt + 1):
        acc = np.ones(ndt, int)
        if first_rej < ndt:
            acc[first_rej] = 0
            acc[first_rej + 1:] = np.random.default_rng(first_rej).integers(0, 2, ndt - first_rej - 1)
        p, L, _, _ = oracle.accept_path(parent, acc, np.zeros(ndt, int), np.zeros(ndt, int), [0, ndt])
        assert p[0] == list(range(first_rej)) and L[0] == first_rej


def test_multiple_sequences_independent():
    parent = np.array([-1, 0, 0, -1, 0, 1, 2])
    acc = np.array([1, 0, 1, 1, 1, 1, 1])
    p, L, _, _ = oracle.accept_path(parent, acc, np.zeros(7, int), np.zeros(7, int), [0, 3, 7])
    assert p == [[0, 2], [0, 1, 2, 3]]
    assert list(L) == [2, 4]
