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


# ------------------------------------------------ readings of "first mismatch"

def _arrays(parent, accept, strict):
    """tokens / row_argmax realising a strict-match mask: every row's top-1 is
    token 0, a strict child drafts 0, any other child drafts 1."""
    n = len(parent)
    row_argmax = np.zeros(n, np.int64)
    tokens = np.array([0 if (i == 0 or strict[i]) else 1 for i in range(n)])
    return (np.array(parent), np.array(accept), row_argmax, tokens, np.array([0, n]))


def _budget_best(parent, accept, strict, budget):
    """Best path below u with at most `budget` promoted nodes, by recursion:
    u followed by the best (longest, then smallest) path of an accepted child,
    a promoted child spending one unit of budget."""
    n = len(parent)
    children = [[] for _ in range(n)]
    for i in range(1, n):
        children[parent[i]].append(i)

    def best(u, k):
        cand = []
        for c in children[u]:
            if not accept[c]:
                continue
            if strict[c]:
                cand.append(best(c, k))
            elif k > 0:
                cand.append(best(c, k - 1))
        if not cand:
            return [u]
        L = max(len(x) for x in cand)
        return [u] + min(x for x in cand if len(x) == L)
    return best(0, budget)


@pytest.mark.parametrize("n", [2, 3, 4, 5])
def test_once_rule_matches_budgeted_recursion(n):
    for parent in _all_trees(n):
        for acc_bits in itertools.product([0, 1], repeat=n - 1):
            accept = [1] + list(acc_bits)
            accepted = [i for i in range(1, n) if accept[i]]
            for st_bits in itertools.product([0, 1], repeat=len(accepted)):
                strict = [1] * n
                for i, b in zip(accepted, st_bits):
                    strict[i] = b
                args = _arrays(parent, accept, strict)
                paths, plen, _, npro = oracle.accept_path(*args, rule=1)
                assert paths[0] == _budget_best(parent, accept, strict, 1), (parent, accept, strict)
                assert npro[0] <= 1


@pytest.mark.parametrize("n", [2, 4, 7])
def test_greedy_rules_reduce_on_chains(n):
    """A chain offers one child per node: the greedy walk is the longest
    accepted prefix and the single-promotion walk the 'once' path."""
    parent = [-1] + list(range(n - 1))
    ratio = np.linspace(0.9, 0.3, n)
    for acc_bits in itertools.product([0, 1], repeat=n - 1):
        accept = [1] + list(acc_bits)
        for st_bits in itertools.product([0, 1], repeat=n - 1):
            strict = [1] + [a and s for a, s in zip(acc_bits, st_bits)]
            args = _arrays(parent, accept, strict)
            r = {k: oracle.accept_path(*args, rule=k, ratio=ratio)[0][0] for k in range(4)}
            assert r[2] == r[0] and r[3] == r[1]


def test_rules_agree_without_promotions():
    """When every accepted node is a strict match (kappa = 1, distinct sibling
    tokens), all four readings give the classic greedy strict walk."""
    rng = np.random.default_rng(4)
    for _ in range(200):
        n = int(rng.integers(1, 40))
        parent = synth.tree_grown(rng, n, int(rng.integers(1, 8)), int(rng.integers(1, 5)))
        n = len(parent)
        strict = [1] + [int(x) for x in rng.integers(0, 2, n - 1)]
        # distinct siblings: at most one strict child per node
        seen = set()
        for i in range(1, n):
            if strict[i] and parent[i] in seen:
                strict[i] = 0
            elif strict[i]:
                seen.add(parent[i])
        args = _arrays(list(parent), strict, strict)
        ratio = rng.random(n)
        r = [oracle.accept_path(*args, rule=k, ratio=ratio)[0][0] for k in range(4)]
        assert r[0] == r[1] == r[2] == r[3]


def test_rule_containments():
    """Rule 2's path is a candidate of rule 0 and rule 3's of rule 1, so they are
    never longer; rules 1 and 3 promote at most once."""
    rng = np.random.default_rng(9)
    for _ in range(300):
        n = int(rng.integers(2, 30))
        parent = list(synth.tree_grown(rng, n, int(rng.integers(1, 7)), int(rng.integers(1, 5))))
        n = len(parent)
        accept = [1] + [int(x) for x in rng.random(n - 1) < 0.7]
        strict = [1] + [int(a and r < 0.5) for a, r in zip(accept[1:], rng.random(n - 1))]
        args = _arrays(parent, accept, strict)
        ratio = rng.random(n)
        out = [oracle.accept_path(*args, rule=k, ratio=ratio) for k in range(4)]
        L = [o[1][0] for o in out]
        assert L[2] <= L[0] and L[3] <= L[1] <= L[0] and L[3] <= L[2]
        assert out[1][3][0] <= 1 and out[3][3][0] <= 1


def test_greedy_rules_hand_worked():
    """Root with two promoted children (1: ratio 0.5, 2: ratio 0.9); node 1 has a
    strict child 3, node 3 a promoted child 4; node 2 has no child.
      longest      0-1-3-4   (length 4, two promotions)
      once         0-1-3     (one promotion allowed: 4 would be the second)
      greedy       0-2       (no strict child of the root; 2 has the larger ratio)
      greedy-once  0-2
    With node 2 rejected the greedy walks take 1, then the strict 3; greedy
    goes on to promote 4, greedy-once stops."""
    parent = [-1, 0, 0, 1, 3]
    accept = [1, 1, 1, 1, 1]
    strict = [1, 0, 0, 1, 0]
    ratio = np.array([np.nan, 0.5, 0.9, 1.0, 0.4])
    args = _arrays(parent, accept, strict)
    got = [oracle.accept_path(*args, rule=k, ratio=ratio) for k in range(4)]
    assert [g[0][0] for g in got] == [[0, 1, 3, 4], [0, 1, 3], [0, 2], [0, 2]]
    assert [int(g[3][0]) for g in got] == [2, 1, 1, 1]
    args = _arrays(parent, [1, 1, 0, 1, 1], strict)
    got = [oracle.accept_path(*args, rule=k, ratio=ratio)[0][0] for k in range(4)]
    assert got == [[0, 1, 3, 4], [0, 1, 3], [0, 1, 3, 4], [0, 1, 3]]


def test_greedy_ties_take_the_lowest_index():
    parent = [-1, 0, 0, 0]
    args = _arrays(parent, [1, 1, 1, 1], [1, 0, 0, 0])
    ratio = np.array([np.nan, 0.3, 0.7, 0.7])
    assert oracle.accept_path(*args, rule=2, ratio=ratio)[0][0] == [0, 2]
    args = _arrays(parent, [1, 1, 1, 1], [1, 0, 1, 1])
    assert oracle.accept_path(*args, rule=2, ratio=ratio)[0][0] == [0, 2]
