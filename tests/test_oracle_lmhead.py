"""Pins for the LM-head / margin-rule oracle (Eq. 1 and the kappa rule)."""
import json
import math
import os

import numpy as np
import pytest
import scipy.special
import torch

import oracle

GOLDEN = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_settings.json")))


def _tree_case(rng, V=37, K=11, parent=(-1, 0, 0, 1, 1, 2)):
    parent = np.array(parent, dtype=np.int32)
    T = len(parent)
    hidden = rng.standard_normal((T, K))
    W = rng.standard_normal((V, K))
    tokens = rng.integers(0, V, size=T)
    return hidden, W, tokens, parent, np.array([0, T])


def test_logits_and_row_stats_match_torch():
    rng = np.random.default_rng(0)
    hidden, W, tokens, parent, cu = _tree_case(rng)
    out = oracle.lmhead_margin(hidden, W, tokens, parent, cu, tau=0.3)
    lg = torch.from_numpy(hidden) @ torch.from_numpy(W).T
    np.testing.assert_allclose(oracle.logits_rows(hidden, W, range(6)), lg.numpy(), rtol=1e-13)
    np.testing.assert_allclose(out["row_max"], lg.max(dim=1).values.numpy(), rtol=1e-13)
    np.testing.assert_array_equal(out["row_argmax"], lg.argmax(dim=1).numpy())
    np.testing.assert_allclose(out["row_lse"], torch.logsumexp(lg, dim=1).numpy(), rtol=1e-13)


def test_equal_logits_closed_form():
    """All logits equal: lse = m + ln V and the lowest index is the argmax."""
    V, K = 50, 4
    hidden = np.ones((2, K))
    W = np.tile(np.array([[0.25, -0.5, 1.0, 2.0]]), (V, 1))
    out = oracle.lmhead_margin(hidden, W, np.array([3, 7]), np.array([-1, 0]), np.array([0, 2]), 0.5)
    m = 0.25 - 0.5 + 1.0 + 2.0
    np.testing.assert_allclose(out["row_max"], [m, m], rtol=1e-15)
    np.testing.assert_allclose(out["row_lse"], [m + math.log(V)] * 2, rtol=1e-15)
    assert list(out["row_argmax"]) == [0, 0]
    # token 7 ties the maximum: ratio 1, promoted by the margin rule (not strict)
    assert out["ratio"][1] == 1.0 and out["accept"][1] == 1


def test_argmax_ties_take_lowest_index():
    hidden = np.array([[1.0]])
    W = np.array([[0.0], [3.0], [1.0], [3.0], [-2.0]])
    out = oracle.lmhead_margin(hidden, W, np.array([0]), np.array([-1]), np.array([0, 1]), 1.0)
    assert out["row_argmax"][0] == 1


def test_eq1_ratio_is_probability_ratio():
    """Eq. 1: p_target(draft) / p_target(top1), evaluated with scipy's softmax."""
    rng = np.random.default_rng(1)
    hidden, W, tokens, parent, cu = _tree_case(rng)
    out = oracle.lmhead_margin(hidden, W, tokens, parent, cu, tau=0.3)
    probs = scipy.special.softmax(hidden @ W.T, axis=1)
    for c in range(1, len(parent)):
        p = parent[c]
        expect = probs[p, tokens[c]] / probs[p].max()
        np.testing.assert_allclose(out["ratio"][c], expect, rtol=1e-12)
        np.testing.assert_allclose(out["l_draft"][c], (hidden @ W.T)[p, tokens[c]], rtol=1e-13)
    assert out["accept"][0] == 1 and np.isnan(out["ratio"][0])


def test_ratio_range_and_unity_only_at_argmax():
    rng = np.random.default_rng(2)
    V = 23
    for trial in range(20):
        hidden, W, _, parent, cu = _tree_case(rng, V=V)
        toks = rng.integers(0, V, size=len(parent))
        out = oracle.lmhead_margin(hidden, W, toks, parent, cu, tau=0.5)
        r = out["ratio"][1:]
        assert np.all(r > 0) and np.all(r <= 1)
        for c in range(1, len(parent)):
            at_max = toks[c] == out["row_argmax"][parent[c]]
            assert (out["ratio"][c] == 1.0) == at_max


def test_tau_one_reduces_to_strict_match():
    rng = np.random.default_rng(3)
    for trial in range(20):
        hidden, W, tokens, parent, cu = _tree_case(rng, V=7)
        out = oracle.lmhead_margin(hidden, W, tokens, parent, cu, tau=1.0)
        strict = np.array([tokens[c] == out["row_argmax"][parent[c]] for c in range(1, len(parent))])
        np.testing.assert_array_equal(out["accept"][1:] == 1, strict)


def test_tau_below_every_ratio_accepts_all():
    rng = np.random.default_rng(4)
    hidden, W, tokens, parent, cu = _tree_case(rng)
    out = oracle.lmhead_margin(hidden, W, tokens, parent, cu, tau=1e-30)
    assert np.all(out["accept"] == 1)


def test_closed_form_margin_example():
    """Logits of the parent row are exactly [2, 1, 0, 0.5].  Drafting token 1
    gives margin e^-1 = 0.368: promoted at kappa 0.2 (the paper's setting) and
    0.3, rejected at 0.5.  Token 2 gives e^-2 = 0.135: rejected at 0.2.  Token
    3 gives e^-1.5 = 0.223: promoted at 0.2.  Token 0 is the strict match."""
    kappa = GOLDEN["kappa_main"]["value"]
    hidden = np.array([[1.0]] * 5)
    W = np.array([[2.0], [1.0], [0.0], [0.5]])
    parent = np.array([-1, 0, 0, 0, 0])
    tokens = np.array([0, 1, 2, 3, 0])
    cu = np.array([0, 5])
    out = oracle.lmhead_margin(hidden, W, tokens, parent, cu, tau=kappa)
    np.testing.assert_allclose(out["ratio"][1:], [math.exp(-1), math.exp(-2), math.exp(-1.5), 1.0],
                               rtol=1e-15)
    assert list(out["accept"]) == [1, 1, 0, 1, 1]
    assert list(oracle.lmhead_margin(hidden, W, tokens, parent, cu, 0.3)["accept"]) == [1, 1, 0, 0, 1]
    assert list(oracle.lmhead_margin(hidden, W, tokens, parent, cu, 0.5)["accept"]) == [1, 0, 0, 0, 1]


def test_children_judged_by_parent_row_not_own_row():
    """Two-level chain where the child's own row would give a different verdict."""
    hidden = np.array([[1.0, 0.0], [0.0, 1.0], [0.0, 0.0]])
    # row 0 logits: [5, 0, 0]; row 1 logits: [0, 5, 0]
    W = np.array([[5.0, 0.0], [0.0, 5.0], [0.0, 0.0]])
    parent = np.array([-1, 0, 1])
    tokens = np.array([2, 0, 1])   # node 1 drafts row-0 top1; node 2 drafts row-1 top1
    out = oracle.lmhead_margin(hidden, W, tokens, parent, np.array([0, 3]), tau=1.0)
    assert list(out["accept"]) == [1, 1, 1]
    tokens2 = np.array([2, 1, 0])  # swapped: each is the other row's top1
    out2 = oracle.lmhead_margin(hidden, W, tokens2, parent, np.array([0, 3]), tau=1.0)
    assert list(out2["accept"]) == [1, 0, 0]


def test_multi_sequence_offsets():
    rng = np.random.default_rng(5)
    V, K = 19, 5
    hidden = rng.standard_normal((7, K))
    W = rng.standard_normal((V, K))
    parent = np.array([-1, 0, 1, -1, 0, 0, 2])
    cu = np.array([0, 3, 7])
    tokens = rng.integers(0, V, size=7)
    out = oracle.lmhead_margin(hidden, W, tokens, parent, cu, tau=0.4)
    lg = hidden @ W.T
    # node 6 (local 3 of seq 1) has local parent 2 -> global 5
    np.testing.assert_allclose(out["l_draft"][6], lg[5, tokens[6]], rtol=1e-13)
    np.testing.assert_allclose(out["l_draft"][4], lg[3, tokens[4]], rtol=1e-13)


def test_row_subset_matches_full():
    rng = np.random.default_rng(6)
    hidden, W, tokens, parent, cu = _tree_case(rng)
    full = oracle.lmhead_margin(hidden, W, tokens, parent, cu, tau=0.3)
    part = oracle.lmhead_margin(hidden, W, tokens, parent, cu, tau=0.3, rows=[1])
    for c in (3, 4):    # children of node 1
        assert part["accept"][c] == full["accept"][c]
        np.testing.assert_allclose(part["l_draft"][c], full["l_draft"][c], rtol=1e-13)
    assert part["row_argmax"][1] == full["row_argmax"][1]


def test_topk_tokens_order():
    hidden = np.array([[1.0]])
    W = np.array([[0.1], [0.9], [0.5], [0.9], [0.7], [0.2]])
    assert list(oracle.topk_tokens(hidden, W, [0], k=5)[0]) == [1, 3, 4, 2, 5]
