"""Pins for the tree-shape policy oracle (Sec. 3.3, Eq. 2) against values the
paper fixes (its hyperparameters and triplet range, tests/golden/
paper_settings.json), closed forms and brute force."""
import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest

from oracle import policy as P

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_settings.json")))
SHALLOW = tuple(GOLD["triplet_shallow_wide"]["value"])
DEEP = tuple(GOLD["triplet_deep_narrow"]["value"])
D = GOLD["dcs_divisor_d"]["value"]
ALPHA = GOLD["rar_ema_alpha"]["value"]
BREAKER = GOLD["circuit_breaker_steps"]["value"]


def test_range_endpoints():
    """Score 0 gives the wide shallow tree, score 1 the deep chain (Sec. 3.3)."""
    assert P.triplet(0.0, SHALLOW, DEEP) == (3, 4, 4)
    assert P.triplet(1.0, SHALLOW, DEEP) == (7, 1, 8)


def _hand_chain():
    """The paper's range worked by hand with exact fractions: n_steps = 3 + 4s
    and ndt = 4 + 4s change at s = 1/8, 3/8, 5/8, 7/8; topk = 1 + 3(1 - s)
    changes at 1 - s = 1/6, 1/2, 5/6, i.e. s = 1/6, 1/2, 5/6 (half up keeps
    the larger value at the breakpoint itself)."""
    cuts = sorted([Fraction(1, 8), Fraction(3, 8), Fraction(5, 8), Fraction(7, 8),
                   Fraction(1, 6), Fraction(1, 2), Fraction(5, 6)])
    chain = [(3, 4, 4), (4, 4, 5), (4, 3, 5), (5, 3, 6), (5, 2, 6), (6, 2, 7), (6, 1, 7),
             (7, 1, 8)]
    return cuts, chain


def test_hand_worked_chain():
    cuts, chain = _hand_chain()
    assert P.reachable_triplets(SHALLOW, DEEP) == chain
    edges = [Fraction(0)] + cuts + [Fraction(1)]
    for k in range(len(chain)):
        mid = float((edges[k] + edges[k + 1]) / 2)
        assert P.triplet(mid, SHALLOW, DEEP) == chain[k], (mid, k)
    # at a breakpoint of n_steps, 3 + 4 * (1/8) = 3.5 rounds up
    assert P.triplet(0.125, SHALLOW, DEEP)[0] == 4
    # at s = 1/2, topk = 1 + 3 * 0.5 = 2.5 rounds up to 3
    assert P.triplet(0.5, SHALLOW, DEEP) == (5, 3, 6)


def _ulp_walk(x, n):
    """The doubles from n steps below x to n steps above it."""
    out, lo, hi = [x], x, x
    for _ in range(n):
        lo, hi = np.nextafter(lo, -1.0), np.nextafter(hi, 2.0)
        out += [float(lo), float(hi)]
    return out


@pytest.mark.parametrize("shallow,deep", [((3, 4, 4), (7, 1, 8)), ((2, 6, 3), (9, 1, 16)),
                                          ((7, 1, 8), (3, 4, 4)), ((3, 1, 4), (3, 1, 4)),
                                          ((4, 8, 10), (6, 2, 10)), ((1, 9, 2), (12, 1, 13))])
def test_reachable_triplets_brute_force(shallow, deep):
    """A dense grid plus every double within 2000 ulps of each mathematical
    breakpoint (where lo + (hi - lo) t is an odd multiple of 1/2, worked with
    exact fractions) sees exactly the listed triplets, in order."""
    pts = set(float(x) for x in np.linspace(0.0, 1.0, 20001))
    for lo, hi, flip in ((shallow[0], deep[0], 0), (deep[1], shallow[1], 1),
                         (shallow[2], deep[2], 0)):
        for j in range(min(lo, hi), max(lo, hi)):
            t = Fraction(2 * j + 1 - 2 * lo, 2 * (hi - lo))
            pts.update(_ulp_walk(float(1 - t if flip else t), 2000))
    seen = []
    for s in sorted(x for x in pts if 0.0 <= x <= 1.0):
        t = P.triplet(s, shallow, deep)
        if not seen or seen[-1] != t:
            seen.append(t)
    assert P.reachable_triplets(shallow, deep) == seen


def test_coincident_breakpoints_give_single_score_triplets():
    """(4,8,10) -> (6,2,10): n_steps = 4 + 2s and topk = 2 + 6(1 - s) both
    sit on a half at s = 3/4, where half up takes n_steps up to 6 and keeps
    topk at 4 for that one score."""
    assert P.triplet(0.75, (4, 8, 10), (6, 2, 10)) == (6, 4, 10)
    assert (6, 4, 10) in P.reachable_triplets((4, 8, 10), (6, 2, 10))
    assert P.triplet(float(np.nextafter(0.75, 0)), (4, 8, 10), (6, 2, 10)) == (5, 4, 10)
    assert P.triplet(float(np.nextafter(0.75, 1)), (4, 8, 10), (6, 2, 10)) == (6, 3, 10)


def test_ndt_is_one_more_than_depth_on_the_paper_range():
    """Both interpolants move by 4 over the range and start one apart."""
    for s in np.linspace(0, 1, 10001):
        n, _, ndt = P.triplet(float(s), SHALLOW, DEEP)
        assert ndt == n + 1


def test_dcs_saturation_and_scaling():
    assert P.dcs(0.5, 1.0, D) == 1.0                 # p * RAR reaches d
    assert P.dcs(0.9, 0.8, D) == 1.0
    assert P.dcs(0.25, 1.0, D) == 0.5                # half of d
    assert P.dcs(0.0, 1.0, D) == 0.0
    assert P.dcs(0.2, 0.5, D) == pytest.approx(0.2)
    # monotone in both factors, and a smaller divisor saturates sooner
    ps = np.linspace(0, 1, 101)
    for r in (0.1, 0.5, 1.0):
        v = [P.dcs(p, r, D) for p in ps]
        assert all(a <= b for a, b in zip(v, v[1:]))
    assert P.dcs(0.3, 0.8, 0.2) == 1.0 and P.dcs(0.3, 0.8, 0.5) < 1.0


def test_p_top1_closed_form():
    logits = np.array([2.0, 1.0, 0.0, 0.5])
    m = logits.max()
    lse = m + math.log(np.exp(logits - m).sum())
    assert P.p_top1(m, lse) == pytest.approx(math.exp(2) / np.exp(logits).sum(), rel=1e-14)
    assert P.p_top1(3.0, 3.0 + math.log(8)) == pytest.approx(1 / 8, rel=1e-14)   # 8 equal logits


def test_ema_closed_form():
    """A constant fraction a for t steps: RAR_t = a + (1 - alpha)^t (RAR_0 - a)."""
    for a_num, n in ((3, 7), (0, 3), (2, 5), (6, 7)):
        st = P.initial_state(1.0)
        a = a_num / (n - 1) if n > 1 else 0.0
        for t in range(1, 30):
            P.update(st, n, a_num + 1, ALPHA, 10**9)
            assert st["rar"] == pytest.approx(a + (1 - ALPHA) ** t * (1.0 - a), abs=1e-14)


def test_acceptance_fraction_on_the_paper_trees():
    """(7,1,8) chain: k accepted of 7 drafted; (3,4,4): k of 3."""
    for n, k in ((8, 0), (8, 3), (8, 7), (4, 2)):
        st = P.initial_state(0.0)
        P.update(st, n, k + 1, 1.0, 10**9)          # alpha = 1 keeps the newest fraction
        assert st["rar"] == k / (n - 1)


def test_circuit_breaker():
    st = P.initial_state(1.0)
    for step in range(BREAKER - 1):
        P.update(st, 8, 1, ALPHA, BREAKER)
        assert st["zero_streak"] == step + 1 and st["breaks"] == 0
    assert st["rar"] == pytest.approx((1 - ALPHA) ** (BREAKER - 1))
    P.update(st, 8, 1, ALPHA, BREAKER)               # the fifth zero-accept step
    assert st == dict(rar=1.0, zero_streak=0, breaks=1)
    # four zero-accept steps, one accept, four more: no reset
    st = P.initial_state(1.0)
    for pl in [1] * 4 + [3] + [1] * 4:
        P.update(st, 8, pl, ALPHA, BREAKER)
    assert st["breaks"] == 0 and st["zero_streak"] == 4


def test_steps_without_drafts_or_with_errors_leave_the_state():
    st = P.initial_state(1.0)
    P.update(st, 8, 3, ALPHA, BREAKER)
    before = dict(st)
    P.update(st, 1, 1, ALPHA, BREAKER)               # only the root verified
    P.update(st, 8, 0, ALPHA, BREAKER)               # malformed sequence
    assert st == before


def test_select_goes_shallow_as_acceptance_collapses():
    """A confident draft with full acceptance keeps the chain; repeated
    rejections shrink RAR and the policy moves to the wide tree, until the
    breaker restores the starting state (Sec. 3.3)."""
    st = P.initial_state(1.0)
    assert P.select(st, 0.9, D, SHALLOW, DEEP) == (1.0, DEEP)
    shapes = []
    for _ in range(BREAKER - 1):
        P.update(st, 8, 1, ALPHA, BREAKER)
        shapes.append(P.select(st, 0.9, D, SHALLOW, DEEP)[1])
    assert shapes[-1] != DEEP and shapes[-1][1] > 1
    assert all(a[0] >= b[0] for a, b in zip(shapes, shapes[1:]))
    P.update(st, 8, 1, ALPHA, BREAKER)
    assert P.select(st, 0.9, D, SHALLOW, DEEP)[1] == DEEP
