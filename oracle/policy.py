"""Oracle for the dynamic tree-shape policy (Sec. 3.3, Eq. 2): the Draft
Confidence Score, the running acceptance rate, the linear mapping of the
score onto the (n_steps, topk, ndt) range and the per-request circuit breaker.

TEST INFRASTRUCTURE ONLY (see oracle/__init__.py).  Plain Python floats
(IEEE binary64); every expression is written in the order given below and is
evaluated one rounded operation at a time, without fused multiply-adds.

Readings where the paper leaves the detail open:
  * the acceptance fraction of a step is the accepted drafted nodes (path
    length minus the root) over the drafted nodes verified (tree size minus
    the root); a step that verified no drafted node, or whose sequence was
    rejected as malformed (path length 0), leaves the state unchanged;
  * the EMA puts weight alpha on the newest fraction:
    RAR <- alpha * a + (1 - alpha) * RAR, starting from rar_init (1.0);
  * the DCS of a step uses the RAR after the previous step's update;
  * the score is saturated after the division by d: min(1, p * RAR / d);
  * each coordinate is interpolated on its own, n_steps and ndt linearly in
    DCS, topk linearly in 1 - DCS, and rounded to the nearest integer with
    halves upward: start + round(span * score), the product in binary64;
  * the circuit breaker counts consecutive steps with zero accepted drafted
    nodes; on the breaker-th one the request returns to its starting state
    (RAR = rar_init, count 0).
"""
import math
import struct


def p_top1(row_max, row_lse):
    """Top-1 softmax probability of a row from its max logit and
    log-sum-exp: exp(m - lse) (the denominators of Eq. 1 written out)."""
    return math.exp(float(row_max) - float(row_lse))


def dcs(p, rar, divisor):
    """Eq. 2 rescaled by the divisor d and saturated at 1 (Sec. 3.3)."""
    p = float(p)
    if not p >= 0.0:                     # a probability that is not a number counts as 0
        p = 0.0
    return min(1.0, (p * float(rar)) / float(divisor))


def round_half_up(y):
    """Nearest integer, halves upward, decided exactly: y - floor(y) is exact
    in binary64 for the magnitudes used here."""
    f = math.floor(y)
    return int(f) + (1 if y - f >= 0.5 else 0)


def _interp(a, b, u):
    """a + (b - a) * u rounded half up.  The product is the only rounded
    operation; the integer start is added after rounding, so two coordinates
    with the same span change value at the same score."""
    return int(a) + round_half_up(float(b - a) * u)


def triplet(score, shallow, deep):
    """(n_steps, topk, ndt) for a score in [0, 1]: depth and verify budget
    interpolate from the shallow-wide end (score 0) to the deep-narrow end
    (score 1) with the score, branching with 1 - score (Sec. 3.3)."""
    s = float(score)
    return (_interp(shallow[0], deep[0], s), _interp(deep[1], shallow[1], 1.0 - s),
            _interp(shallow[2], deep[2], s))


def _bits(x):
    return struct.unpack("<q", struct.pack("<d", x))[0]


def _from_bits(b):
    return struct.unpack("<d", struct.pack("<q", b))[0]


def reachable_triplets(shallow, deep):
    """Every triplet the mapping returns for some double score in [0, 1], in
    the order of increasing score (one CUDA graph per triplet, Sec. 3.3).

    Each coordinate, as evaluated in binary64, is a monotone step function of
    the score (every operation is a rounded monotone map), so it changes value
    at a handful of doubles.  Each such threshold is found by bisection over
    the bit patterns of the non-negative doubles (ordered like their values);
    between consecutive thresholds the triplet is constant, so evaluating it
    at every threshold, at the double just below it, and at 0 and 1 lists
    every triplet, including the ones that exist for a single score where two
    coordinates change at (nearly) the same place."""
    lo_b, hi_b = _bits(0.0), _bits(1.0)
    cands = {0.0, 1.0}
    for k in range(3):
        g = lambda b, k=k: triplet(_from_bits(b), shallow, deep)[k]  # noqa: E731
        g0, g1 = g(lo_b), g(hi_b)
        step = 1 if g1 > g0 else -1
        for v in range(g0, g1, step):
            # the smallest score whose coordinate has moved past v
            a, b = lo_b, hi_b                     # g(a) at v or before, g(b) past v
            while b - a > 1:
                m = (a + b) // 2
                if (g(m) - v) * step > 0:
                    b = m
                else:
                    a = m
            cands.add(_from_bits(b))
            cands.add(_from_bits(a))
    out = []
    for c in sorted(cands):
        t = triplet(c, shallow, deep)
        if not out or out[-1] != t:
            out.append(t)
    return out


def initial_state(rar_init=1.0):
    return dict(rar=float(rar_init), zero_streak=0, breaks=0)


def update(state, n_nodes, path_len, alpha, breaker, rar_init=1.0):
    """One verify step's effect on a request's policy state (Sec. 3.3):
    the EMA of the accepted fraction, then the circuit breaker."""
    n_nodes, path_len = int(n_nodes), int(path_len)
    if n_nodes <= 1 or path_len <= 0 or path_len > n_nodes:
        return state
    accepted = path_len - 1
    a = accepted / (n_nodes - 1)
    state["rar"] = alpha * a + (1.0 - alpha) * state["rar"]
    state["zero_streak"] = state["zero_streak"] + 1 if accepted == 0 else 0
    if state["zero_streak"] >= breaker:
        state["rar"] = float(rar_init)
        state["zero_streak"] = 0
        state["breaks"] += 1
    return state


def select(state, p, divisor, shallow, deep):
    """The step's score and triplet from the draft's top-1 probability and
    the request's RAR."""
    score = dcs(p, state["rar"], divisor)
    return score, triplet(score, shallow, deep)
