"""Oracle for the LM head and the margin rule (Sec. 3.2, Eq. 1).

logits[i, v] = sum_k hidden[i, k] * W[v, k]          (W is [vocab, hidden])
row_max[i]    = max_v logits[i, v]
row_argmax[i] = smallest v attaining row_max[i]
row_lse[i]    = row_max[i] + log(sum_v exp(logits[i, v] - row_max[i]))

For every non-root node c with parent p, the drafted token is tokens[c] and the
target distribution that judges it is row p.  Eq. 1 defines
  margin(c) = p_target(draft) / p_target(top1) = exp(l_draft - row_max[p]),
since both probabilities share the softmax denominator.  The node is accepted
when its token is the target's top-1 (strict match) or margin >= kappa (the
threshold rule right after Eq. 1; kappa is called tau in this library).
"""
import numpy as np

_VOCAB_BLOCK = 8192


def logits_rows(hidden, W, rows):
    """float64 logits of the listed rows against the full vocabulary."""
    h = np.asarray(hidden, dtype=np.float64)[np.asarray(rows, dtype=np.int64)]
    V = W.shape[0]
    out = np.empty((h.shape[0], V))
    for v0 in range(0, V, _VOCAB_BLOCK):  # pieces of one matmul, to bound memory
        v1 = min(V, v0 + _VOCAB_BLOCK)
        out[:, v0:v1] = h @ np.asarray(W[v0:v1], dtype=np.float64).T
    return out


def row_stats(logits):
    """(max, lowest-index argmax, log-sum-exp) of each row."""
    m = logits.max(axis=1)
    a = np.argmax(logits, axis=1)          # numpy returns the first maximum
    lse = m + np.log(np.exp(logits - m[:, None]).sum(axis=1))
    return m, a, lse


def topk_tokens(hidden, W, rows, k=5):
    """Token ids of the k largest logits of each listed row, largest first
    (equal logits ordered by token id)."""
    lg = logits_rows(hidden, W, rows)
    out = np.empty((len(rows), k), dtype=np.int64)
    kk = min(k, lg.shape[1])
    for r in range(len(rows)):
        kth = np.partition(lg[r], lg.shape[1] - kk)[lg.shape[1] - kk]
        cand = np.nonzero(lg[r] >= kth)[0]          # every id tied with the k-th value too
        order = cand[np.lexsort((cand, -lg[r, cand]))]
        out[r, :kk] = order[:kk]
    return out


def lmhead_margin(hidden, W, tokens, parent, cu_nodes, tau, rows=None):
    """Per-node outputs of the margin rule.

    Returns a dict of float64/int arrays of length T: row_max, row_argmax,
    row_lse, l_draft, ratio, accept.  Roots get accept = 1 and NaN l_draft /
    ratio.  With `rows` given, only the listed rows are evaluated, together
    with every child whose parent row is listed (others hold NaN / -1).
    """
    T = int(cu_nodes[-1])
    gp = np.asarray(parent, dtype=np.int64).copy()
    for b in range(len(cu_nodes) - 1):
        s, e = int(cu_nodes[b]), int(cu_nodes[b + 1])
        seg = gp[s:e]
        seg[seg >= 0] += s
    rows = np.arange(T) if rows is None else np.asarray(sorted(set(int(r) for r in rows)))
    lg = logits_rows(hidden, W, rows)
    m, a, lse = row_stats(lg)
    row_max = np.full(T, np.nan)
    row_argmax = np.full(T, -1, dtype=np.int64)
    row_lse = np.full(T, np.nan)
    row_max[rows], row_argmax[rows], row_lse[rows] = m, a, lse
    where = {int(r): j for j, r in enumerate(rows)}
    l_draft = np.full(T, np.nan)
    ratio = np.full(T, np.nan)
    accept = np.full(T, -1, dtype=np.int64)
    for c in range(T):
        p = int(gp[c])
        if p < 0:
            if c in where:
                accept[c] = 1
            continue
        if p not in where:
            continue
        ld = lg[where[p], int(tokens[c])]
        l_draft[c] = ld
        ratio[c] = np.exp(ld - row_max[p])
        strict = int(tokens[c]) == int(row_argmax[p])
        accept[c] = 1 if (strict or ratio[c] >= tau) else 0
    return dict(row_max=row_max, row_argmax=row_argmax, row_lse=row_lse,
                l_draft=l_draft, ratio=ratio, accept=accept)
