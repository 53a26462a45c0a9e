"""Oracle for choosing the accepted path (Sec. 3.2; Fig. 1 caption).

The verifier commits the drafted tokens along one root-to-node path of the
tree whose every non-root node is accepted (strict match or promoted by the
margin rule).  The root (node 0) is the last committed token and is always on
the path; the bonus token is the target's top-1 at the last node.

The paper states the margin rule "at the first mismatch position" of a
verification walk and says nothing about trees with several candidate
children or what happens after a promotion.  Four readings (`rule`):

  0  longest: the longest root-to-node path of accepted nodes; among equally
     long paths the lexicographically smallest node-index sequence;
  1  once: as 0, over the paths holding at most one promoted node (accepted
     but not a strict match of the parent row's top-1);
  2  greedy: walk from the root; at node u take a strict child if there is
     one (lowest index), else the accepted child with the largest ratio
     (lowest index on ties), else stop;
  3  greedy-once: as 2, but once a child has been promoted only strict
     children may follow.

Rules 0 and 1 enumerate every root-to-node path literally; rules 2 and 3 run
the walk node by node.
"""
import numpy as np


def _root_path(parent_local, u):
    path = []
    while u >= 0:
        path.append(u)
        u = int(parent_local[u])
    return path[::-1]


def _strict(tokens, row_argmax, s, par, v):
    return int(tokens[s + v]) == int(row_argmax[s + par[v]])


def accept_path(parent, accept, row_argmax, tokens, cu_nodes, max_path=None, rule=0,
                ratio=None):
    """Returns (paths, path_len, bonus, n_promoted).

    paths: list of local-id lists (root first); path_len includes the root;
    n_promoted counts path nodes accepted by the margin rule but not a strict
    match of the parent row's top-1.  `ratio` (per node, Eq. 1) is needed by
    the greedy rules 2 and 3 only.
    """
    if rule not in (0, 1, 2, 3):
        raise ValueError("rule must be 0, 1, 2 or 3")
    if rule >= 2 and ratio is None:
        raise ValueError("the greedy rules need the ratios")
    B = len(cu_nodes) - 1
    paths, plen, bonus, npro = [], [], [], []
    for b in range(B):
        s, e = int(cu_nodes[b]), int(cu_nodes[b + 1])
        par = [int(x) for x in parent[s:e]]
        acc = [int(x) for x in accept[s:e]]
        if rule <= 1:
            candidates = []
            for u in range(e - s):
                p = _root_path(par, u)
                if not all(acc[v] == 1 for v in p[1:]):
                    continue
                promoted = sum(1 for v in p[1:] if not _strict(tokens, row_argmax, s, par, v))
                if rule == 1 and promoted > 1:
                    continue
                candidates.append(p)
            L = max(len(p) for p in candidates)
            best = min(p for p in candidates if len(p) == L)
        else:
            best, u, used = [0], 0, 0
            while True:
                kids = [c for c in range(e - s) if par[c] == u and acc[c] == 1]
                strict = [c for c in kids if _strict(tokens, row_argmax, s, par, c)]
                if strict:
                    u = min(strict)
                elif kids and not (rule == 3 and used):
                    top = max(float(ratio[s + c]) for c in kids)
                    u = min(c for c in kids if float(ratio[s + c]) == top)
                    used += 1
                else:
                    break
                best.append(u)
        paths.append(best)
        plen.append(len(best))
        bonus.append(int(row_argmax[s + best[-1]]))
        npro.append(sum(1 for v in best[1:] if not _strict(tokens, row_argmax, s, par, v)))
    return paths, np.array(plen), np.array(bonus), np.array(npro)
