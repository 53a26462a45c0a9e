"""Oracle for choosing the accepted path (Sec. 3.2; Fig. 1 caption).

The verifier commits the drafted tokens along one root-to-node path of the
tree whose every non-root node is accepted (strict match or promoted by the
margin rule).  The committed path is the longest such path; among equally long
paths the one whose node-index sequence is lexicographically smallest wins.
The root (node 0) is the last committed token and is always on the path.

This oracle enumerates every root-to-node path literally and keeps the best.
The bonus token is the target's top-1 at the last node of the path.
"""
import numpy as np


def _root_path(parent_local, u):
    path = []
    while u >= 0:
        path.append(u)
        u = int(parent_local[u])
    return path[::-1]


def accept_path(parent, accept, row_argmax, tokens, cu_nodes, max_path=None):
    """Returns (paths, path_len, bonus, n_promoted).

    paths: list of local-id lists (root first); path_len includes the root;
    n_promoted counts path nodes accepted by the margin rule but not a strict
    match of the parent row's top-1.
    """
    B = len(cu_nodes) - 1
    paths, plen, bonus, npro = [], [], [], []
    for b in range(B):
        s, e = int(cu_nodes[b]), int(cu_nodes[b + 1])
        par = [int(x) for x in parent[s:e]]
        acc = [int(x) for x in accept[s:e]]
        candidates = []
        for u in range(e - s):
            p = _root_path(par, u)
            if all(acc[v] == 1 for v in p[1:]):
                candidates.append(p)
        L = max(len(p) for p in candidates)
        best = min(p for p in candidates if len(p) == L)
        paths.append(best)
        plen.append(L)
        bonus.append(int(row_argmax[s + best[-1]]))
        npro.append(sum(1 for v in best[1:]
                        if int(tokens[s + v]) != int(row_argmax[s + par[v]])))
    return paths, np.array(plen), np.array(bonus), np.array(npro)
