"""Checks of the seeded input generator (shapes, determinism, tree recipes)."""
import numpy as np
import pytest
import torch

from paper_2609_02897_gb300 import synth


def test_bf16_rounding_matches_torch():
    x = np.random.default_rng(0).standard_normal(100000).astype(np.float32) * 3
    x[:4] = [1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -1.5 - 2 ** -9, 0.0]   # ties and exact
    ref = torch.from_numpy(x).to(torch.bfloat16).float().numpy()
    np.testing.assert_array_equal(synth.round_bf16(x), ref)


def test_c1_tree_shape():
    assert list(synth.tree_fixed_c1()) == [-1, 0, 1, 2, 3, 0, 1, 2]


def _check_topo(p):
    assert p[0] == -1
    assert all(0 <= p[i] < i for i in range(1, len(p)))


def test_eagle_tree_recipe():
    rng = np.random.default_rng(3)
    for _ in range(5):
        p = synth.tree_eagle(rng, 8, 10, 60)
        _check_topo(p)
        assert len(p) == 60
        assert synth.depths(p).max() <= 8
        assert np.bincount(p[1:]).max() <= 10
        d = synth.depths(p)
        assert np.all(np.diff(d) >= 0)   # numbered by depth


def test_paper_trees():
    """The paper's (n_steps, top-k, ndt) shapes, ndt counting the root: the
    top-1 triplets are chains of ndt nodes; (3, 4, 4) keeps 4 nodes of a
    depth-3, 4-way expansion, ancestor-closed."""
    rng = np.random.default_rng(5)
    np.testing.assert_array_equal(synth.tree_eagle(rng, 7, 1, 8), [-1, 0, 1, 2, 3, 4, 5, 6])
    np.testing.assert_array_equal(synth.tree_eagle(rng, 3, 1, 4), [-1, 0, 1, 2])
    for _ in range(20):
        p = synth.tree_eagle(rng, 3, 4, 4)
        assert len(p) == 4 and p[0] == -1
        _check_topo(p)
        depth = [0] * 4
        for i in range(1, 4):
            depth[i] = depth[p[i]] + 1
        assert max(depth) <= 3
        assert max(np.bincount(p[1:], minlength=4)) <= 4
    for cfg, shape in ((6, (7, 1, 8)), (7, (3, 4, 4)), (8, (3, 1, 4))):
        assert synth.WORKLOADS[cfg]["tree"] == ("eagle",) + shape
        assert 0.2 in synth.WORKLOADS[cfg]["tau"]


def test_grown_tree_limits_and_spine():
    rng = np.random.default_rng(4)
    for n, dep, wid in [(64, 10, 10), (128, 12, 16), (96, 3, 1), (30, 5, 2)]:
        p = synth.tree_grown(rng, n, dep, wid)
        _check_topo(p)
        assert synth.depths(p).max() == min(dep, n - 1)
        assert np.bincount(p[1:], minlength=len(p)).max() <= wid
        cap = sum(wid ** k for k in range(dep + 1))
        assert len(p) == min(n, cap)


def test_relabel_keeps_topological_order():
    rng = np.random.default_rng(5)
    p = synth.tree_grown(rng, 40, 6, 4)
    q = synth.random_topological_relabel(p, rng)
    _check_topo(q)
    assert sorted(np.bincount(q[1:], minlength=40)) == sorted(np.bincount(p[1:], minlength=40))


@pytest.mark.parametrize("cfg", sorted(synth.WORKLOADS))
def test_small_workloads_deterministic_and_consistent(cfg):
    a = synth.make_workload(cfg, small=True)
    b = synth.make_workload(cfg, small=True)
    for f in ["q", "tree_k", "k_cache", "hidden", "w", "parent", "cu_nodes", "ctx_len"]:
        np.testing.assert_array_equal(getattr(a, f), getattr(b, f))
    assert a.cu_nodes[-1] == a.q.shape[0] == a.hidden.shape[0]
    assert a.ctx_len.max() + a.max_path <= a.ctx_max
    if a.dtype == "bf16":
        np.testing.assert_array_equal(synth.round_bf16(a.w), a.w)
    if a.page_size:
        flat = a.page_table.ravel()
        assert len(np.unique(flat)) == len(flat)
        assert flat.max() < a.k_cache.shape[0]


def test_token_mixture_distinct_siblings_and_rates():
    wl = synth.make_workload(3, small=True)
    rows = wl.parents_needed()
    V = wl.vocab
    ranks = {int(p): np.array([p % V, (p + 1) % V, (p + 2) % V, (p + 3) % V, (p + 4) % V]) for p in rows}
    toks = synth.attach_tokens(wl, ranks)
    gp = wl.global_parent()
    top1 = 0
    n = 0
    for p in rows:
        kids = np.where(gp == p)[0]
        assert len(set(toks[kids])) == len(kids)
        top1 += int(np.sum(toks[kids] == ranks[int(p)][0]))
        n += len(kids)
    assert 0.3 < top1 / n <= 0.6
    assert toks.min() >= 0 and toks.max() < V
