"""Pins for the tree-attention oracle against routines it does not share code
with: torch's scaled_dot_product_attention (causal, masked and unmasked), a
boolean transitive closure for the ancestor set, and scalar brute force."""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle
from paper_2609_02897_gb300 import synth


def _rand(rng, *shape):
    return rng.standard_normal(shape)


def _sdpa(q, k, v, mask=None, causal=False):
    """q [L,H,D], k/v [S,H,D] in float64 via torch."""
    qt = torch.from_numpy(q).permute(1, 0, 2)[None]
    kt = torch.from_numpy(k).permute(1, 0, 2)[None]
    vt = torch.from_numpy(v).permute(1, 0, 2)[None]
    m = None if mask is None else torch.from_numpy(mask)
    o = F.scaled_dot_product_attention(qt, kt, vt, attn_mask=m, is_causal=causal)
    return o[0].permute(1, 0, 2).numpy()


def _expand_kv(x, G):
    return np.repeat(x, G, axis=1)   # head h uses KV head h // G


def _case(rng, parent, ctx, Hq=4, Hkv=2, D=16):
    N = len(parent)
    q = _rand(rng, N, Hq, D)
    tk, tv = _rand(rng, N, Hkv, D), _rand(rng, N, Hkv, D)
    ctx_max = ctx + 4
    kc, vc = _rand(rng, 1, Hkv, ctx_max, D), _rand(rng, 1, Hkv, ctx_max, D)
    return q, tk, tv, kc, vc


def test_chain_tree_equals_causal_attention():
    rng = np.random.default_rng(1)
    N, ctx, Hq, Hkv = 6, 9, 4, 2
    parent = synth.tree_chain(N)
    q, tk, tv, kc, vc = _case(rng, parent, ctx, Hq, Hkv)
    got = oracle.tree_attention(q, kc, vc, [ctx], tk, tv, parent, [0, N])
    # causal attention of the last N positions of the sequence [context; chain]
    K = np.concatenate([kc[0, :, :ctx].transpose(1, 0, 2), tk])
    V = np.concatenate([vc[0, :, :ctx].transpose(1, 0, 2), tv])
    mask = np.arange(ctx + N)[None, :] <= (ctx + np.arange(N))[:, None]
    ref = _sdpa(q, _expand_kv(K, Hq // Hkv), _expand_kv(V, Hq // Hkv), mask)
    np.testing.assert_allclose(got, ref, rtol=1e-12, atol=1e-12)


def test_chain_without_context_is_causal_self_attention():
    rng = np.random.default_rng(2)
    N, Hq, Hkv = 7, 4, 4
    parent = synth.tree_chain(N)
    q, tk, tv, kc, vc = _case(rng, parent, 0, Hq, Hkv)
    got = oracle.tree_attention(q, kc, vc, [0], tk, tv, parent, [0, N])
    ref = _sdpa(q, tk, tv, causal=True)
    np.testing.assert_allclose(got, ref, rtol=1e-12, atol=1e-12)


def test_single_node_tree_is_plain_decode_attention():
    rng = np.random.default_rng(3)
    ctx, Hq, Hkv = 33, 8, 2
    parent = np.array([-1], dtype=np.int32)
    q, tk, tv, kc, vc = _case(rng, parent, ctx, Hq, Hkv)
    got = oracle.tree_attention(q, kc, vc, [ctx], tk, tv, parent, [0, 1])
    K = np.concatenate([kc[0, :, :ctx].transpose(1, 0, 2), tk])
    V = np.concatenate([vc[0, :, :ctx].transpose(1, 0, 2), tv])
    ref = _sdpa(q, _expand_kv(K, 4), _expand_kv(V, 4))
    np.testing.assert_allclose(got, ref, rtol=1e-12, atol=1e-12)


def _closure(parent):
    """anc[i, j] = j is i or an ancestor of i, via powers of the adjacency."""
    n = len(parent)
    A = np.zeros((n, n), dtype=np.int64)
    for i in range(1, n):
        A[i, parent[i]] = 1
    R = np.eye(n, dtype=np.int64)
    P = np.eye(n, dtype=np.int64)
    for _ in range(n):
        P = (P @ A > 0).astype(np.int64)
        R = ((R + P) > 0).astype(np.int64)
    return R.astype(bool)


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_branched_tree_matches_masked_sdpa(seed):
    rng = np.random.default_rng(10 + seed)
    parent = synth.random_topological_relabel(
        synth.tree_grown(np.random.default_rng(seed), 14, 4, 3), rng)
    N, ctx, Hq, Hkv = len(parent), 11, 6, 3
    q, tk, tv, kc, vc = _case(rng, parent, ctx, Hq, Hkv)
    got = oracle.tree_attention(q, kc, vc, [ctx], tk, tv, parent, [0, N])
    K = np.concatenate([kc[0, :, :ctx].transpose(1, 0, 2), tk])
    V = np.concatenate([vc[0, :, :ctx].transpose(1, 0, 2), tv])
    mask = np.concatenate([np.ones((N, ctx), dtype=bool), _closure(parent)], axis=1)
    ref = _sdpa(q, _expand_kv(K, 2), _expand_kv(V, 2), mask)
    np.testing.assert_allclose(got, ref, rtol=1e-12, atol=1e-12)


def test_paged_layout_matches_contiguous():
    rng = np.random.default_rng(5)
    B, Hkv, D, ps = 3, 2, 8, 4
    ctx = np.array([9, 16, 3])
    ctx_max = 20
    parents = [synth.tree_chain(3), np.array([-1, 0, 0, 1]), np.array([-1])]
    cu = np.array([0, 3, 7, 8])
    T = 8
    q = _rand(rng, T, 4, D)
    tk, tv = _rand(rng, T, Hkv, D), _rand(rng, T, Hkv, D)
    kc, vc = _rand(rng, B, Hkv, ctx_max, D), _rand(rng, B, Hkv, ctx_max, D)
    parent = np.concatenate(parents)
    ref = oracle.tree_attention(q, kc, vc, ctx, tk, tv, parent, cu)
    # scatter the contiguous cache into a shuffled page pool
    pages = ctx_max // ps
    perm = rng.permutation(B * pages + 2)
    table = perm[:B * pages].reshape(B, pages)
    kp = np.full((B * pages + 2, Hkv, ps, D), np.nan)
    vp = np.full_like(kp, np.nan)
    for b in range(B):
        for s in range(ctx_max):
            kp[table[b, s // ps], :, s % ps] = kc[b, :, s]
            vp[table[b, s // ps], :, s % ps] = vc[b, :, s]
    got = oracle.tree_attention(q, kp, vp, ctx, tk, tv, parent, cu, table, ps)
    np.testing.assert_array_equal(got, ref)


def test_scalar_brute_force():
    """Scalar loops with math.exp on a tiny tree (no numpy arithmetic)."""
    rng = np.random.default_rng(6)
    parent = np.array([-1, 0, 0, 2, 1], dtype=np.int32)
    N, ctx, Hq, Hkv, D = 5, 3, 2, 1, 4
    q, tk, tv, kc, vc = _case(rng, parent, ctx, Hq, Hkv, D)
    got = oracle.tree_attention(q, kc, vc, [ctx], tk, tv, parent, [0, N])
    anc = {0: [0], 1: [0, 1], 2: [0, 2], 3: [0, 2, 3], 4: [0, 1, 4]}
    for i in range(N):
        keys = [list(kc[0, 0, j]) for j in range(ctx)] + [list(tk[a, 0]) for a in anc[i]]
        vals = [list(vc[0, 0, j]) for j in range(ctx)] + [list(tv[a, 0]) for a in anc[i]]
        for h in range(Hq):
            sc = [sum(q[i, h, d] * k[d] for d in range(D)) / math.sqrt(D) for k in keys]
            mx = max(sc)
            w = [math.exp(s - mx) for s in sc]
            z = sum(w)
            o = [sum(w[j] * vals[j][d] for j in range(len(keys))) / z for d in range(D)]
            np.testing.assert_allclose(got[i, h], o, rtol=1e-12, atol=1e-12)


def test_node_subset_leaves_other_rows_nan():
    rng = np.random.default_rng(7)
    parent = synth.tree_chain(4)
    q, tk, tv, kc, vc = _case(rng, parent, 5)
    full = oracle.tree_attention(q, kc, vc, [5], tk, tv, parent, [0, 4])
    part = oracle.tree_attention(q, kc, vc, [5], tk, tv, parent, [0, 4], nodes=[2])
    np.testing.assert_array_equal(part[2], full[2])
    assert np.isnan(part[[0, 1, 3]]).all()
