"""Pins for the K/V commit oracle: invariants that hold for any copy."""
import numpy as np

import oracle


def test_contiguous_copy_invariants():
    rng = np.random.default_rng(0)
    B, Hkv, ctx_max, D = 2, 3, 12, 4
    kc, vc = rng.standard_normal((B, Hkv, ctx_max, D)), rng.standard_normal((B, Hkv, ctx_max, D))
    tk, tv = rng.standard_normal((9, Hkv, D)), rng.standard_normal((9, Hkv, D))
    cu = [0, 4, 9]
    ctx = np.array([5, 7])
    paths = [[0, 2, 3], [0, 4]]
    k2, v2, out = oracle.kv_compact(kc, vc, tk, tv, cu, paths, ctx)
    assert list(out) == [8, 9]
    touched = np.zeros((B, ctx_max), bool)
    for b, path in enumerate(paths):
        for k, u in enumerate(path):
            np.testing.assert_array_equal(k2[b, :, ctx[b] + k], tk[cu[b] + u])
            np.testing.assert_array_equal(v2[b, :, ctx[b] + k], tv[cu[b] + u])
            touched[b, ctx[b] + k] = True
    np.testing.assert_array_equal(k2.transpose(0, 2, 1, 3)[~touched], kc.transpose(0, 2, 1, 3)[~touched])
    np.testing.assert_array_equal(v2.transpose(0, 2, 1, 3)[~touched], vc.transpose(0, 2, 1, 3)[~touched])
    # inputs untouched
    assert not np.shares_memory(k2, kc)


def test_paged_equals_contiguous_through_page_table():
    rng = np.random.default_rng(1)
    B, Hkv, D, ps, pages = 2, 2, 3, 4, 5
    ctx_max = ps * pages
    kc, vc = rng.standard_normal((B, Hkv, ctx_max, D)), rng.standard_normal((B, Hkv, ctx_max, D))
    perm = rng.permutation(B * pages + 3)
    table = perm[:B * pages].reshape(B, pages)
    kp = rng.standard_normal((B * pages + 3, Hkv, ps, D))
    vp = rng.standard_normal((B * pages + 3, Hkv, ps, D))
    for b in range(B):
        for s in range(ctx_max):
            kp[table[b, s // ps], :, s % ps] = kc[b, :, s]
            vp[table[b, s // ps], :, s % ps] = vc[b, :, s]
    spare = perm[B * pages:]
    tk, tv = rng.standard_normal((6, Hkv, D)), rng.standard_normal((6, Hkv, D))
    cu = [0, 3, 6]
    ctx = np.array([3, 14])     # seq 0 crosses a page boundary at slot 4
    paths = [[0, 1, 2], [0, 2]]
    kc2, vc2, o1 = oracle.kv_compact(kc, vc, tk, tv, cu, paths, ctx)
    kp2, vp2, o2 = oracle.kv_compact(kp, vp, tk, tv, cu, paths, ctx, table, ps)
    np.testing.assert_array_equal(o1, o2)
    for b in range(B):
        for s in range(ctx_max):
            np.testing.assert_array_equal(kp2[table[b, s // ps], :, s % ps], kc2[b, :, s])
            np.testing.assert_array_equal(vp2[table[b, s // ps], :, s % ps], vc2[b, :, s])
    np.testing.assert_array_equal(kp2[spare], kp[spare])
