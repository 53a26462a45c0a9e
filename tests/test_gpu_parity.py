"""GPU parity of every libasd entry point against the fp64 oracle on reduced
workloads that span several tiles and ragged tails (all five workload
families, every tau of each), plus edge cases, error reporting, determinism
and CUDA-graph replay.  All calls go through the C ABI."""
import numpy as np
import pytest

import _helpers as H
from paper_2609_02897_gb300 import synth

pytestmark = pytest.mark.gpu

CASES = [(cfg, tau) for cfg in sorted(synth.WORKLOADS) for tau in synth.WORKLOADS[cfg]["tau"]]


@pytest.fixture(scope="module")
def dev():
    import torch
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    import _device
    return _device


def _written(wl, out):
    return [(b, int(wl.ctx_len[b]) + k) for b in range(wl.B) for k in range(int(out["path_len"][b]))]


@pytest.mark.parametrize("cfg,tau", CASES)
def test_verify_step_small(dev, cfg, tau):
    wl = H.prepared(cfg, small=True)
    out, status, _, _ = dev.run_verify(wl, tau)
    assert status == 0
    rep = H.compare_verify(wl, tau, out)
    H.untouched_cache_equal(wl, out, _written(wl, out))
    print(wl.name, tau, rep)
    assert rep.checked_seqs >= 1


@pytest.mark.parametrize("over", [dict(D=64), dict(page_size=32), dict(page_size=64),
                                  dict(page_size=8), dict(page_size=16, D=64),
                                  dict(page_size=256)])
def test_verify_variants(dev, over):
    cfg = 5 if "page_size" in over else 2
    wl = H.prepared(cfg, small=True, overrides=over)
    out, status, _, _ = dev.run_verify(wl, 0.3)
    assert status == 0
    H.compare_verify(wl, 0.3, out)
    H.untouched_cache_equal(wl, out, _written(wl, out))


def test_separate_calls_match_verify_step(dev):
    import torch
    from paper_2609_02897_gb300 import asd
    wl = H.prepared(3, small=True)
    tau = 0.5
    ref, status, _, _ = dev.run_verify(wl, tau)
    assert status == 0
    d = dev.to_device(wl)
    dims = dev.dims_of(wl)
    T, B = wl.T, wl.B
    ws = asd.alloc_workspace(dims, T)
    att = torch.empty(T, wl.Hq, wl.D, dtype=dev.dtype_of(wl), device="cuda")
    asd.asd_tree_attention(dims, d["q"], d["k_cache"], d["v_cache"], d["page_table"], d["ctx_len"],
                           d["tree_k"], d["tree_v"], d["parent"], d["cu_nodes"], att, ws)
    f = lambda: torch.empty(T, dtype=torch.float32, device="cuda")  # noqa: E731
    i = lambda n: torch.empty(n, dtype=torch.int32, device="cuda")  # noqa: E731
    rm, ra, rl, ld, rt = f(), i(T), f(), f(), f()
    acc = torch.empty(T, dtype=torch.uint8, device="cuda")
    asd.asd_lmhead_margin(dims, d["hidden"], d["w_lm"], d["tokens"], d["parent"], d["cu_nodes"], tau,
                          rm, ra, rl, ld, rt, acc, ws)
    path = torch.empty(B, dims.max_path, dtype=torch.int32, device="cuda")
    plen, bonus, npro, cout = i(B), i(B), i(B), i(B)
    asd.asd_accept_path(dims, d["parent"], d["tokens"], acc, ra, d["cu_nodes"], path, plen, bonus,
                        npro, ws)
    asd.asd_kv_compact(dims, d["tree_k"], d["tree_v"], d["cu_nodes"], T, path, plen, d["ctx_len"],
                       d["page_table"], d["k_cache"], d["v_cache"], cout, ws)
    torch.cuda.synchronize()
    assert asd.asd_get_device_status(ws) == 0
    np.testing.assert_array_equal(att.float().cpu().numpy(), ref["attn_out"])
    for name, t in [("row_max", rm), ("row_argmax", ra), ("row_lse", rl), ("ratio", rt),
                    ("accept", acc), ("path", path), ("path_len", plen), ("bonus", bonus),
                    ("n_promoted", npro), ("ctx_len_out", cout)]:
        np.testing.assert_array_equal(t.cpu().numpy(), ref[name], err_msg=name)
    np.testing.assert_array_equal(ld.cpu().numpy(), ref["l_draft"])
    np.testing.assert_array_equal(d["k_cache"].float().cpu().numpy(), ref["k_cache"])


@pytest.mark.parametrize("seed", [0, 1, 2, 3])
def test_random_trees_random_numbering(dev, seed):
    rng = np.random.default_rng(100 + seed)
    trees = []
    for b in range(4):
        t = synth.tree_grown(rng, int(rng.integers(2, 100)), int(rng.integers(1, 12)),
                             int(rng.integers(1, 8)))
        trees.append(synth.random_topological_relabel(t, rng))
    wl = H.prepared(3, small=True, rep=seed, tree_override=trees, overrides=dict(B=4))
    for tau in (1.0, 0.3, 0.05):
        out, status, _, _ = dev.run_verify(wl, tau)
        assert status == 0
        H.compare_verify(wl, tau, out)


def test_edge_shapes(dev):
    """Single-node trees, empty contexts, a 128-node chain (mask bits 64-127) and
    a 128-node star, in one ragged batch."""
    trees = [np.array([-1]), synth.tree_chain(128), np.array([-1] + [0] * 127), synth.tree_chain(2)]
    wl = synth.make_workload(3, small=True, tree_override=trees, overrides=dict(B=4, ctx=(0, 70)))
    wl.ctx_len[:] = [0, 70, 1, 0]
    synth.attach_tokens(wl, H.ranks_via_oracle(wl))
    for tau in (1.0, 0.5, 1e-30):
        out, status, _, _ = dev.run_verify(wl, tau)
        assert status == 0
        H.compare_verify(wl, tau, out)
        H.untouched_cache_equal(wl, out, _written(wl, out))


def test_duplicate_sibling_tokens(dev):
    """Siblings drafting the same token get the same logit and verdict; the
    walk breaks the tie between their equal-length paths by node index."""
    parent = np.array([-1, 0, 0, 1, 2, 0])
    wl = synth.make_workload(2, small=True, tree_override=[parent])
    synth.attach_tokens(wl, H.ranks_via_oracle(wl))
    wl.tokens[1] = wl.tokens[2] = wl.tokens[5]
    wl.tokens[3] = wl.tokens[4]
    for tau in (1.0, 1e-30):
        out, status, _, _ = dev.run_verify(wl, tau)
        assert status == 0
        H.compare_verify(wl, tau, out)
        assert out["l_draft"][1] == out["l_draft"][2] == out["l_draft"][5]
    assert list(out["path"][0][:3]) == [0, 1, 3]


def test_tau_one_is_strict_and_tiny_tau_accepts_all(dev):
    wl = H.prepared(2, small=True)
    out, _, _, _ = dev.run_verify(wl, 1.0)
    gp = wl.global_parent()
    for c in range(wl.T):
        if gp[c] >= 0:
            strict = wl.tokens[c] == out["row_argmax"][gp[c]]
            assert out["accept"][c] == (1 if strict else 0) or abs(out["ratio"][c] - 1) < 1e-3
    out, _, _, _ = dev.run_verify(wl, 1e-30)
    assert np.all(out["accept"] == 1)


def test_device_errors_are_reported(dev):
    import torch
    wl = H.prepared(3, small=True)
    base = dev.to_device(wl)
    # malformed parent in sequence 1: its path is empty and the cache untouched
    d = dict(base)
    par = wl.parent.copy()
    s1 = int(wl.cu_nodes[1])
    par[s1 + 2] = 5
    d["parent"] = torch.from_numpy(par.astype(np.int32)).cuda()
    kc0 = d["k_cache"].clone()
    out, status, _, _ = dev.run_verify(wl, 0.5, dev=d)
    assert status == 3                      # ASD_ERR_TREE
    assert out["path_len"][1] == 0
    assert out["path_len"][0] >= 1          # the other sequences still run
    b = 1
    np.testing.assert_array_equal(d["k_cache"][b].float().cpu().numpy(), kc0[b].float().cpu().numpy())
    # token out of range
    d = dict(base)
    tok = wl.tokens.copy()
    tok[int(wl.cu_nodes[2]) + 1] = wl.vocab + 7
    d["tokens"] = torch.from_numpy(tok.astype(np.int32)).cuda()
    out, status, _, _ = dev.run_verify(wl, 0.5, dev=d)
    assert status == 4                      # ASD_ERR_TOKEN_RANGE
    assert out["path_len"][2] == 0
    # context longer than the cache
    d = dict(base)
    cl = wl.ctx_len.copy()
    cl[0] = wl.ctx_max + 1
    d["ctx_len"] = torch.from_numpy(cl.astype(np.int32)).cuda()
    out, status, _, _ = dev.run_verify(wl, 0.5, dev=d)
    assert status == 5                      # ASD_ERR_CTX_RANGE
    assert out["path_len"][0] == 0


def test_page_id_out_of_range_is_reported(dev):
    import torch
    wl = H.prepared(5, small=True)
    d = dev.to_device(wl)
    pt = wl.page_table.copy()
    pt[3, 1] = wl.num_pages + 100
    d["page_table"] = torch.from_numpy(pt.astype(np.int32)).cuda()
    out, status, _, _ = dev.run_verify(wl, 0.3, dev=d)
    assert status == 5


def test_host_errors(dev):
    import torch
    from paper_2609_02897_gb300 import asd
    wl = H.prepared(2, small=True)
    d = dev.to_device(wl)
    dims = dev.dims_of(wl)
    step = asd.VerifyStep(dims, wl.T)
    with pytest.raises(asd.AsdError) as e:
        step.bind(tau=0.0, **d).run()
    assert e.value.code == 1
    with pytest.raises(asd.AsdError) as e:
        step.bind(tau=1.5, **d).run()
    assert e.value.code == 1
    small_ws = torch.empty(1024, dtype=torch.uint8, device="cuda")
    with pytest.raises(asd.AsdError) as e:
        asd.asd_verify_step(dims, step.bind(tau=0.3, **d).args, small_ws)
    assert e.value.code == 6
    bad = dev.dims_of(wl)
    bad.head_dim = 96
    with pytest.raises(asd.AsdError) as e:
        asd.asd_workspace_bytes(bad, wl.T)
    assert e.value.code == 2


def test_deterministic(dev):
    wl = H.prepared(5, small=True)
    a, _, _, _ = dev.run_verify(wl, 0.3)
    b, _, _, _ = dev.run_verify(wl, 0.3)
    for k in a:
        np.testing.assert_array_equal(a[k], b[k], err_msg=k)


def test_cuda_graph_replay_matches_eager(dev):
    import torch
    from paper_2609_02897_gb300 import asd
    wl = H.prepared(4, small=True)
    eager, _, _, _ = dev.run_verify(wl, 0.3)
    d = dev.to_device(wl)
    step = asd.VerifyStep(dev.dims_of(wl), wl.T)
    step.bind(tau=0.3, **d)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        step.run(s)   # warm-up (sets kernel attributes outside the capture)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        step.run(s)
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    for k, v in step.out.items():
        got = v.float().cpu().numpy() if v.is_floating_point() else v.cpu().numpy()
        np.testing.assert_array_equal(got, eager[k], err_msg=k)


@pytest.mark.parametrize("rule", [1, 2, 3])
@pytest.mark.parametrize("cfg,tau", [(2, 0.3), (3, 0.5), (5, 0.1), (6, 0.2), (7, 0.2)])
def test_accept_rules(dev, cfg, tau, rule):
    """The other readings of the first-mismatch rule (asd_accept_rule) against
    the oracle's literal enumeration / walk."""
    wl = H.prepared(cfg, small=True)
    out, status, _, _ = dev.run_verify(wl, tau, rule=rule)
    assert status == 0
    rep = H.compare_verify(wl, tau, out, rule=rule)
    H.untouched_cache_equal(wl, out, _written(wl, out))
    if rule in (1, 3):
        assert np.all(out["n_promoted"] <= 1)
    print(wl.name, tau, rule, rep)


@pytest.mark.parametrize("rule", [2, 3])
def test_greedy_accept_path_call_matches_verify_step(dev, rule):
    """asd_accept_path with the ratios asd_lmhead_margin wrote gives the verify
    step's path."""
    import torch
    from paper_2609_02897_gb300 import asd
    wl = H.prepared(3, small=True)
    ref, status, _, _ = dev.run_verify(wl, 0.1, rule=rule)
    assert status == 0
    d = dev.to_device(wl)
    dims = dev.dims_of(wl)
    dims.accept_rule = rule
    T, B = wl.T, wl.B
    ws = asd.alloc_workspace(dims, T)
    f = lambda: torch.empty(T, dtype=torch.float32, device="cuda")  # noqa: E731
    i = lambda n: torch.empty(n, dtype=torch.int32, device="cuda")  # noqa: E731
    rm, ra, rl, ld, rt = f(), i(T), f(), f(), f()
    acc = torch.empty(T, dtype=torch.uint8, device="cuda")
    asd.asd_lmhead_margin(dims, d["hidden"], d["w_lm"], d["tokens"], d["parent"], d["cu_nodes"], 0.1,
                          rm, ra, rl, ld, rt, acc, ws)
    path = torch.empty(B, dims.max_path, dtype=torch.int32, device="cuda")
    plen, bonus, npro = i(B), i(B), i(B)
    asd.asd_accept_path(dims, d["parent"], d["tokens"], acc, ra, d["cu_nodes"], path, plen, bonus,
                        npro, ws, ratio=rt)
    torch.cuda.synchronize()
    assert asd.asd_get_device_status(ws) == 0
    for name, t in [("path", path), ("path_len", plen), ("bonus", bonus), ("n_promoted", npro)]:
        np.testing.assert_array_equal(t.cpu().numpy(), ref[name], err_msg=name)
    with pytest.raises(asd.AsdError) as e:   # the greedy rules read the ratios
        asd.asd_accept_path(dims, d["parent"], d["tokens"], acc, ra, d["cu_nodes"], path, plen,
                            bonus, npro, ws)
    assert e.value.code == 1


@pytest.mark.parametrize("B", [2, 3, 4, 5, 7, 8, 9])
def test_lm_head_node_groups(dev, B):
    """Trees of 128 nodes, B of them: beyond one 128-node tile the LM head
    shares every W stage between a pair of node tiles (odd B: the last pair
    has one tile) and covers 256 vocabulary rows per MMA."""
    wl = H.prepared(5, small=True, overrides=dict(B=B))
    assert wl.T == 128 * B
    out, status, _, _ = dev.run_verify(wl, 0.3)
    assert status == 0
    H.compare_verify(wl, 0.3, out)
    H.untouched_cache_equal(wl, out, _written(wl, out))


def test_captured_step_with_host_copies(dev):
    """VerifyStep.capture: input copies from pinned host memory, the verify
    step and the result copies to pinned host memory, replayed as one graph,
    give the eagerly launched step's results."""
    import torch
    from paper_2609_02897_gb300 import asd
    wl = H.prepared(3, small=True)
    ref, status, _, _ = dev.run_verify(wl, 0.5)
    assert status == 0
    d = dev.to_device(wl)
    host = {k: d[k].cpu().pin_memory() for k in ("q", "tree_k", "tree_v", "hidden", "tokens",
                                                  "parent", "cu_nodes", "ctx_len")}
    for k in host:
        d[k].zero_()                         # only the captured copies bring the inputs
    step = asd.VerifyStep(dev.dims_of(wl), wl.T, attn_dtype=dev.dtype_of(wl))
    step.bind(tau=0.5, **d)
    outs = ("path", "path_len", "bonus", "row_lse", "accept")
    host_out = {k: torch.empty_like(step.out[k], device="cpu").pin_memory() for k in outs}
    g = step.capture([(d[k], v) for k, v in host.items()],
                     [(v, step.out[k]) for k, v in host_out.items()])
    g.replay()
    torch.cuda.synchronize()
    assert step.device_status() == 0
    for k in outs:
        np.testing.assert_array_equal(host_out[k].numpy(), ref[k], err_msg=k)
