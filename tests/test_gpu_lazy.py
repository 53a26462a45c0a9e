"""The lazy, level-synchronous LM-head schedule (asd_lm_schedule
ASD_LM_LAZY_LEVELS) against the oracle: the rows it computes are exactly the
roots and the nodes reached through accepted nodes (a node's verdict needs its
parent's row, Eq. 1 and the kappa rule of Sec. 3.2); the oracle evaluates the
same rows, and their statistics, their children's verdicts, the committed
path, bonus token, n_promoted, attention output and cache are compared with
it as for the every-row schedule.  In addition the lazy outputs equal the
every-row schedule's bit for bit on every computed row and judged node.  All
calls go through the C ABI."""
import numpy as np
import pytest

import _helpers as H

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    import torch
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    import _device
    return _device


def _check(wl, eager, lazy):
    """The lazy outputs against the every-row schedule's, bit for bit."""
    for k in ("path", "path_len", "bonus", "n_promoted", "ctx_len_out", "attn_out", "k_cache",
              "v_cache"):
        np.testing.assert_array_equal(lazy[k], eager[k], err_msg=k)
    reach = H.reached_rows(wl, eager["accept"])
    computed = ~np.isnan(lazy["row_max"])
    np.testing.assert_array_equal(computed, reach, err_msg="rows computed")
    for k in ("row_max", "row_argmax", "row_lse"):
        np.testing.assert_array_equal(lazy[k][reach], eager[k][reach], err_msg=k)
    assert np.all(np.isnan(lazy["row_lse"][~reach])) and np.all(lazy["row_argmax"][~reach] == -1)
    judged = np.zeros(wl.T, bool)
    for b in range(wl.B):
        s, e = int(wl.cu_nodes[b]), int(wl.cu_nodes[b + 1])
        for i in range(s + 1, e):
            judged[i] = reach[s + int(wl.parent[i])]
    for k in ("l_draft", "ratio", "accept"):
        np.testing.assert_array_equal(lazy[k][judged], eager[k][judged], err_msg=k)
    roots = wl.cu_nodes[:-1].astype(int)
    assert np.all(lazy["accept"][roots] == 1)
    other = ~judged
    other[roots] = False
    assert np.all(lazy["accept"][other] == 0)
    assert np.all(np.isnan(lazy["ratio"][other])) and np.all(np.isnan(lazy["l_draft"][other]))
    return int(reach.sum())


@pytest.mark.parametrize("cfg,tau,rule", [(2, 0.3, 0), (2, 1.0, 0), (3, 0.5, 0), (3, 0.1, 2),
                                          (5, 1.0, 0), (5, 0.3, 1), (5, 0.1, 3), (6, 0.2, 0),
                                          (7, 0.2, 0), (8, 1.0, 0)])
def test_lazy_matches_oracle(dev, cfg, tau, rule):
    wl = H.prepared(cfg, small=True)
    eager, s0, _, _ = dev.run_verify(wl, tau, rule=rule)
    lazy, s1, _, _ = dev.run_verify(wl, tau, rule=rule, schedule=1)
    assert s0 == 0 and s1 == 0
    rep = H.compare_verify(wl, tau, lazy, rule=rule, lazy=True)
    n = _check(wl, eager, lazy)
    print(wl.name, tau, rule, f"{n} of {wl.T} rows computed", rep)


@pytest.mark.parametrize("B", [1, 3, 9])
def test_lazy_many_rows_per_level(dev, B):
    """Trees of 128 nodes at tau 0.1 (wide accepted regions: levels of more
    than one 128-row tile)."""
    wl = H.prepared(5, small=True, overrides=dict(B=B))
    eager, s0, _, _ = dev.run_verify(wl, 0.1)
    lazy, s1, _, _ = dev.run_verify(wl, 0.1, schedule=1)
    assert s0 == 0 and s1 == 0
    rep = H.compare_verify(wl, 0.1, lazy, lazy=True)
    _check(wl, eager, lazy)
    print(wl.name, B, rep)


def test_lazy_lmhead_margin_call(dev):
    """asd_lmhead_margin under the lazy schedule writes what the verify step
    writes."""
    import torch
    from paper_2609_02897_gb300 import asd
    wl = H.prepared(3, small=True)
    ref, status, _, _ = dev.run_verify(wl, 0.5, schedule=1)
    assert status == 0
    d = dev.to_device(wl)
    dims = dev.dims_of(wl)
    dims.lm_head_schedule = asd.ASD_LM_LAZY_LEVELS
    T = wl.T
    ws = asd.alloc_workspace(dims, T)
    f = [torch.empty(T, dtype=torch.float32, device="cuda") for _ in range(5)]
    ra = torch.empty(T, dtype=torch.int32, device="cuda")
    acc = torch.empty(T, dtype=torch.uint8, device="cuda")
    asd.asd_lmhead_margin(dims, d["hidden"], d["w_lm"], d["tokens"], d["parent"], d["cu_nodes"],
                          0.5, f[0], ra, f[1], f[2], f[3], acc, ws)
    torch.cuda.synchronize()
    assert asd.asd_get_device_status(ws) == 0
    got = dict(row_max=f[0], row_argmax=ra, row_lse=f[1], l_draft=f[2], ratio=f[3], accept=acc)
    for k, t in got.items():
        np.testing.assert_array_equal(t.cpu().numpy(), ref[k], err_msg=k)


def test_lazy_step_in_a_cuda_graph(dev):
    """The lazy schedule (a memset and two kernels per level) captured once
    and replayed gives the eager-launch results."""
    import torch
    from paper_2609_02897_gb300 import asd
    wl = H.prepared(5, small=True)
    ref, status, _, _ = dev.run_verify(wl, 0.3, schedule=1)
    assert status == 0
    d = dev.to_device(wl)
    dims = dev.dims_of(wl)
    dims.lm_head_schedule = asd.ASD_LM_LAZY_LEVELS
    step = asd.VerifyStep(dims, wl.T, attn_dtype=dev.dtype_of(wl))
    k0, v0 = d["k_cache"].clone(), d["v_cache"].clone()
    step.bind(tau=0.3, **d)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            step.run(s)
    torch.cuda.current_stream().wait_stream(s)
    d["k_cache"].copy_(k0)
    d["v_cache"].copy_(v0)
    g.replay()
    torch.cuda.synchronize()
    assert step.device_status() == 0
    for k in ("path", "path_len", "bonus", "row_max", "accept"):
        np.testing.assert_array_equal(step.out[k].cpu().numpy(), ref[k], err_msg=k)
