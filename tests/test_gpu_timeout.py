"""The failure path of the bounded waits (a wait that gives up), in the form
that leaves the GPU usable: the test shortens the wait bound through the
library's test hook (asd_debug_set_wait_cycles) so that a kernel's first
wait on its own copy or MMA gives up, and checks that the call reports
ASD_ERR_TIMEOUT, commits nothing (every path empty, the cache untouched,
ctx_len_out = ctx_len), and that the next call with the default bound is
clean and gives the results of an ordinary call bit for bit.  Covered: the
weight-streaming LM head with the bf16 attention beside it (60-node tree) and
the wide LM head in its unclustered form with the one-tile tensor-core
attention (768 nodes), and the ping-pong attention on its own; the clustered
form of the wide LM head is not driven into a timeout here.  All calls go
through the C ABI."""
import numpy as np
import pytest

import _helpers as H

pytestmark = pytest.mark.gpu

ASD_ERR_TIMEOUT = 8


@pytest.fixture(scope="module")
def dev():
    import torch
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    import _device
    return _device


@pytest.mark.parametrize("cfg,tau", [(2, 0.3), (5, 0.3)])
def test_a_wait_that_gives_up_reports_and_commits_nothing(dev, cfg, tau):
    from paper_2609_02897_gb300 import asd
    wl = H.prepared(cfg, small=True)
    if cfg == 5:
        # at most three 256-node pairs of tiles: the wide LM head runs unclustered
        assert wl.T <= 768, wl.T
    ref, status, _, _ = dev.run_verify(wl, tau)
    assert status == 0
    asd.asd_debug_set_wait_cycles(64)
    try:
        out, status, _, _ = dev.run_verify(wl, tau)
    finally:
        asd.asd_debug_set_wait_cycles(0)
    assert status == ASD_ERR_TIMEOUT, asd.STATUS.get(status, status)
    assert np.all(out["path_len"] == 0)
    np.testing.assert_array_equal(out["ctx_len_out"], wl.ctx_len)
    H.untouched_cache_equal(wl, out, [])
    again, status, _, _ = dev.run_verify(wl, tau)
    assert status == 0
    for k in ref:
        np.testing.assert_array_equal(again[k], ref[k], err_msg=k)
    H.compare_verify(wl, tau, again)



def test_pingpong_attention_wait_that_gives_up(dev):
    """The ping-pong attention (two producer warps, two MMA-issuing threads,
    eight softmax warps) under the shortened bound: the call reports
    ASD_ERR_TIMEOUT, and the next call with the default bound gives the
    ordinary output bit for bit.  The standalone attention call, so no LM head
    runs: the batch that selects this kernel would take the clustered wide LM
    head, which is not driven into a timeout."""
    import torch
    from paper_2609_02897_gb300 import asd, synth
    nsm = torch.cuda.get_device_properties(0).multi_processor_count
    spec = dict(synth.WORKLOADS[5])
    spec.update(synth.SMALL[5])
    hkv, g = spec["Hkv"], spec["Hq"] // spec["Hkv"]
    b = 1   # sequences of 128 nodes that give two waves of 256-row items
    while hkv * ((b * 128 * g + 255) // 256) < 2 * nsm:
        b += 1
    wl = H.prepared(5, small=True, overrides=dict(B=b))
    d = dev.to_device(wl)
    dims = dev.dims_of(wl)
    assert asd.asd_attention_variant(dims, wl.T) == 3
    ws = asd.alloc_workspace(dims, wl.T)

    def attend():
        out = torch.full((wl.T, wl.Hq, wl.D), float("nan"), dtype=dev.dtype_of(wl), device="cuda")
        asd.asd_tree_attention(dims, d["q"], d["k_cache"], d["v_cache"], d["page_table"],
                               d["ctx_len"], d["tree_k"], d["tree_v"], d["parent"], d["cu_nodes"],
                               out, ws)
        torch.cuda.synchronize()
        return out, asd.asd_get_device_status(ws)

    ref, status = attend()
    assert status == 0
    asd.asd_debug_set_wait_cycles(64)
    try:
        _, status = attend()
    finally:
        asd.asd_debug_set_wait_cycles(0)
    assert status == ASD_ERR_TIMEOUT, asd.STATUS.get(status, status)
    again, status = attend()
    assert status == 0
    assert torch.equal(again.view(torch.int16), ref.view(torch.int16))
