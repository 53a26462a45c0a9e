"""The tensor-core attention in its two-query-tile (ping-pong) form, which
serves steps whose 256-row items fill at least two waves of CTAs: the paged
workload drawn with enough sequences to select it (checked through
asd_attention_variant), 128- and 64-dim heads, against the oracle on sampled
sequences (attention of all their nodes and heads, LM-head rows, path, bonus
and commit) plus the any-size properties on every sequence.  The smaller
workloads of the other GPU tests run the one-tile form."""
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


def _batch_for_pingpong(nsm, hkv, g, nodes):
    """Sequences of `nodes` nodes that give at least two waves of 256-row items."""
    per_seq_rows = nodes * g
    b = 1
    while hkv * ((b * per_seq_rows + 255) // 256) < 2 * nsm:
        b += 1
    return b


@pytest.mark.parametrize("over", [dict(), dict(D=64)])
def test_pingpong_attention_matches_the_oracle(dev, over):
    import torch
    from paper_2609_02897_gb300 import asd, synth
    nsm = torch.cuda.get_device_properties(0).multi_processor_count
    spec = dict(synth.WORKLOADS[5])
    spec.update(synth.SMALL[5])
    B = _batch_for_pingpong(nsm, spec["Hkv"], spec["Hq"] // spec["Hkv"], 128)
    wl = H.prepared(5, small=True, overrides=dict(B=B, **over))
    dims = dev.dims_of(wl)
    assert asd.asd_attention_variant(dims, wl.T) == 3
    # a smaller batch of the same shape takes the one-tile form
    assert asd.asd_attention_variant(dims, 4 * 128) == 2
    tau = 0.3
    out, status, _, _ = dev.run_verify(wl, tau)
    assert status == 0
    seqs = [0, B // 2, B - 1]
    rep = H.compare_verify(wl, tau, out, seqs=seqs)
    gp = wl.global_parent()
    kids = gp >= 0
    assert np.all(out["ratio"][kids] >= 0) and np.all(out["ratio"][kids] <= 1)
    written = []
    for b in range(wl.B):
        s, e = int(wl.cu_nodes[b]), int(wl.cu_nodes[b + 1])
        plen = int(out["path_len"][b])
        path = [int(x) for x in out["path"][b][:plen]]
        assert H.valid_path(list(wl.parent[s:e]), list(out["accept"][s:e]), path), b
        written += [(b, int(wl.ctx_len[b]) + k) for k in range(plen)]
    H.untouched_cache_equal(wl, out, written)
    print(wl.name, B, over, rep)
