"""GPU parity at the full workload sizes, in the launch configuration the
benchmark times (asd_verify_step).  The oracle recomputes every output of a
few sampled sequences (attention of all their nodes and heads, their LM-head
rows over the full vocabulary, path, bonus and commit); every other sequence
is checked through properties that hold at any size (valid longest path for
the accept mask, committed rows equal the path's tree K/V, untouched cache
bytes unchanged, ratio in [0, 1])."""
import numpy as np
import pytest

import _helpers as H
from paper_2609_02897_gb300 import synth

pytestmark = pytest.mark.gpu

SAMPLED = {1: None, 2: None, 3: [0, 7, 15], 4: [0, 5], 5: [0, 41], 6: None, 7: None, 8: None}


@pytest.fixture(scope="module")
def dev():
    import torch
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    import _device
    return _device


def _properties(wl, out):
    gp = wl.global_parent()
    kids = gp >= 0
    assert np.all(out["ratio"][kids] >= 0) and np.all(out["ratio"][kids] <= 1)
    assert np.all(out["accept"][~kids] == 1)
    written = []
    for b in range(wl.B):
        s, e = int(wl.cu_nodes[b]), int(wl.cu_nodes[b + 1])
        plen = int(out["path_len"][b])
        path = [int(x) for x in out["path"][b][:plen]]
        assert H.valid_path(list(wl.parent[s:e]), list(out["accept"][s:e]), path), b
        assert int(out["bonus"][b]) == int(out["row_argmax"][s + path[-1]])
        assert int(out["ctx_len_out"][b]) == int(wl.ctx_len[b]) + plen
        written += [(b, int(wl.ctx_len[b]) + k) for k in range(plen)]
    H.untouched_cache_equal(wl, out, written)


@pytest.mark.parametrize("cfg", sorted(synth.WORKLOADS))
def test_full_size(dev, cfg):
    wl = synth.make_workload(cfg)
    seqs = SAMPLED[cfg]
    synth.attach_tokens(wl, H.ranks_via_oracle(wl))
    for tau in synth.WORKLOADS[cfg]["tau"]:
        out, status, _, _ = dev.run_verify(wl, tau)
        assert status == 0
        rep = H.compare_verify(wl, tau, out, seqs=seqs)
        _properties(wl, out)
        print(f"{wl.name} tau={tau} T={wl.T} {rep} mean_path={out['path_len'].mean():.2f}")
