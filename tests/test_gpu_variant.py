"""Which LM-head kernel a call runs (asd_lm_head_variant): the clustered wide
kernel, whose W multicast may read only the calling GPU's own memory, is
chosen for a weight in device memory of the current device and never for a
weight in host memory (pinned or pageable); small trees take the
weight-streaming kernel, fp32 workloads the fp32 kernel.  Nothing is
launched."""
import pytest

from paper_2609_02897_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    import torch
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    import _device
    return _device


def test_cluster_form_only_for_a_weight_on_this_gpu(dev):
    import torch
    from paper_2609_02897_gb300 import asd
    wl = synth.make_workload(5, small=True, overrides=dict(B=8))   # 1024 nodes: 4 tile pairs
    dims = dev.dims_of(wl)
    nsm = torch.cuda.get_device_properties(0).multi_processor_count
    ranges = max(1, min(nsm, 256, (wl.vocab + 31) // 32))
    w_dev = torch.empty(64, dtype=torch.bfloat16, device="cuda")
    w_pinned = torch.empty(64, dtype=torch.bfloat16).pin_memory()
    w_pageable = torch.empty(64, dtype=torch.bfloat16)
    assert asd.asd_lm_head_variant(dims, wl.T, w_dev) == (3 if ranges % 2 == 0 else 2)
    assert asd.asd_lm_head_variant(dims, wl.T, w_pinned) == 2
    assert asd.asd_lm_head_variant(dims, wl.T, w_pageable) == 2
    # two tile pairs: clustered (with pairing ranges); three: unclustered (one
    # CTA of a cluster would idle through the second round)
    assert asd.asd_lm_head_variant(dims, 512, w_dev) == (3 if ranges % 2 == 0 else 2)
    assert asd.asd_lm_head_variant(dims, 768, w_dev) == 2
    assert asd.asd_lm_head_variant(dims, 256, w_dev) == 2
    # the lazy schedule's levels run the wide kernel unclustered
    dims.lm_head_schedule = asd.ASD_LM_LAZY_LEVELS
    assert asd.asd_lm_head_variant(dims, wl.T, w_dev) == 2


def test_small_trees_and_fp32(dev):
    import torch
    from paper_2609_02897_gb300 import asd
    w_dev = torch.empty(64, dtype=torch.bfloat16, device="cuda")
    small = synth.make_workload(2, small=True)
    assert asd.asd_lm_head_variant(dev.dims_of(small), small.T, w_dev) == 1
    tiny = synth.make_workload(1)
    assert asd.asd_lm_head_variant(dev.dims_of(tiny), tiny.T, w_dev) == 4
    assert asd.asd_lm_head_variant(dev.dims_of(small), 0, w_dev) == 0


def test_attention_variant(dev):
    import torch
    from paper_2609_02897_gb300 import asd
    nsm = torch.cuda.get_device_properties(0).multi_processor_count
    small = synth.make_workload(2, small=True)
    assert asd.asd_attention_variant(dev.dims_of(small), small.T) == 1
    tiny = synth.make_workload(1)
    assert asd.asd_attention_variant(dev.dims_of(tiny), tiny.T) == 4
    wl = synth.make_workload(5, small=True)        # 6 x 128 nodes, 2 KV heads, G = 4
    dims = dev.dims_of(wl)
    assert asd.asd_attention_variant(dims, wl.T) == 2
    # the two-tile form once its 256-row items fill two waves of CTAs
    dims.batch = 4 * nsm
    items = dims.num_kv_heads * ((dims.batch * 128 * 4 + 255) // 256)
    assert items >= 2 * nsm
    assert asd.asd_attention_variant(dims, dims.batch * 128) == 3
    assert asd.asd_attention_variant(dims, 0) == 0
