"""The allocation-free LM-head entry point (asd_lmhead_margin_noalloc) gives
the same outputs as asd_lmhead_margin with a caller workspace.

Some callers cannot allocate device memory themselves (a plugin inside a
serving engine that has reserved all free memory for its KV-cache pool, or a
latency-critical loop that cannot afford cudaMalloc's synchronisation); this
entry point serves them from a static scratch array inside the library.  The
test calls it twice in a row through the C ABI, because the scratch keeps the
previous call's contents, and checks a request larger than the scratch is
refused.  This file is named to be collected last."""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu


def _outputs(T, device="cuda"):
    import torch
    nan = float("nan")
    return dict(row_max=torch.full((T,), nan, device=device),
                row_argmax=torch.full((T,), -7, dtype=torch.int32, device=device),
                row_lse=torch.full((T,), nan, device=device),
                l_draft=torch.full((T,), nan, device=device),
                ratio=torch.full((T,), nan, device=device),
                accept=torch.full((T,), 9, dtype=torch.uint8, device=device))


def test_noalloc_matches_workspace_entry_point():
    import torch
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    import _device
    import _helpers as H
    from paper_2609_02897_gb300 import asd

    for cfg in (2, 1):
        wl = H.prepared(cfg, small=True)
        tau = wl.taus[-1]
        d = _device.to_device(wl)
        dims = _device.dims_of(wl)
        T = wl.T
        ws = asd.alloc_workspace(dims, T)
        ref = _outputs(T)
        asd.asd_lmhead_margin(dims, d["hidden"], d["w_lm"], d["tokens"], d["parent"],
                              d["cu_nodes"], tau, ref["row_max"], ref["row_argmax"],
                              ref["row_lse"], ref["l_draft"], ref["ratio"], ref["accept"], ws)
        torch.cuda.synchronize()
        assert asd.asd_get_device_status(ws) == 0
        atol, rtol = H.tol(wl)
        for call in range(2):
            got = _outputs(T)
            status = torch.full((1,), -1, dtype=torch.int32, device="cuda")
            asd.asd_lmhead_margin_noalloc(dims, d["hidden"], d["w_lm"], d["tokens"], d["parent"],
                                          d["cu_nodes"], tau, got["row_max"], got["row_argmax"],
                                          got["row_lse"], got["l_draft"], got["ratio"],
                                          got["accept"], status)
            torch.cuda.synchronize()
            assert int(status.item()) == 0, f"call {call}: device status {int(status.item())}"
            for k in ("row_max", "row_lse"):
                H.assert_close(got[k].cpu().numpy(), ref[k].cpu().numpy(), atol, rtol, k)
            gp = wl.global_parent()
            kids = gp >= 0
            for k in ("l_draft", "ratio"):   # defined for drafted nodes; NaN at roots
                H.assert_close(got[k].cpu().numpy()[kids], ref[k].cpu().numpy()[kids],
                               atol, rtol, k)
                assert np.isnan(got[k].cpu().numpy()[~kids]).all()
            np.testing.assert_array_equal(got["row_argmax"].cpu().numpy(),
                                          ref["row_argmax"].cpu().numpy())
            np.testing.assert_array_equal(got["accept"].cpu().numpy(), ref["accept"].cpu().numpy())


def test_noalloc_rejects_requests_larger_than_its_scratch():
    import torch
    import _device
    import _helpers as H
    from paper_2609_02897_gb300 import asd

    wl = H.prepared(2, small=True)
    d = _device.to_device(wl)
    dims = _device.dims_of(wl)
    # enough trees of 128 nodes that the scratch need (16 bytes per node per
    # LM-head range, one range per SM up to the vocabulary's 32-row groups,
    # plus the children lists) exceeds the limit on this GPU, whatever its SM count
    dims.max_nodes = 128
    dims.batch = 1
    while asd.asd_workspace_bytes(dims, dims.batch * 128) <= asd.NOALLOC_SCRATCH_BYTES:
        dims.batch += 1
    T = dims.batch * 128
    big = torch.zeros(T, dtype=torch.int32, device="cuda")
    out = _outputs(T)
    with pytest.raises(asd.AsdError) as e:
        asd.asd_lmhead_margin_noalloc(dims, d["hidden"], d["w_lm"], big, big, big, 0.3,
                                      out["row_max"], out["row_argmax"], out["row_lse"],
                                      out["l_draft"], out["ratio"], out["accept"])
    assert e.value.code == 6
