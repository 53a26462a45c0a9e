"""The packed streaming layout of the LM-head weight (asd_pack_lm_head): the
packed bytes match the layout documented in include/asd.h and csrc/kernels.h
(re-derived here with numpy), and every output of a verify step or of the LM
head alone is bit-identical whichever layout W is passed in.  All calls go
through the C ABI."""
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


def _pack_reference(w_bits, ranges):
    """Packed layout from its definition: header, then per range, per tile of
    up to 4 groups of 32 rows, per k-block of 64 columns: the tile's rows x
    128 bytes with 16-byte chunk c of row r stored at chunk c ^ (r & 7)."""
    V, K = w_bits.shape
    ng_all, nkb = -(-V // 32), -(-K // 64)
    wp = np.zeros((ng_all * 32, nkb * 64), np.uint16)
    wp[:V, :K] = w_bits
    out = np.zeros(256 + ng_all * nkb * 4096, np.uint8)
    out[:20] = np.array([0x57445341, 1, V, K, ranges], np.uint32).view(np.uint8)
    for c in range(ranges):
        gs, ge = c * ng_all // ranges, (c + 1) * ng_all // ranges
        for g0 in range(gs, ge, 4):
            ng = min(4, ge - g0)
            R = ng * 32
            rr = np.arange(R)[:, None]
            swz = np.arange(8)[None, :] ^ (rr & 7)
            for kb in range(nkb):
                blk = wp[g0 * 32:g0 * 32 + R, kb * 64:(kb + 1) * 64].reshape(R, 8, 8)
                sw = np.empty_like(blk)
                sw[rr, swz] = blk
                off = 256 + 4096 * (nkb * g0 + kb * ng)
                out[off:off + R * 128] = sw.reshape(-1).view(np.uint8)
    return out


def test_packed_bytes_match_layout(dev):
    import torch
    from paper_2609_02897_gb300 import asd
    V, K = 20007, 200                     # ragged in both: 626 groups, 4 k-blocks (last 8 cols)
    g = torch.Generator().manual_seed(7)
    w = torch.randn(V, K, generator=g).to(torch.bfloat16).cuda()
    dims = asd.make_dims(1, 4, 4, 64, K, V, asd.ASD_BF16, 0, 64, 0, 8, 5, asd.ASD_LM_PACKED)
    packed = asd.pack_lm_head(dims, w)
    torch.cuda.synchronize()
    nsm = torch.cuda.get_device_properties(0).multi_processor_count
    ranges = max(1, min(nsm, 256, -(-V // 32)))
    ref = _pack_reference(w.view(torch.int16).cpu().numpy().view(np.uint16), ranges)
    got = packed.cpu().numpy()
    assert got.shape == ref.shape
    np.testing.assert_array_equal(got, ref)


def _run(dev, wl, tau, packed):
    from paper_2609_02897_gb300 import asd
    import torch
    d = dev.to_device(wl)
    dims = dev.dims_of(wl)
    if packed:
        dims.lm_head_layout = asd.ASD_LM_PACKED
        d["w_lm"] = asd.pack_lm_head(dims, d["w_lm"])
    step = asd.VerifyStep(dims, wl.T, attn_dtype=dev.dtype_of(wl))
    step.bind(tau=tau, **d)
    step.run()
    torch.cuda.synchronize()
    out = {k: v.float().cpu().numpy() if v.is_floating_point() else v.cpu().numpy()
           for k, v in step.out.items()}
    out["k_cache"] = d["k_cache"].float().cpu().numpy()
    out["v_cache"] = d["v_cache"].float().cpu().numpy()
    return out, step.device_status()


@pytest.mark.parametrize("cfg,over", [(2, None), (3, None), (4, None), (5, None), (2, dict(D=64)),
                                      (5, dict(B=8)), (5, dict(B=9))])
def test_packed_verify_step_is_bit_identical(dev, cfg, over):
    """Both weight layouts give the same bits; B = 8, 9 at 128 nodes each run
    the LM head in clusters of two (multicast of the packed copies, an odd
    number of node pairs for B = 9)."""
    wl = H.prepared(cfg, small=True, overrides=over)
    tau = 0.3
    rows, s0 = _run(dev, wl, tau, packed=False)
    pk, s1 = _run(dev, wl, tau, packed=True)
    assert s0 == 0 and s1 == 0
    for k in rows:
        np.testing.assert_array_equal(pk[k], rows[k], err_msg=k)
    H.compare_verify(wl, tau, pk)


def test_packed_lmhead_margin_is_bit_identical(dev):
    import torch
    from paper_2609_02897_gb300 import asd
    wl = H.prepared(3, small=True)
    d = dev.to_device(wl)
    T = wl.T
    res = []
    for packed in (False, True):
        dims = dev.dims_of(wl)
        w = d["w_lm"]
        if packed:
            dims.lm_head_layout = asd.ASD_LM_PACKED
            w = asd.pack_lm_head(dims, w)
        ws = asd.alloc_workspace(dims, T)
        f = [torch.empty(T, dtype=torch.float32, device="cuda") for _ in range(5)]
        ra = torch.empty(T, dtype=torch.int32, device="cuda")
        acc = torch.empty(T, dtype=torch.uint8, device="cuda")
        asd.asd_lmhead_margin(dims, d["hidden"], w, d["tokens"], d["parent"], d["cu_nodes"], 0.5,
                              f[0], ra, f[1], f[2], f[3], acc, ws)
        torch.cuda.synchronize()
        assert asd.asd_get_device_status(ws) == 0
        res.append([t.cpu().numpy() for t in (*f[:4], ra, acc)])
    for a, b in zip(*res):
        np.testing.assert_array_equal(a, b)


def test_packed_header_mismatch_is_reported(dev):
    import torch
    from paper_2609_02897_gb300 import asd
    wl = H.prepared(2, small=True)
    d = dev.to_device(wl)
    dims = dev.dims_of(wl)
    dims.lm_head_layout = asd.ASD_LM_PACKED
    good = asd.pack_lm_head(dims, d["w_lm"])
    bad = good.clone()
    bad[:4] = 0                                   # not a packed weight
    for w, want in ((bad, 2), (good, 0)):         # the error, then a clean call
        dd = dict(d)
        dd["w_lm"] = w
        step = asd.VerifyStep(dims, wl.T)
        step.bind(tau=0.3, **dd)
        step.run()
        torch.cuda.synchronize()
        assert step.device_status() == want
