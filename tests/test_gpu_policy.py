"""GPU parity of the tree-shape policy kernels (asd_policy_init / update /
select, Sec. 3.3, Eq. 2) against the oracle: the per-request state is
bit-identical after every step (both sides evaluate the same binary64
operations one rounding at a time), the DCS agrees to the last few ulps (the
only difference is the exp of the device's math library), and the triplet is
exactly the oracle's mapping of the device's DCS.  All calls go through the C
ABI."""
import math

import numpy as np
import pytest

from oracle import policy as P

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch_cuda():
    import torch
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2609_02897_gb300 import asd
    return torch, asd


def _state_np(pol):
    rar, streak, breaks = pol.state_arrays()
    return rar.cpu().numpy(), streak.cpu().numpy(), breaks.cpu().numpy()


def _near_half(score, shallow, deep, eps=1e-12):
    """True when one of the score's interpolants lies within eps of a
    rounding boundary (the exp of two math libraries may then decide it
    differently)."""
    for a, b, u in ((shallow[0], deep[0], score), (deep[1], shallow[1], 1.0 - score),
                    (shallow[2], deep[2], score)):
        y = (b - a) * u
        if abs(y - math.floor(y) - 0.5) < eps:
            return True
    return False


SETTINGS = [dict(), dict(alpha=0.5, divisor=0.3, rar_init=0.6, shallow=(2, 6, 3),
                         deep=(9, 1, 16), breaker=3)]


@pytest.mark.parametrize("kw", SETTINGS)
def test_policy_steps_match_the_oracle(torch_cuda, kw):
    torch, asd = torch_cuda
    B, steps = 300, 40                       # three 128-thread blocks, ragged tail
    rng = np.random.default_rng(17)
    params = asd.make_policy_params(**kw)
    shallow, deep = tuple(params.shallow), tuple(params.deep)
    pol = asd.TreePolicy(B, params)
    ref = [P.initial_state(params.rar_init) for _ in range(B)]
    reported = 0
    for t in range(steps):
        # one verify step: tree sizes 1..12, path lengths weighted towards
        # zero-accept so that breakers fire, plus malformed (0) and out-of-range
        n = rng.integers(1, 13, B)
        pl = np.where(rng.random(B) < 0.45, 1, rng.integers(0, 13, B))
        pl = np.minimum(pl, n + (rng.random(B) < 0.02))
        cu = np.concatenate([[0], np.cumsum(n)]).astype(np.int32)
        pol.update(torch.from_numpy(cu).cuda(), torch.from_numpy(pl.astype(np.int32)).cuda())
        for b in range(B):
            P.update(ref[b], n[b], pl[b], params.alpha, params.breaker, params.rar_init)
        rar, streak, breaks = _state_np(pol)
        np.testing.assert_array_equal(rar, [r["rar"] for r in ref], err_msg=f"rar step {t}")
        np.testing.assert_array_equal(streak, [r["zero_streak"] for r in ref])
        np.testing.assert_array_equal(breaks, [r["breaks"] for r in ref])
        # the draft LM head's row statistics of each request's root
        rows = rng.permutation(B).astype(np.int32)
        m = rng.normal(0, 3, B).astype(np.float32)
        lse = (m + rng.exponential(1.5, B)).astype(np.float32)
        trip = pol.select(torch.from_numpy(m).cuda(), torch.from_numpy(lse).cuda(),
                          torch.from_numpy(rows).cuda()).cpu().numpy()
        dcs = pol.dcs.cpu().numpy()
        for b in range(B):
            r = rows[b]
            score, want = P.select(ref[b], P.p_top1(m[r], lse[r]), params.divisor, shallow, deep)
            assert dcs[b] == pytest.approx(score, rel=4e-16, abs=1e-300), (t, b)
            assert tuple(trip[b]) == P.triplet(float(dcs[b]), shallow, deep), (t, b)
            if tuple(trip[b]) != want:
                assert _near_half(score, shallow, deep), (t, b, score, trip[b], want)
                reported += 1
    assert reported == 0 or reported < B * steps // 1000
    assert max(r["breaks"] for r in ref) >= 1       # the breaker fired somewhere
    every = set(asd.asd_policy_triplets(params))
    assert set(map(tuple, trip.tolist())) <= every


def test_policy_select_edges(torch_cuda):
    """Saturation, zero probability, a NaN probability and a row index outside
    the row statistics."""
    torch, asd = torch_cuda
    params = asd.make_policy_params()
    pol = asd.TreePolicy(5, params)
    m = torch.tensor([0.0, 0.0, -1e30, float("nan"), 0.0], device="cuda")
    lse = torch.tensor([0.0, 100.0, 0.0, 0.0, 0.7], device="cuda")
    rows = torch.tensor([0, 1, 2, 3, 7], dtype=torch.int32, device="cuda")
    trip = pol.select(m, lse, rows).cpu().numpy()
    dcs = pol.dcs.cpu().numpy()
    assert tuple(trip[0]) == (7, 1, 8) and dcs[0] == 1.0        # p = 1, RAR = 1
    assert tuple(trip[1]) == (3, 4, 4) and 0.0 < dcs[1] < 1e-40  # p = exp(-100)
    assert tuple(trip[2]) == (3, 4, 4) and dcs[2] == 0.0        # exp(-1e30) = 0
    assert tuple(trip[3]) == (3, 4, 4) and dcs[3] == 0.0        # NaN counts as 0
    assert tuple(trip[4]) == (0, 0, 0) and math.isnan(dcs[4])   # row 7 of 5
    # rows = NULL: request b reads row b
    trip = pol.select(m, lse).cpu().numpy()
    assert tuple(trip[4]) == P.triplet(P.dcs(math.exp(-0.7), 1.0, 0.5), (3, 4, 4), (7, 1, 8))


def test_policy_from_the_lm_head_statistics(torch_cuda):
    """The draft's p(top1) taken from asd_lmhead_margin's row_max / row_lse:
    the chain LM head -> policy.select runs on the device and agrees with the
    oracle's LM head and policy within the fp32 statistics' precision."""
    torch, asd = torch_cuda
    import _helpers as H
    import _device
    import oracle
    wl = H.prepared(3, small=True)
    d = _device.to_device(wl)
    dims = _device.dims_of(wl)
    T = wl.T
    ws = asd.alloc_workspace(dims, T)
    f = [torch.empty(T, dtype=torch.float32, device="cuda") for _ in range(5)]
    ra = torch.empty(T, dtype=torch.int32, device="cuda")
    acc = torch.empty(T, dtype=torch.uint8, device="cuda")
    asd.asd_lmhead_margin(dims, d["hidden"], d["w_lm"], d["tokens"], d["parent"], d["cu_nodes"],
                          0.5, f[0], ra, f[1], f[2], f[3], acc, ws)
    pol = asd.TreePolicy(wl.B)
    roots = d["cu_nodes"][:-1].contiguous()
    trip = pol.select(f[0], f[1], roots).cpu().numpy()
    torch.cuda.synchronize()
    assert asd.asd_get_device_status(ws) == 0
    lm = oracle.lmhead_margin(wl.hidden, wl.w, wl.tokens, wl.parent, wl.cu_nodes, 0.5)
    dcs = pol.dcs.cpu().numpy()
    for b in range(wl.B):
        r = int(wl.cu_nodes[b])
        p = P.p_top1(lm["row_max"][r], lm["row_lse"][r])
        score, want = P.select(P.initial_state(), p, 0.5, (3, 4, 4), (7, 1, 8))
        assert dcs[b] == pytest.approx(score, rel=1e-5, abs=1e-12)
        assert tuple(trip[b]) == P.triplet(float(dcs[b]), (3, 4, 4), (7, 1, 8))


def test_policy_in_a_cuda_graph(torch_cuda):
    """update + select captured once and replayed give the eager results."""
    torch, asd = torch_cuda
    B = 64
    rng = np.random.default_rng(3)
    n = torch.from_numpy(np.concatenate([[0], np.cumsum(rng.integers(2, 9, B))]).astype(
        np.int32)).cuda()
    pl = torch.ones(B, dtype=torch.int32, device="cuda")
    m = torch.zeros(B, device="cuda")
    lse = torch.full((B,), 0.4, device="cuda")
    eager, graph = asd.TreePolicy(B), asd.TreePolicy(B)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            graph.update(n, pl, stream=s)
            graph.select(m, lse, stream=s)
    torch.cuda.current_stream().wait_stream(s)
    for _ in range(7):                                # crosses the breaker (5)
        eager.update(n, pl)
        eager.select(m, lse)
        g.replay()
    torch.cuda.synchronize()
    for a, b in zip(eager.state_arrays(), graph.state_arrays()):
        assert torch.equal(a, b)
    assert torch.equal(eager.triplet, graph.triplet) and torch.equal(eager.dcs, graph.dcs)
    assert int(eager.state_arrays()[2][0]) == 1
