#!/usr/bin/env python3
"""Verify-step benchmark on the Llama-3.1-8B-shaped workload (batch 1, context
2048, 32 query / 8 KV heads, head dim 128, hidden 4096, vocab 128256, 60-node
EAGLE-style tree of depth <= 8 and top-k 10, tau = 0.3), synthetic seeded data.

One step = the whole hot path through the C ABI (asd_verify_step): tree
preparation, tree attention + split combine, the tcgen05 LM head with the
fused margin epilogue, and the merge / accepted-path / K/V-commit tail.

  python bench.py [--gpus N --steps K --warmup W] [--impl reference]

Prints one JSON line.  Under torchrun every rank runs its own replica of the
workload (weak scaling, no data-path collective); value = all ranks' nodes /
the slowest rank's time.  `--impl reference` times the fp64 CPU oracle on a
bounded sample instead (rank 0 only).
"""
import argparse
import csv
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "verified tree nodes/s"
UNIT = "nodes/s"
CONFIG = 2
TAU = 0.3
N_STAGE_KERNELS = 4   # prep, LM head, attention (splits merged in-kernel), tail
STAGES = ("prep", "lmhead", "attention", "tail")   # order of the stage events
# DRAM bytes (read + write) of one LM-head launch on this workload, from the
# ncu capture summarised in profiles/verify_step_llama8b_b1_ctx2048_tree60.md;
# set to None whenever lmhead_tc.cu changes until it is captured again.
LMHEAD_TRAFFIC_BYTES = 1054301744
# DRAM bytes (read + write) of one LM-head launch from an ncu capture of the current
# kernel, per workload (packed weight): 60 nodes (lmhead_tc_kernel) and 907 nodes
# (lmhead_wide_kernel in clusters of two: 2 W passes)
LMHEAD_TRAFFIC_BY_CONFIG = {2: LMHEAD_TRAFFIC_BYTES, 3: 2099486768}


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=50)
    ap.add_argument("--impl", default="asd", choices=["asd", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-clocks", action="store_true")
    ap.add_argument("--config", type=int, default=CONFIG,
                    help="workload number (synth.WORKLOADS); the default is the headline "
                         "Llama-3.1-8B-shaped verify step, the others are for the record")
    ap.add_argument("--tau", type=float, default=None,
                    help="margin threshold (default: the workload's first)")
    ap.add_argument("--lm-layout", default="packed", choices=["packed", "rows"],
                    help="LM-head weight as packed once at load (default) or as [V, K] rows")
    ap.add_argument("--lm-schedule", default="every-row", choices=["every-row", "lazy"],
                    help="LM-head rows: every node's (default) or, level by level, only those "
                         "the accepted-path walk can reach")
    return ap.parse_args()


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def tensor_peak():
    """Dense bf16 TFLOP/s: the measured burst figure, else the fallback."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["bf16_tflops"]), "measured"
    except Exception:
        return 1900.0, "fallback"


def workload_config(wl):
    if CONFIG == 2:
        desc = ("llama3.1-8b-shaped verify step: batch 1, context 2048, 32 q / 8 kv heads, "
                "head_dim 128, hidden 4096, vocab 128256, 60-node EAGLE-style tree "
                "(depth<=8, top-k 10), tau 0.3, bf16")
    else:
        desc = (f"{wl.name}: batch {wl.B}, context {int(wl.ctx_len.min())}-{int(wl.ctx_len.max())}, "
                f"{wl.Hq} q / {wl.Hkv} kv heads, head_dim {wl.D}, hidden {wl.hidden_dim}, "
                f"vocab {wl.vocab}, {wl.T} tree nodes"
                + (f", paged ({wl.page_size} tokens per page)" if wl.page_size else "")
                + f", tau {TAU}, {wl.dtype}")
    return {
        "workload": desc,
        "batch": wl.B, "ctx": int(wl.ctx_len[0]), "tree_nodes": wl.T,
        "tree_depth": int(wl.max_path - 1), "tau": TAU,
        "l2": "inputs larger than L2: the 1.05 GB LM-head weight is streamed every step",
    }


def esz(wl):
    """Bytes per element of the workload's tensors."""
    return 2 if wl.dtype == "bf16" else 4


def lmhead_bytes(wl, rows=None, passes=1):
    """Algorithmic bytes of the LM head: W read once per pass, the hidden states of
    the computed rows read once, per-row statistics written (every row and one pass
    unless given)."""
    rows = wl.T if rows is None else rows
    return (passes * wl.vocab + rows) * wl.hidden_dim * esz(wl) + rows * 16


def lazy_work(wl, row_max):
    """Rows the lazy schedule computed (row_max not NaN) and the tree levels they
    span (one W pass each)."""
    reach = ~np.isnan(row_max)
    depth = np.zeros(wl.T, np.int64)
    for b in range(wl.B):
        s, e = int(wl.cu_nodes[b]), int(wl.cu_nodes[b + 1])
        for i in range(s + 1, e):
            depth[i] = depth[s + int(wl.parent[i])] + 1
    return int(reach.sum()), int(depth[reach].max()) + 1 if reach.any() else 0


def tree_keys(parent):
    """Tree keys a node sees: its ancestors and itself (node depth + 1)."""
    depth = [0] * len(parent)
    for i in range(1, len(parent)):
        depth[i] = depth[int(parent[i])] + 1
    return sum(depth) + len(parent)


def step_flops(wl, lm_rows=None):
    """Algorithmic flops of one verify step: 4*Hq*D per (query node, visible key)
    in attention, 2*hidden*V per computed LM-head row (every row unless given)."""
    keys = 0
    for b in range(wl.B):
        s, e = int(wl.cu_nodes[b]), int(wl.cu_nodes[b + 1])
        keys += (e - s) * int(wl.ctx_len[b])
        keys += tree_keys(wl.parent[s:e])
    return 4 * keys * wl.Hq * wl.D + 2 * (wl.T if lm_rows is None else lm_rows) * wl.hidden_dim * wl.vocab


def step_bytes(wl, mean_path, lm_bytes=None):
    """Algorithmic bytes of one verify step (every input read once, outputs written)."""
    ctx = int(wl.ctx_len.sum())
    e = esz(wl)
    attn = (ctx * wl.Hkv * wl.D * 2 * e            # context K and V
            + wl.T * wl.Hkv * wl.D * 2 * e        # tree K and V
            + wl.T * wl.Hq * wl.D * 2 * e)        # Q read, O written
    commit = mean_path * wl.B * wl.Hkv * wl.D * 2 * 2 * e
    return attn + (lmhead_bytes(wl) if lm_bytes is None else lm_bytes) + commit


class Clocks:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index, enabled=True):
        self.proc = None
        self.path = None
        self.gpu_index = gpu_index
        if not enabled:
            return
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(gpu_index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        rows = []
        with open(self.path) as f:
            for r in csv.reader(f):
                if len(r) >= 9:
                    rows.append([x.strip() for x in r])
        os.unlink(self.path)
        note = None
        if not rows:
            # a timed region shorter than the sampling interval: one sample at its end
            try:
                out = subprocess.run(["nvidia-smi", "-i", str(self.gpu_index),
                                      f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits"],
                                     capture_output=True, text=True, timeout=10).stdout
                rows = [[x.strip() for x in r] for r in csv.reader(out.splitlines()) if len(r) >= 9]
                note = "timed region shorter than the 200 ms sampling interval: one sample at its end"
            except Exception:
                rows = []
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in rows for n, v in zip(names, r[5:9]) if v.lower() == "active"})
        res = {"sm_mhz": statistics.median(sm) if sm else None,
               "sm_max_mhz": max(mx) if mx else None, "reasons": reasons, "samples": len(rows)}
        if note:
            res["note"] = note
        return res


def slowest_rank(values, world, device):
    """Element-wise maximum of per-rank timings over all ranks (the job is as
    fast as its slowest replica)."""
    if world == 1:
        return list(values)
    import torch
    import torch.distributed as dist
    t = torch.tensor(values, dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(x) for x in t]


def job_value(nodes_per_rank, world, seconds):
    """Whole-job throughput: every rank verifies its own replica (weak scaling)."""
    return world * nodes_per_rank / seconds


def ranks_torch(wl, device):
    """Top-5 tokens of every parent row, for the drafted-token mixture (input
    synthesis with a torch fp32 matmul on the device, outside any timing)."""
    import torch
    rows = wl.parents_needed()
    h = torch.from_numpy(wl.hidden[rows]).to(device)
    w = torch.from_numpy(wl.w).to(device=device, dtype=torch.bfloat16)
    lg = torch.empty(len(rows), wl.vocab, device=device)
    for v0 in range(0, wl.vocab, 16384):
        lg[:, v0:v0 + 16384] = h @ w[v0:v0 + 16384].float().T
    top = torch.topk(lg, 5, dim=1).indices.cpu().numpy()
    del w, lg
    return {int(r): top[j] for j, r in enumerate(rows)}


def oracle_arrays(wl):
    return dict(q=wl.q, k_cache=wl.k_cache, v_cache=wl.v_cache, ctx_len=wl.ctx_len,
                tree_k=wl.tree_k, tree_v=wl.tree_v, parent=wl.parent, cu_nodes=wl.cu_nodes,
                page_table=wl.page_table, page_size=wl.page_size, hidden=wl.hidden, w=wl.w,
                tokens=wl.tokens)


def cores_used():
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count()


def cpu_baseline(wl, min_seconds=10.0, max_reps=200):
    """The oracle's whole verify step on the full workload, repeated until at
    least `min_seconds` of host time have passed."""
    import oracle
    arrays = oracle_arrays(wl)
    t0 = time.perf_counter()
    reps = 0
    while True:
        oracle.verify_step(arrays, TAU)
        reps += 1
        el = time.perf_counter() - t0
        if el >= min_seconds or reps >= max_reps:
            break
    return {"value": reps * wl.T / el, "unit": UNIT, "cores": cores_used(), "kind": "oracle",
            "sample": f"{reps} full verify step(s) of the same workload ({wl.T} nodes, full vocab "
                      f"and context) by the fp64 numpy oracle, {el:.1f} s"}


def run_reference(args):
    """The fp64 oracle as the reference arm, on a bounded sample per step."""
    import oracle
    from paper_2609_02897_gb300 import synth
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    full = synth.make_workload(CONFIG)
    steps, warm = args.steps, args.warmup
    budget = 120.0
    target = budget / max(1, steps + warm)

    def macs(wl):
        anc = sum(len(oracle.ancestors_of(wl.parent, i)) for i in range(wl.T))
        attn = 2 * wl.Hq * wl.D * (wl.T * int(wl.ctx_len[0]) + anc)
        return attn + wl.T * wl.hidden_dim * wl.vocab

    def sample(s):
        wl = synth.make_workload(CONFIG, overrides=dict(vocab=max(64, full.vocab // s),
                                                        ctx=(max(16, 2048 // s),) * 2))
        rows = wl.parents_needed()
        top = oracle.topk_tokens(wl.hidden, wl.w, rows, 5)
        synth.attach_tokens(wl, {int(r): top[j] for j, r in enumerate(rows)})
        return wl

    s = 64
    wl = sample(s)
    t0 = time.perf_counter()
    oracle.verify_step(oracle_arrays(wl), TAU)
    t1 = time.perf_counter() - t0
    s = int(min(4096, max(1, 2 ** round(np.log2(max(1e-9, s * t1 / target))))))
    wl = sample(s)
    arrays = oracle_arrays(wl)
    for _ in range(warm):
        oracle.verify_step(arrays, TAU)
    t0 = time.perf_counter()
    for _ in range(steps):
        oracle.verify_step(arrays, TAU)
    el = time.perf_counter() - t0
    frac = macs(wl) / macs(full)
    value = full.T * frac / (el / steps)
    desc = (f"each step: the oracle's full verify step on the same tree and heads with the "
            f"vocabulary cut to {wl.vocab} rows and the context to {int(wl.ctx_len[0])} tokens "
            f"({frac:.2e} of the workload's multiply-adds); value scaled by that fraction")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": steps, "warmup": warm, "ms_per_step": 1e3 * el / steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": workload_config(full),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores_used(), "kind": "oracle",
                         "sample": desc},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }))


def run_asd(args):
    import torch
    import torch.distributed as dist

    from paper_2609_02897_gb300 import asd, synth

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    device = f"cuda:{local}"
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device(device))

    wl = synth.make_workload(CONFIG, rep=rank)
    synth.attach_tokens(wl, ranks_torch(wl, device))
    torch.cuda.empty_cache()
    is_bf16 = wl.dtype == "bf16"
    bf = torch.bfloat16 if is_bf16 else torch.float32

    def f(x):
        return torch.from_numpy(np.ascontiguousarray(x)).to(device=device, dtype=bf)

    def i(x):
        return torch.from_numpy(np.ascontiguousarray(x, dtype=np.int32)).to(device)

    inputs = dict(q=f(wl.q), tree_k=f(wl.tree_k), tree_v=f(wl.tree_v), hidden=f(wl.hidden),
                  tokens=i(wl.tokens), parent=i(wl.parent), cu_nodes=i(wl.cu_nodes),
                  ctx_len=i(wl.ctx_len))
    if wl.page_table is not None:
        inputs["page_table"] = i(wl.page_table)
    # the step's inputs live in one device buffer (256-byte aligned views), so
    # that a step's inputs arrive in one host-to-device copy
    offs, off = {}, 0
    for k2, v in inputs.items():
        offs[k2] = off
        off = (off + v.numel() * v.element_size() + 255) // 256 * 256
    in_arena = torch.empty(off, dtype=torch.uint8, device=device)
    for k2, v in list(inputs.items()):
        nb = v.numel() * v.element_size()
        view = in_arena[offs[k2]:offs[k2] + nb].view(v.dtype).view(v.shape)
        view.copy_(v)
        inputs[k2] = view
    k_cache, v_cache = f(wl.k_cache), f(wl.v_cache)
    packed = args.lm_layout == "packed" and is_bf16   # the packed layout is bf16 only
    dims = asd.make_dims(wl.B, wl.Hq, wl.Hkv, wl.D, wl.hidden_dim, wl.vocab,
                         asd.ASD_BF16 if is_bf16 else asd.ASD_F32, wl.page_size,
                         wl.ctx_max, wl.num_pages, int(np.diff(wl.cu_nodes).max()), wl.max_path,
                         asd.ASD_LM_PACKED if packed else asd.ASD_LM_ROWS)
    lazy = args.lm_schedule == "lazy"
    if lazy:
        dims.lm_head_schedule = asd.ASD_LM_LAZY_LEVELS
    w_lm = f(wl.w)
    if packed:
        # model load: the LM-head weight is repacked once into the streaming layout
        w_rows = w_lm
        w_lm = asd.pack_lm_head(dims, w_rows)
        torch.cuda.synchronize()
        del w_rows
        torch.cuda.empty_cache()
    step = asd.VerifyStep(dims, wl.T, device=device, attn_dtype=bf)
    step.bind(w_lm=w_lm, k_cache=k_cache, v_cache=v_cache, tau=TAU, **inputs)
    stream = torch.cuda.current_stream()

    K, W = args.steps, args.warmup
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(5)] for _ in range(K)]
    for row in evs:
        for e in row:
            e.record(stream)   # creates the underlying CUDA events
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    clocks = Clocks(local, enabled=not args.no_clocks)
    for _ in range(W):
        step.run(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    # timed region: K back-to-back steps; consecutive kernels overlap through
    # programmatic dependent launch, so no events sit between them
    t_start.record(stream)
    for k in range(K):
        step.run(stream)
    t_end.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    status = step.device_status()
    if status != 0:
        raise RuntimeError(f"device status {asd.STATUS.get(status, status)}")
    ms = t_start.elapsed_time(t_end) / K

    # second timed region (same K): events at the stage boundaries of every
    # step give each kernel's own duration; an event between two kernels
    # serialises them, so this region is slower than the one above
    torch.cuda.synchronize()
    for k in range(K):
        for j in range(5):
            step.args.stage_events[j] = evs[k][j].cuda_event
        step.run(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    for j in range(5):
        step.args.stage_events[j] = None
    stage = np.array([[evs[k][j].elapsed_time(evs[k][j + 1]) for j in range(4)] for k in range(K)])
    stage_ms = stage.mean(axis=0)
    staged_ms = float(np.mean([evs[k][0].elapsed_time(evs[k][4]) for k in range(K)]))
    lm_ms = float(stage_ms[STAGES.index("lmhead")])
    ms, lm_ms = slowest_rank([ms, lm_ms], world, device)
    mean_path = float(step.out["path_len"].float().mean())

    # end to end through the public API: per step, H2D of the step's inputs
    # from pinned host memory, the verify step, D2H of its results, host sync
    e2e = None
    if not args.no_e2e:
        # the inputs' pinned host mirror and the results (path, path_len, bonus,
        # n_promoted, ctx_len_out, accept, row_lse: the head of the output arena)
        host_in = in_arena.cpu().pin_memory()
        host_out = torch.empty_like(step.results, device="cpu").pin_memory()
        h2d = host_in.numel()
        d2h = host_out.numel()
        for j in range(5):
            step.args.stage_events[j] = None
        # one CUDA graph per step: H2D of every input from pinned host memory, the
        # verify step, D2H of the results; the host replays it and waits for it
        graph = step.capture([(in_arena, host_in)], [(host_out, step.results)])
        for _ in range(min(W, 20)):
            graph.replay()
            stream.synchronize()
        if world > 1:
            dist.barrier()
        t0 = time.perf_counter()
        for _ in range(K):
            graph.replay()
            stream.synchronize()
        e2e_s = (time.perf_counter() - t0) / K
        (e2e_s,) = slowest_rank([e2e_s], world, device)
        e2e = {"value": job_value(wl.T, world, e2e_s), "unit": UNIT, "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "us_per_step": 1e6 * e2e_s,
               "mode": "per step: one CUDA-graph replay (H2D of the inputs from pinned host "
                       "memory, the verify step, D2H of the results) and a host sync"}

    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return
    peak, peak_kind = peaks()
    lm_rows, lm_passes = wl.T, 1
    if lazy:
        lm_rows, lm_passes = lazy_work(wl, step.out["row_max"].float().cpu().numpy())
    lmb = lmhead_bytes(wl, lm_rows, lm_passes)
    achieved = lmb / (lm_ms * 1e-3) / 1e9
    sb = step_bytes(wl, mean_path, lmb)
    fl = step_flops(wl, lm_rows)
    tpk, tpk_kind = tensor_peak()
    t_bytes, t_flops = sb / (peak * 1e9), fl / (tpk * 1e12)
    lm_flops = 2 * lm_rows * wl.hidden_dim * wl.vocab
    # up to one 128-node tile: the weight-streaming kernel; more: the wide one
    lm_kernel = "lmhead_tc_kernel" if wl.T <= 128 else "lmhead_wide_kernel"
    if wl.dtype != "bf16":
        lm_kernel = "lmhead_f32_kernel"
    if lazy:
        lm_kernel = (f"lmhead_wide_kernel + lazy_level_kernel, {lm_passes} non-empty levels of "
                     f"{wl.max_path} (LM-head stage total)")
    if lm_flops / lmb <= (tpk * 1e12) / (peak * 1e9):
        lm_roofline = {"kernel": lm_kernel, "bound": "hbm", "achieved": achieved,
                       "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                       "peak_source": peak_kind + " hbm_gbs (MEASURED_PEAKS.json)",
                       "algorithmic_bytes_per_launch": lmb, "avg_launch_us": 1e3 * lm_ms,
                       "traffic": LMHEAD_TRAFFIC_BY_CONFIG.get(CONFIG) if packed and not lazy else None}
    else:
        tf = lm_flops / (lm_ms * 1e-3) / 1e12
        lm_roofline = {"kernel": lm_kernel, "bound": "tensor", "achieved": tf,
                       "peak": tpk, "unit": "TFLOP/s", "frac": tf / tpk,
                       "peak_source": tpk_kind + " bf16_tflops (MEASURED_PEAKS.json)",
                       "algorithmic_flops_per_launch": lm_flops, "avg_launch_us": 1e3 * lm_ms,
                       "traffic": LMHEAD_TRAFFIC_BY_CONFIG.get(CONFIG) if packed and not lazy else None}
    line = {
        "metric": METRIC, "value": job_value(wl.T, world, ms * 1e-3), "unit": UNIT, "n_gpus": world,
        "steps": K, "warmup": W, "ms_per_step": ms, "us_per_step": 1e3 * ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16" if is_bf16 else "f32",
        "data": "synthetic (seeded; Llama-3.1-8B-shaped tensors, random weights)",
        "config": workload_config(wl),
        "lm_head_weight": ("packed once at load by asd_pack_lm_head (same bytes, streaming order)"
                           if packed else "[vocab, hidden] rows"),
        "lm_head_schedule": (f"lazy levels: {lm_rows} of {wl.T} rows computed, {lm_passes} W passes"
                             if lazy else "every row"),
        "hbm_gbs": sb / (ms * 1e-3) / 1e9, "hbm_frac_of_" + peak_kind: sb / (ms * 1e-3) / 1e9 / peak,
        # the whole step against the binding resource: the time its bytes take at
        # the measured copy bandwidth or its flops at the measured bf16 rate
        "step_bound": {"binding": "hbm" if t_bytes >= t_flops else "tensor",
                       "bytes": sb, "flops": fl, "t_bytes_us": 1e6 * t_bytes,
                       "t_flops_us": 1e6 * t_flops,
                       "frac": max(t_bytes, t_flops) / (ms * 1e-3),
                       "peaks": f"{peak_kind} hbm_gbs {peak}, {tpk_kind} bf16_tflops {tpk}"},
        "roofline": lm_roofline,
        "stages_us": {**{name: 1e3 * stage_ms[j] for j, name in enumerate(STAGES)},
                      "step_with_stage_events": 1e3 * staged_ms,
                      "note": "second timed region with events between kernels (no overlap)"},
        "mean_path_len": mean_path,
        # every rank's launches in the timed region (the whole job, like `value`)
        "gpu_launches": world * K * (N_STAGE_KERNELS + (1 + 2 * wl.max_path - 1 if lazy else 0)),
        "clocks": clk,
        "e2e": e2e,
    }
    if world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(wl)
    print(json.dumps(line))
    if world > 1:
        dist.destroy_process_group()


def main():
    global CONFIG, TAU
    args = parse()
    from paper_2609_02897_gb300 import synth
    if args.config not in synth.WORKLOADS:
        raise SystemExit(f"unknown workload {args.config}")
    if args.config != CONFIG:
        args.no_cpu_baseline = True   # the oracle's full step is far too slow beyond the headline
    CONFIG = args.config
    TAU = args.tau if args.tau is not None else synth.WORKLOADS[CONFIG]["tau"][0]
    if args.impl == "reference":
        run_reference(args)
    else:
        run_asd(args)


if __name__ == "__main__":
    main()
