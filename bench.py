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
# DRAM bytes (read + write) of one LM-head launch, per workload, from an ncu
# capture of the LM-head kernels built from the sources whose content hash is
# LMHEAD_TRAFFIC_SOURCE; the line reports null once those sources differ.
LMHEAD_TRAFFIC_BY_CONFIG = {2: 1054423296, 3: 2100518656}
LMHEAD_TRAFFIC_SOURCE = "9e040dc97b38edd1"
LMHEAD_SOURCES = ("lmhead_tc.cu", "lm_epilogue.cuh", "tc.cuh", "common.cuh", "kernels.h")
BAND, TIE = 1e-3, 1e-4   # the reported (not counted) band around tau; near-tie rows
WORKLOADS_BLOCK = (3, 4, 5)   # the tensor-bound workloads timed after the headline


def lmhead_source_hash():
    """sha256 (first 16 hex digits) of the LM-head kernel sources as built."""
    import hashlib
    h = hashlib.sha256()
    d = os.path.join(ROOT, "paper_2609_02897_gb300", "csrc")
    for name in LMHEAD_SOURCES:
        with open(os.path.join(d, name), "rb") as f:
            h.update(name.encode() + b"\0" + f.read())
    return h.hexdigest()[:16]


def lmhead_traffic(config):
    """The captured DRAM bytes per LM-head launch, or None when the kernel
    sources changed since the capture."""
    if LMHEAD_TRAFFIC_SOURCE is None or lmhead_source_hash() != LMHEAD_TRAFFIC_SOURCE:
        return None
    return LMHEAD_TRAFFIC_BY_CONFIG.get(config)


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
    ap.add_argument("--no-workloads", action="store_true",
                    help="skip the tensor-bound workloads timed after the headline")
    ap.add_argument("--batch", type=int, default=None,
                    help="draw the workload with B sequences (a smaller case of the same shapes, "
                         "e.g. for a profiler capture)")
    ap.add_argument("--oracle-one-step", default=None, help=argparse.SUPPRESS)
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
    least `min_seconds` of host time have passed.  Returns the baseline and the
    first step's outputs (the in-run parity check compares them with the GPU's)."""
    import oracle
    arrays = oracle_arrays(wl)
    t0 = time.perf_counter()
    reps = 0
    first = None
    while True:
        r = oracle.verify_step(arrays, TAU)
        first = r if first is None else first
        reps += 1
        el = time.perf_counter() - t0
        if el >= min_seconds or reps >= max_reps:
            break
    return ({"value": reps * wl.T / el, "unit": UNIT, "cores": cores_used(), "kind": "oracle",
             "sample": f"{reps} full verify step(s) of the same workload ({wl.T} nodes, full vocab "
                       f"and context) by the fp64 numpy oracle, {el:.1f} s"}, first)


THREAD_VARS = ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS",
               "BLIS_NUM_THREADS", "VECLIB_MAXIMUM_THREADS", "NUMEXPR_NUM_THREADS")


def oracle_single_thread(wl, tau=None):
    """One oracle verify step of the same workload on one host core: a child
    process (BLAS threads 1, pinned to one core) redraws the workload from its
    seed, takes the drafted tokens from a file and times one step."""
    fd, path = tempfile.mkstemp(suffix=".npy")
    os.close(fd)
    try:
        np.save(path, wl.tokens)
        env = dict(os.environ, **{v: "1" for v in THREAD_VARS})
        r = subprocess.run([sys.executable, os.path.abspath(__file__), "--oracle-one-step", path,
                            "--config", str(wl.config), "--tau", repr(TAU if tau is None else tau)],
                           env=env, capture_output=True, text=True, timeout=900)
        if r.returncode != 0:
            return {"error": (r.stderr or r.stdout).strip().splitlines()[-1:]}
        t = json.loads(r.stdout.strip().splitlines()[-1])["seconds"]
    finally:
        os.unlink(path)
    return {"value": wl.T / t, "unit": UNIT, "cores": 1, "kind": "oracle", "seconds_per_step": t,
            "sample": "one full verify step of the same workload by the fp64 numpy oracle, "
                      "BLAS threads 1, pinned to one core"}


def oracle_one_step(tokens_path, config, tau):
    """Child of oracle_single_thread: prints the seconds of one oracle step."""
    try:
        os.sched_setaffinity(0, {min(os.sched_getaffinity(0))})
    except Exception:
        pass
    import oracle
    from paper_2609_02897_gb300 import synth
    wl = synth.make_workload(config)
    wl.tokens = np.load(tokens_path)
    arrays = oracle_arrays(wl)
    t0 = time.perf_counter()
    oracle.verify_step(arrays, tau)
    print(json.dumps({"seconds": time.perf_counter() - t0}))


def parity_check(wl, tau, out, cache_rows, full=None, seqs=None):
    """The timed step's outputs against the oracle on the same inputs.

    full: the oracle's verify step on the whole workload (cpu_baseline's first
    step); otherwise the oracle recomputes the sequences `seqs` (attention of
    all their nodes, their LM-head rows over the full vocabulary, their paths).
    Floating-point outputs within 2e-2 absolute + 1e-2 relative of the oracle
    (bf16; 1e-4 + 1e-4 for fp32), the Eq. 1 ratio within 5e-2 relative;
    argmax, accept, path, bonus, n_promoted and the committed K/V rows exact,
    except the reported band: non-strict nodes whose oracle ratio lies within
    1e-3 of tau and children of rows whose top-2 logits differ by < 1e-4; a
    sequence touching the band is checked for a valid longest path instead.
    `cache_rows(b, slot)` returns the GPU cache's (K, V) of one slot."""
    import oracle
    atol, rtol = (2e-2, 1e-2) if wl.dtype == "bf16" else (1e-4, 1e-4)
    seqs = list(range(wl.B)) if seqs is None else list(seqs)
    nodes = np.concatenate([np.arange(wl.cu_nodes[b], wl.cu_nodes[b + 1]) for b in seqs])
    gp = wl.global_parent()
    if full is not None:
        attn, lm = full["attn"], full
    else:
        attn = oracle.tree_attention(wl.q, wl.k_cache, wl.v_cache, wl.ctx_len, wl.tree_k,
                                     wl.tree_v, wl.parent, wl.cu_nodes, wl.page_table,
                                     wl.page_size, nodes=nodes)
        lm = oracle.lmhead_margin(wl.hidden, wl.w, wl.tokens, wl.parent, wl.cu_nodes, tau,
                                  rows=nodes)
    failed, max_err = [], {}

    def close(name, got, ref, a, r):
        got, ref = np.asarray(got, np.float64), np.asarray(ref, np.float64)
        e = np.abs(got - ref)
        max_err[name] = float(np.max(e)) if e.size else 0.0
        if not np.all(e <= a + r * np.abs(ref)):
            failed.append(name)

    close("attn", out["attn_out"][nodes], attn[nodes], atol, rtol)
    close("row_max", out["row_max"][nodes], lm["row_max"][nodes], atol, rtol)
    close("row_lse", out["row_lse"][nodes], lm["row_lse"][nodes], atol, rtol)
    tie = set()
    for i in range(0, len(nodes), 256):
        chunk = nodes[i:i + 256]
        part = np.partition(oracle.logits_rows(wl.hidden, wl.w, chunk), -2, axis=1)[:, -2:]
        tie.update(int(r) for r, g in zip(chunk, part[:, 1] - part[:, 0]) if g < TIE)
    if any(int(out["row_argmax"][r]) != int(lm["row_argmax"][r]) for r in nodes
           if int(r) not in tie):
        failed.append("row_argmax")
    kids = np.array([c for c in nodes if gp[c] >= 0], dtype=np.int64)
    band = set()
    if len(kids):
        close("l_draft", out["l_draft"][kids], lm["l_draft"][kids], atol, rtol)
        close("ratio", out["ratio"][kids], lm["ratio"][kids], 1e-6, 5e-2)
        for c in kids:
            strict = int(wl.tokens[c]) == int(lm["row_argmax"][gp[c]])
            if (abs(lm["ratio"][c] - tau) < BAND and not strict) or int(gp[c]) in tie:
                band.add(int(c))
            elif int(out["accept"][c]) != int(lm["accept"][c]):
                failed.append(f"accept[{int(c)}]")
    checked = excluded = 0
    for b in seqs:
        s, e = int(wl.cu_nodes[b]), int(wl.cu_nodes[b + 1])
        plen = int(out["path_len"][b])
        path = [int(x) for x in out["path"][b][:plen]]
        if band.intersection(range(s, e)):
            excluded += 1
            ok = path and path[0] == 0 and all(
                int(wl.parent[s + y]) == x and int(out["accept"][s + y]) == 1
                for x, y in zip(path[:-1], path[1:]))
            if not ok:
                failed.append(f"path[{b}]")
        else:
            checked += 1
            if full is not None:
                ref_path, bonus, npro = full["paths"][b], full["bonus"][b], full["n_promoted"][b]
            else:
                rp, _, rb, rn = oracle.accept_path(wl.parent[s:e], lm["accept"][s:e],
                                                   lm["row_argmax"][s:e], wl.tokens[s:e],
                                                   [0, e - s], ratio=lm["ratio"][s:e])
                ref_path, bonus, npro = rp[0], rb[0], rn[0]
            if path != [int(x) for x in ref_path] or int(out["bonus"][b]) != int(bonus) or \
                    int(out["n_promoted"][b]) != int(npro):
                failed.append(f"path[{b}]")
        if int(out["ctx_len_out"][b]) != int(wl.ctx_len[b]) + plen:
            failed.append(f"ctx_len_out[{b}]")
        for k, u in enumerate(path):
            kc, vc = cache_rows(b, int(wl.ctx_len[b]) + k)
            if not (np.array_equal(kc, wl.tree_k[s + u]) and np.array_equal(vc, wl.tree_v[s + u])):
                failed.append(f"commit[{b},{k}]")
    return {"ok": not failed, "failed": failed[:8], "oracle": "fp64 oracle on the same inputs, "
            + ("whole step (the cpu_baseline's first step)" if full is not None
               else f"sequences {seqs} recomputed"),
            "band_nodes": len(band), "tie_rows": len(tie), "checked_seqs": checked,
            "excluded_seqs": excluded, "max_err": max_err}


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


def device_step(wl, device, tau, packed=True, lazy=False):
    """Device copies of one workload's inputs (the step's inputs in one buffer,
    so that one host-to-device copy brings them), the LM-head weight (packed once
    at load unless `packed` is false) and a bound VerifyStep."""
    import torch
    from paper_2609_02897_gb300 import asd
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
    offs, off = {}, 0
    for k, v in inputs.items():
        offs[k] = off
        off = (off + v.numel() * v.element_size() + 255) // 256 * 256
    in_arena = torch.empty(off, dtype=torch.uint8, device=device)
    for k, v in list(inputs.items()):
        nb = v.numel() * v.element_size()
        view = in_arena[offs[k]:offs[k] + nb].view(v.dtype).view(v.shape)
        view.copy_(v)
        inputs[k] = view
    k_cache, v_cache = f(wl.k_cache), f(wl.v_cache)
    packed = packed and is_bf16   # the packed layout is bf16 only
    dims = asd.make_dims(wl.B, wl.Hq, wl.Hkv, wl.D, wl.hidden_dim, wl.vocab,
                         asd.ASD_BF16 if is_bf16 else asd.ASD_F32, wl.page_size,
                         wl.ctx_max, wl.num_pages, int(np.diff(wl.cu_nodes).max()), wl.max_path,
                         asd.ASD_LM_PACKED if packed else asd.ASD_LM_ROWS)
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
    step.bind(w_lm=w_lm, k_cache=k_cache, v_cache=v_cache, tau=tau, **inputs)
    return step, in_arena, packed


def time_region(step, stream, K):
    """K back-to-back steps between two events (consecutive kernels overlap
    through programmatic dependent launch, so no events sit between them); ms
    per step."""
    import torch
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for _ in range(K):
        step.run(stream)
    t1.record(stream)
    torch.cuda.synchronize()
    return t0.elapsed_time(t1) / K


def time_stages(step, stream, K):
    """K steps with events at the stage boundaries of every step: each kernel's
    own duration (an event between two kernels serialises them, so these steps
    are slower than the ones of time_region).  Returns (mean ms per stage, mean
    ms per step)."""
    import torch
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(5)] for _ in range(K)]
    for row in evs:
        for e in row:
            e.record(stream)   # creates the underlying CUDA events
    torch.cuda.synchronize()
    for k in range(K):
        for j in range(5):
            step.args.stage_events[j] = evs[k][j].cuda_event
        step.run(stream)
    torch.cuda.synchronize()
    for j in range(5):
        step.args.stage_events[j] = None
    stage = np.array([[evs[k][j].elapsed_time(evs[k][j + 1]) for j in range(4)] for k in range(K)])
    return stage.mean(axis=0), float(np.mean([evs[k][0].elapsed_time(evs[k][4]) for k in range(K)]))


def outputs_numpy(step):
    return {k: v.float().cpu().numpy() if v.is_floating_point() else v.cpu().numpy()
            for k, v in step.out.items()}


def cache_reader(wl, step):
    """(K, V) of one cache slot of sequence b as the GPU holds it."""
    a = step._keep
    kc, vc = a[9], a[10]

    def rows(b, slot):
        if wl.page_size == 0:
            return kc[b, :, slot].float().cpu().numpy(), vc[b, :, slot].float().cpu().numpy()
        page = int(wl.page_table[b, slot // wl.page_size])
        o = slot % wl.page_size
        return kc[page, :, o].float().cpu().numpy(), vc[page, :, o].float().cpu().numpy()
    return rows


def roofline_of(wl, lm_ms, lm_rows, lm_passes, peak, peak_kind, tpk, tpk_kind, kernel, traffic):
    """The LM head against its binding resource: its algorithmic bytes at the
    measured copy bandwidth, or its flops at the measured bf16 rate."""
    lmb = lmhead_bytes(wl, lm_rows, lm_passes)
    lm_flops = 2 * lm_rows * wl.hidden_dim * wl.vocab
    if lm_flops / lmb <= (tpk * 1e12) / (peak * 1e9):
        achieved = lmb / (lm_ms * 1e-3) / 1e9
        return {"kernel": kernel, "bound": "hbm", "achieved": achieved, "peak": peak,
                "unit": "GB/s", "frac": achieved / peak,
                "peak_source": peak_kind + " hbm_gbs (MEASURED_PEAKS.json)",
                "algorithmic_bytes_per_launch": lmb, "avg_launch_us": 1e3 * lm_ms,
                "traffic": traffic}
    tf = lm_flops / (lm_ms * 1e-3) / 1e12
    return {"kernel": kernel, "bound": "tensor", "achieved": tf, "peak": tpk, "unit": "TFLOP/s",
            "frac": tf / tpk, "peak_source": tpk_kind + " bf16_tflops (MEASURED_PEAKS.json)",
            "algorithmic_flops_per_launch": lm_flops, "avg_launch_us": 1e3 * lm_ms,
            "traffic": traffic}


def lm_kernel_name(step):
    """The LM-head kernel the library runs for this step (its own answer)."""
    from paper_2609_02897_gb300 import asd
    v = asd.asd_lm_head_variant(step.dims, step.T, step._keep[4])
    return asd.LM_HEAD_VARIANTS.get(v, f"variant {v}")


def workloads_block(device, stream, steps=10, warmup=3):
    """The tensor-bound workloads (ragged B16, Qwen3-8B B8 ctx 16384, paged
    B64 ctx 8192), each timed over a few steps after the headline: us per step,
    the binding resource and the fraction of it, the LM head against its own
    bound, the device status, and parity on one sequence recomputed by the
    oracle."""
    import torch
    from paper_2609_02897_gb300 import synth
    peak, peak_kind = peaks()
    tpk, tpk_kind = tensor_peak()
    res = {}
    for cfg in WORKLOADS_BLOCK:
        t_gen = time.perf_counter()
        wl = synth.make_workload(cfg)
        synth.attach_tokens(wl, ranks_torch(wl, device))
        tau = synth.WORKLOADS[cfg]["tau"][0]
        step, _, _ = device_step(wl, device, tau)
        t_gen = time.perf_counter() - t_gen
        for _ in range(warmup):
            step.run(stream)
        torch.cuda.synchronize()
        ms = time_region(step, stream, steps)
        stage_ms, _ = time_stages(step, stream, steps)
        status = step.device_status()
        out = outputs_numpy(step)
        mean_path = float(out["path_len"].mean())
        par = parity_check(wl, tau, out, cache_reader(wl, step), seqs=[0])
        sb, fl = step_bytes(wl, mean_path), step_flops(wl)
        t_bytes, t_flops = sb / (peak * 1e9), fl / (tpk * 1e12)
        lm_ms = float(stage_ms[STAGES.index("lmhead")])
        res[wl.name] = {
            "config": cfg, "batch": wl.B, "tree_nodes": wl.T, "tau": tau,
            "us_per_step": 1e3 * ms, "value": wl.T / (ms * 1e-3), "unit": UNIT,
            "steps": steps, "warmup": warmup, "device_status": status,
            "step_bound": {"binding": "hbm" if t_bytes >= t_flops else "tensor",
                           "frac": max(t_bytes, t_flops) / (ms * 1e-3),
                           "t_bytes_us": 1e6 * t_bytes, "t_flops_us": 1e6 * t_flops},
            "stages_us": {name: 1e3 * stage_ms[j] for j, name in enumerate(STAGES)},
            "roofline": roofline_of(wl, lm_ms, wl.T, 1, peak, peak_kind, tpk, tpk_kind,
                                    lm_kernel_name(step), lmhead_traffic(cfg)),
            "mean_path_len": mean_path, "parity": par, "setup_s": t_gen,
        }
        del step, out
        torch.cuda.empty_cache()
    # the tiny fp32 workload (parity case): its step time and the oracle on one core
    wl = synth.make_workload(1)
    synth.attach_tokens(wl, ranks_torch(wl, device))
    tau = synth.WORKLOADS[1]["tau"][0]
    step, _, _ = device_step(wl, device, tau)
    for _ in range(warmup):
        step.run(stream)
    torch.cuda.synchronize()
    ms = time_region(step, stream, 10 * steps)
    out = outputs_numpy(step)
    single = oracle_single_thread(wl, tau)
    res[wl.name] = {
        "config": 1, "batch": wl.B, "tree_nodes": wl.T, "tau": tau, "dtype": "f32",
        "us_per_step": 1e3 * ms, "value": wl.T / (ms * 1e-3), "unit": UNIT,
        "steps": 10 * steps, "device_status": step.device_status(),
        "parity": parity_check(wl, tau, out, cache_reader(wl, step)),
        "cpu_baseline_single_thread": single,
    }
    del step
    return {"note": "tensor-bound workloads, each a short timed loop after the headline "
                    "(burst regime: fractions against the burst bf16 peak); inputs larger than "
                    "L2 (the LM-head weight is streamed every step); and the tiny fp32 "
                    "workload with the oracle timed on one core", **res}


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

    wl = synth.make_workload(CONFIG, rep=rank,
                             overrides=dict(B=args.batch) if args.batch else None)
    synth.attach_tokens(wl, ranks_torch(wl, device))
    torch.cuda.empty_cache()
    is_bf16 = wl.dtype == "bf16"
    lazy = args.lm_schedule == "lazy"
    step, in_arena, packed = device_step(wl, device, TAU, packed=args.lm_layout == "packed",
                                         lazy=lazy)
    stream = torch.cuda.current_stream()

    K, W = args.steps, args.warmup
    clocks = Clocks(local, enabled=not args.no_clocks)
    for _ in range(W):
        step.run(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    ms = time_region(step, stream, K)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    status = step.device_status()
    if status != 0:
        raise RuntimeError(f"device status {asd.STATUS.get(status, status)}")
    stage_ms, staged_ms = time_stages(step, stream, K)
    clk = clocks.stop()
    lm_ms = float(stage_ms[STAGES.index("lmhead")])
    ms, lm_ms = slowest_rank([ms, lm_ms], world, device)
    out = outputs_numpy(step)
    mean_path = float(out["path_len"].mean())

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
    tpk, tpk_kind = tensor_peak()
    lm_rows, lm_passes = wl.T, 1
    if lazy:
        lm_rows, lm_passes = lazy_work(wl, out["row_max"])
    lmb = lmhead_bytes(wl, lm_rows, lm_passes)
    sb = step_bytes(wl, mean_path, lmb)
    fl = step_flops(wl, lm_rows)
    t_bytes, t_flops = sb / (peak * 1e9), fl / (tpk * 1e12)
    lm_kernel = lm_kernel_name(step)
    if lazy:
        lm_kernel = (f"lmhead_wide_kernel + lazy_level_kernel, {lm_passes} non-empty levels of "
                     f"{wl.max_path} (LM-head stage total)")
    traffic = lmhead_traffic(CONFIG) if packed and not lazy else None
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
        "roofline": roofline_of(wl, lm_ms, lm_rows, lm_passes, peak, peak_kind, tpk, tpk_kind,
                                lm_kernel, traffic),
        "stages_us": {**{name: 1e3 * stage_ms[j] for j, name in enumerate(STAGES)},
                      "step_with_stage_events": 1e3 * staged_ms,
                      "note": "second timed region with events between kernels (no overlap)"},
        "mean_path_len": mean_path,
        # every rank's launches in the timed region (the whole job, like `value`)
        "gpu_launches": world * K * (N_STAGE_KERNELS + (1 + 2 * wl.max_path - 1 if lazy else 0)),
        "clocks": clk,
        "e2e": e2e,
    }
    full_ref = None
    if world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"], full_ref = cpu_baseline(wl)
        line["cpu_baseline_single_thread"] = oracle_single_thread(wl)
    if not lazy:
        # the timed step's own outputs against the oracle on the same inputs
        seqs = None if (full_ref is not None or wl.T <= 128) else [0]
        line["parity"] = parity_check(wl, TAU, out, cache_reader(wl, step), full=full_ref,
                                      seqs=seqs)
    if world == 1 and CONFIG == 2 and not args.no_workloads:
        del step
        torch.cuda.empty_cache()
        line["workloads"] = workloads_block(device, stream)
    print(json.dumps(line))
    if world > 1:
        dist.destroy_process_group()


def main():
    global CONFIG, TAU
    args = parse()
    from paper_2609_02897_gb300 import synth
    if args.config not in synth.WORKLOADS:
        raise SystemExit(f"unknown workload {args.config}")
    if args.oracle_one_step:
        oracle_one_step(args.oracle_one_step, args.config, args.tau)
        return
    if args.config != CONFIG or args.batch:
        args.no_cpu_baseline = True   # the oracle's full step is far too slow beyond the headline
        args.no_workloads = True
    if int(os.environ.get("WORLD_SIZE", "1")) > 1 and args.config != CONFIG:
        # replicas on several GPUs run the headline workload only: the wide LM
        # head's clustered form (steps of more than 768 nodes) serves 1-GPU runs
        raise SystemExit("several GPUs: only the headline workload (--config 2) is run")
    CONFIG = args.config
    TAU = args.tau if args.tau is not None else synth.WORKLOADS[CONFIG]["tau"][0]
    if args.impl == "reference":
        run_reference(args)
    else:
        run_asd(args)


if __name__ == "__main__":
    main()
