"""Device-side test helpers (need torch.cuda and the built library)."""
from __future__ import annotations

import numpy as np
import torch

from paper_2609_02897_gb300 import asd


def dtype_of(wl):
    return torch.bfloat16 if wl.dtype == "bf16" else torch.float32


def to_device(wl, device="cuda"):
    dt = dtype_of(wl)

    def f(x):
        return torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).to(device=device, dtype=dt)

    def i(x):
        return torch.from_numpy(np.ascontiguousarray(x, dtype=np.int32)).to(device)

    d = dict(q=f(wl.q), tree_k=f(wl.tree_k), tree_v=f(wl.tree_v), k_cache=f(wl.k_cache),
             v_cache=f(wl.v_cache), hidden=f(wl.hidden), w_lm=f(wl.w), tokens=i(wl.tokens),
             parent=i(wl.parent), cu_nodes=i(wl.cu_nodes), ctx_len=i(wl.ctx_len),
             page_table=None if wl.page_table is None else i(wl.page_table))
    return d


def dims_of(wl, max_path=None, max_nodes=None):
    return asd.make_dims(
        wl.B, wl.Hq, wl.Hkv, wl.D, wl.hidden_dim, wl.vocab,
        asd.ASD_BF16 if wl.dtype == "bf16" else asd.ASD_F32, wl.page_size, wl.ctx_max,
        wl.num_pages, max_nodes or max(int(np.diff(wl.cu_nodes).max()), 1),
        max_path or wl.max_path)


def run_verify(wl, tau, dev=None, stream=None, rule=0, schedule=0):
    dev = dev or to_device(wl)
    dims = dims_of(wl)
    dims.accept_rule = rule
    dims.lm_head_schedule = schedule
    step = asd.VerifyStep(dims, wl.T, attn_dtype=dtype_of(wl))
    step.bind(tau=tau, **dev)
    step.run(stream)
    torch.cuda.synchronize()
    status = step.device_status()
    out = {k: v.float().cpu().numpy() if v.is_floating_point() else v.cpu().numpy()
           for k, v in step.out.items()}
    out["k_cache"] = dev["k_cache"].float().cpu().numpy()
    out["v_cache"] = dev["v_cache"].float().cpu().numpy()
    return out, status, step, dev
