"""ctypes binding of libasd (include/asd.h).  Argument marshalling only: every
step of the verify path runs in the library's CUDA kernels.  Tensors are torch
tensors used as device memory; the stream defaults to torch's current stream.

Importing this module loads libasd.so and raises ImportError if it has not
been built (paper_2609_02897_gb300.build.build()).  There is no fallback.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

import torch

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "_lib", "libasd.so")
if not os.path.exists(_LIB_PATH):
    raise ImportError(f"libasd is not built ({_LIB_PATH} missing); run "
                      "`python -c 'import __graft_entry__ as g; g.build()'`")
_lib = ctypes.CDLL(_LIB_PATH)

ASD_F32, ASD_BF16 = 0, 1
ASD_LM_ROWS, ASD_LM_PACKED = 0, 1
ASD_ACCEPT_LONGEST, ASD_ACCEPT_ONCE, ASD_ACCEPT_GREEDY, ASD_ACCEPT_GREEDY_ONCE = 0, 1, 2, 3
ASD_LM_EVERY_ROW, ASD_LM_LAZY_LEVELS = 0, 1
MAX_TREE_NODES = 128
NOALLOC_SCRATCH_BYTES = 8 << 20   # ASD_NOALLOC_SCRATCH_BYTES
NUM_STAGE_EVENTS = 5
STATUS = {0: "ASD_OK", 1: "ASD_ERR_INVALID_ARG", 2: "ASD_ERR_SHAPE", 3: "ASD_ERR_TREE",
          4: "ASD_ERR_TOKEN_RANGE", 5: "ASD_ERR_CTX_RANGE", 6: "ASD_ERR_WORKSPACE",
          7: "ASD_ERR_CUDA", 8: "ASD_ERR_TIMEOUT", 9: "ASD_ERR_UNSUPPORTED"}
EXPORTS = ["asd_workspace_bytes", "asd_tree_attention", "asd_lmhead_margin", "asd_accept_path",
           "asd_kv_compact", "asd_verify_step", "asd_get_device_status", "asd_status_string",
           "asd_abi_version", "asd_lmhead_margin_noalloc", "asd_lm_head_packed_bytes",
           "asd_pack_lm_head",
           "asd_policy_triplets", "asd_policy_init", "asd_policy_update", "asd_policy_select",
           "asd_debug_set_wait_cycles", "asd_lm_head_variant", "asd_attention_variant"]


class AsdError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        super().__init__(f"{where}: {STATUS.get(code, code)} "
                         f"({_lib.asd_status_string(code).decode()})")


class Dims(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "batch", "num_q_heads", "num_kv_heads", "head_dim", "hidden", "vocab", "dtype",
        "page_size", "ctx_max", "num_pages", "max_nodes", "max_path", "lm_head_layout",
        "accept_rule", "lm_head_schedule")]


_vp = ctypes.c_void_p
_i32p = ctypes.c_void_p


class VerifyArgs(ctypes.Structure):
    _fields_ = [
        ("q", _vp), ("tree_k", _vp), ("tree_v", _vp), ("hidden", _vp), ("w_lm", _vp),
        ("tokens", _vp), ("parent", _vp), ("cu_nodes", _vp), ("ctx_len", _vp),
        ("page_table", _vp), ("total_nodes", ctypes.c_int32), ("tau", ctypes.c_float),
        ("k_cache", _vp), ("v_cache", _vp),
        ("attn_out", _vp), ("row_max", _vp), ("row_argmax", _vp), ("row_lse", _vp),
        ("l_draft", _vp), ("ratio", _vp), ("accept", _vp), ("path", _vp), ("path_len", _vp),
        ("bonus", _vp), ("n_promoted", _vp), ("ctx_len_out", _vp),
        ("stage_events", _vp * NUM_STAGE_EVENTS),
    ]


class PolicyParams(ctypes.Structure):
    """asd_policy_params: the tree-shape policy's settings (Sec. 3.3)."""
    _fields_ = [("alpha", ctypes.c_double), ("divisor", ctypes.c_double),
                ("rar_init", ctypes.c_double), ("shallow", ctypes.c_int32 * 3),
                ("deep", ctypes.c_int32 * 3), ("breaker", ctypes.c_int32),
                ("reserved", ctypes.c_int32)]


POLICY_STATE_BYTES = 16


def make_policy_params(alpha=0.3, divisor=0.5, rar_init=1.0, shallow=(3, 4, 4), deep=(7, 1, 8),
                       breaker=5) -> PolicyParams:
    """Defaults: the paper's settings (Sec. 3.3, Sec. 4.2)."""
    return PolicyParams(alpha, divisor, rar_init, (ctypes.c_int32 * 3)(*shallow),
                        (ctypes.c_int32 * 3)(*deep), breaker, 0)


_P = ctypes.POINTER(Dims)
_PP = ctypes.POINTER(PolicyParams)
_lib.asd_abi_version.restype = ctypes.c_int32
_lib.asd_status_string.restype = ctypes.c_char_p
_lib.asd_status_string.argtypes = [ctypes.c_int32]
_lib.asd_workspace_bytes.restype = ctypes.c_size_t
_lib.asd_workspace_bytes.argtypes = [_P, ctypes.c_int32]
_lib.asd_tree_attention.restype = ctypes.c_int
_lib.asd_tree_attention.argtypes = [_P] + [_vp] * 9 + [ctypes.c_int32, _vp, _vp, ctypes.c_size_t, _vp]
_lib.asd_lmhead_margin.restype = ctypes.c_int
_lib.asd_lmhead_margin.argtypes = [_P] + [_vp] * 5 + [ctypes.c_int32, ctypes.c_float] + [_vp] * 6 + [
    _vp, ctypes.c_size_t, _vp]
_lib.asd_accept_path.restype = ctypes.c_int
_lib.asd_accept_path.argtypes = [_P] + [_vp] * 6 + [ctypes.c_int32] + [_vp] * 4 + [
    _vp, ctypes.c_size_t, _vp]
_lib.asd_kv_compact.restype = ctypes.c_int
_lib.asd_kv_compact.argtypes = [_P, _vp, _vp, _vp, ctypes.c_int32] + [_vp] * 7 + [
    _vp, ctypes.c_size_t, _vp]
_lib.asd_verify_step.restype = ctypes.c_int
_lib.asd_verify_step.argtypes = [_P, ctypes.POINTER(VerifyArgs), _vp, ctypes.c_size_t, _vp]
_lib.asd_lmhead_margin_noalloc.restype = ctypes.c_int
_lib.asd_lmhead_margin_noalloc.argtypes = [_P] + [_vp] * 5 + [ctypes.c_int32, ctypes.c_float] + [
    _vp] * 6 + [_vp, _vp]
_lib.asd_attention_variant.restype = ctypes.c_int32
_lib.asd_attention_variant.argtypes = [_P, ctypes.c_int32]
_lib.asd_lm_head_variant.restype = ctypes.c_int32
_lib.asd_lm_head_variant.argtypes = [_P, ctypes.c_int32, _vp]
_lib.asd_debug_set_wait_cycles.restype = ctypes.c_int
_lib.asd_debug_set_wait_cycles.argtypes = [ctypes.c_int64]
_lib.asd_get_device_status.restype = ctypes.c_int
_lib.asd_get_device_status.argtypes = [_vp, ctypes.POINTER(ctypes.c_int32), _vp]
_lib.asd_lm_head_packed_bytes.restype = ctypes.c_size_t
_lib.asd_lm_head_packed_bytes.argtypes = [_P]
_lib.asd_pack_lm_head.restype = ctypes.c_int
_lib.asd_pack_lm_head.argtypes = [_P, _vp, _vp, ctypes.c_size_t, _vp]
_lib.asd_policy_triplets.restype = ctypes.c_int32
_lib.asd_policy_triplets.argtypes = [_PP, _vp, ctypes.c_int32]
_lib.asd_policy_init.restype = ctypes.c_int
_lib.asd_policy_init.argtypes = [_PP, _vp, ctypes.c_int32, _vp]
_lib.asd_policy_update.restype = ctypes.c_int
_lib.asd_policy_update.argtypes = [_PP, _vp, _vp, ctypes.c_int32, _vp, _vp]
_lib.asd_policy_select.restype = ctypes.c_int
_lib.asd_policy_select.argtypes = [_PP, _vp, _vp, _vp, ctypes.c_int32, ctypes.c_int32, _vp, _vp,
                                   _vp, _vp]


def lib_path() -> str:
    return _LIB_PATH


def abi_version() -> int:
    return int(_lib.asd_abi_version())


def make_dims(batch, num_q_heads, num_kv_heads, head_dim, hidden, vocab, dtype, page_size,
              ctx_max, num_pages, max_nodes, max_path, lm_head_layout=0, accept_rule=0,
              lm_head_schedule=0) -> Dims:
    return Dims(batch, num_q_heads, num_kv_heads, head_dim, hidden, vocab, dtype, page_size,
                ctx_max, num_pages, max_nodes, max_path, lm_head_layout, accept_rule,
                lm_head_schedule)


def _ptr(t: Optional[torch.Tensor]):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("libasd takes device tensors")
    if not t.is_contiguous():
        raise ValueError("libasd takes contiguous tensors")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


def _check(code: int, where: str):
    if code != 0:
        raise AsdError(code, where)


def asd_workspace_bytes(dims: Dims, total_nodes: int) -> int:
    n = int(_lib.asd_workspace_bytes(ctypes.byref(dims), int(total_nodes)))
    if n == 0:
        raise AsdError(2, "asd_workspace_bytes")
    return n


def asd_lm_head_packed_bytes(dims: Dims) -> int:
    n = int(_lib.asd_lm_head_packed_bytes(ctypes.byref(dims)))
    if n == 0:
        raise AsdError(2, "asd_lm_head_packed_bytes")
    return n


def asd_pack_lm_head(dims: Dims, w: torch.Tensor, w_packed: torch.Tensor, stream=None):
    _check(_lib.asd_pack_lm_head(ctypes.byref(dims), _ptr(w), _ptr(w_packed), w_packed.numel(),
                                 _stream(stream)), "asd_pack_lm_head")


def pack_lm_head(dims: Dims, w: torch.Tensor, stream=None) -> torch.Tensor:
    """A new device buffer holding w in the LM head's packed streaming layout
    (use it with dims.lm_head_layout = ASD_LM_PACKED)."""
    out = torch.empty(asd_lm_head_packed_bytes(dims), dtype=torch.uint8, device=w.device)
    asd_pack_lm_head(dims, w, out, stream)
    return out


def alloc_workspace(dims: Dims, total_nodes: int, device="cuda") -> torch.Tensor:
    return torch.empty(asd_workspace_bytes(dims, total_nodes), dtype=torch.uint8, device=device)


def asd_tree_attention(dims, q, k_cache, v_cache, page_table, ctx_len, tree_k, tree_v, parent,
                       cu_nodes, out, workspace, stream=None):
    _check(_lib.asd_tree_attention(
        ctypes.byref(dims), _ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(page_table),
        _ptr(ctx_len), _ptr(tree_k), _ptr(tree_v), _ptr(parent), _ptr(cu_nodes),
        int(parent.numel()), _ptr(out), _ptr(workspace), workspace.numel(), _stream(stream)),
        "asd_tree_attention")


def asd_lmhead_margin(dims, hidden, w_lm, tokens, parent, cu_nodes, tau, row_max, row_argmax,
                      row_lse, l_draft, ratio, accept, workspace, stream=None):
    _check(_lib.asd_lmhead_margin(
        ctypes.byref(dims), _ptr(hidden), _ptr(w_lm), _ptr(tokens), _ptr(parent), _ptr(cu_nodes),
        int(parent.numel()), float(tau), _ptr(row_max), _ptr(row_argmax), _ptr(row_lse),
        _ptr(l_draft), _ptr(ratio), _ptr(accept), _ptr(workspace), workspace.numel(),
        _stream(stream)), "asd_lmhead_margin")


def asd_lmhead_margin_noalloc(dims, hidden, w_lm, tokens, parent, cu_nodes, tau, row_max,
                              row_argmax, row_lse, l_draft, ratio, accept, device_status=None,
                              stream=None):
    """asd_lmhead_margin with the library's static scratch instead of a workspace
    (for callers that cannot allocate device memory).  device_status: optional
    int32 device tensor that receives the device-side status word."""
    _check(_lib.asd_lmhead_margin_noalloc(
        ctypes.byref(dims), _ptr(hidden), _ptr(w_lm), _ptr(tokens), _ptr(parent), _ptr(cu_nodes),
        int(parent.numel()), float(tau), _ptr(row_max), _ptr(row_argmax), _ptr(row_lse),
        _ptr(l_draft), _ptr(ratio), _ptr(accept), _ptr(device_status), _stream(stream)),
        "asd_lmhead_margin_noalloc")


def asd_accept_path(dims, parent, tokens, accept, row_argmax, cu_nodes, path, path_len, bonus,
                    n_promoted, workspace, stream=None, ratio=None):
    _check(_lib.asd_accept_path(
        ctypes.byref(dims), _ptr(parent), _ptr(tokens), _ptr(accept), _ptr(row_argmax),
        _ptr(ratio), _ptr(cu_nodes), int(parent.numel()), _ptr(path), _ptr(path_len), _ptr(bonus),
        _ptr(n_promoted), _ptr(workspace), workspace.numel(), _stream(stream)),
        "asd_accept_path")


def asd_kv_compact(dims, tree_k, tree_v, cu_nodes, total_nodes, path, path_len, ctx_len,
                   page_table, k_cache, v_cache, ctx_len_out, workspace, stream=None):
    _check(_lib.asd_kv_compact(
        ctypes.byref(dims), _ptr(tree_k), _ptr(tree_v), _ptr(cu_nodes), int(total_nodes),
        _ptr(path), _ptr(path_len), _ptr(ctx_len), _ptr(page_table), _ptr(k_cache),
        _ptr(v_cache), _ptr(ctx_len_out), _ptr(workspace), workspace.numel(), _stream(stream)),
        "asd_kv_compact")


def asd_verify_step(dims, args: VerifyArgs, workspace, stream=None):
    _check(_lib.asd_verify_step(ctypes.byref(dims), ctypes.byref(args), _ptr(workspace),
                                workspace.numel(), _stream(stream)), "asd_verify_step")


LM_HEAD_VARIANTS = {1: "lmhead_tc_kernel", 2: "lmhead_wide_kernel", 3: "lmhead_wide_kernel (clusters of two)",
                    4: "lmhead_f32_kernel"}


def asd_lm_head_variant(dims: Dims, total_nodes: int, w_lm) -> int:
    """Which LM-head kernel a call runs (include/asd.h): 1-4, 0 for invalid
    arguments.  `w_lm`: a tensor (device or host) or a raw address."""
    ptr = ctypes.c_void_p(w_lm.data_ptr() if hasattr(w_lm, "data_ptr") else int(w_lm))
    return int(_lib.asd_lm_head_variant(ctypes.byref(dims), int(total_nodes), ptr))


ATTENTION_VARIANTS = {1: "attn_bf16_kernel", 2: "attn_tc_kernel", 3: "attn_pp_kernel",
                      4: "attn_f32_kernel"}


def asd_attention_variant(dims: Dims, total_nodes: int) -> int:
    """Which tree-attention kernel a call runs (include/asd.h): 1-4, 0 for
    invalid arguments."""
    return int(_lib.asd_attention_variant(ctypes.byref(dims), int(total_nodes)))


def asd_debug_set_wait_cycles(cycles: int):
    """Test hook: the kernels' bounded waits give up after `cycles` SM clock
    cycles in later calls (0 restores the default of about 2 s)."""
    _check(_lib.asd_debug_set_wait_cycles(int(cycles)), "asd_debug_set_wait_cycles")


def asd_get_device_status(workspace, stream=None) -> int:
    out = ctypes.c_int32(-1)
    _check(_lib.asd_get_device_status(_ptr(workspace), ctypes.byref(out), _stream(stream)),
           "asd_get_device_status")
    return int(out.value)


class VerifyStep:
    """Owns the output tensors of one verify-step shape and the argument block.

    Inputs are bound once (`bind`); `run()` enqueues asd_verify_step on the
    stream.  `events` (optional list of 5 torch.cuda.Event with timing) are
    recorded at the stage boundaries documented in asd.h.
    """

    OUT_FIELDS = ("attn_out", "row_max", "row_argmax", "row_lse", "l_draft", "ratio", "accept",
                  "path", "path_len", "bonus", "n_promoted", "ctx_len_out")
    # the walk's results and the per-node verdicts lead the output arena, so
    # that one copy (`results`) brings back what a decode loop reads per step
    RESULT_FIELDS = ("path", "path_len", "bonus", "n_promoted", "ctx_len_out", "accept", "row_lse")

    def __init__(self, dims: Dims, total_nodes: int, device="cuda", attn_dtype=torch.bfloat16):
        self.dims = dims
        self.T = int(total_nodes)
        T, B, i32, f32 = self.T, dims.batch, torch.int32, torch.float32
        shapes = dict(path=((B, dims.max_path), i32), path_len=((B,), i32), bonus=((B,), i32),
                      n_promoted=((B,), i32), ctx_len_out=((B,), i32),
                      accept=((T,), torch.uint8), row_lse=((T,), f32), row_max=((T,), f32),
                      row_argmax=((T,), i32), l_draft=((T,), f32), ratio=((T,), f32),
                      attn_out=((T, dims.num_q_heads, dims.head_dim), attn_dtype))
        order = self.RESULT_FIELDS + tuple(f for f in self.OUT_FIELDS if f not in self.RESULT_FIELDS)
        offs, off = {}, 0
        for f in order:
            shape, dt = shapes[f]
            n = 1
            for x in shape:
                n *= x
            offs[f] = off
            off = (off + n * torch.empty((), dtype=dt).element_size() + 255) // 256 * 256
            if f == self.RESULT_FIELDS[-1]:
                self._results_bytes = off
        self.arena = torch.empty(off, dtype=torch.uint8, device=device)
        self.out = {}
        for f in order:
            shape, dt = shapes[f]
            n = 1
            for x in shape:
                n *= x
            nb = n * torch.empty((), dtype=dt).element_size()
            self.out[f] = self.arena[offs[f]:offs[f] + nb].view(dt).view(*shape)
        self.results = self.arena[:self._results_bytes]
        self.workspace = alloc_workspace(dims, T, device)
        self.args = VerifyArgs()
        self._keep = []

    def bind(self, *, q, tree_k, tree_v, hidden, w_lm, tokens, parent, cu_nodes, ctx_len,
             k_cache, v_cache, tau, page_table=None, events: Optional[Sequence] = None):
        a = self.args
        self._keep = [q, tree_k, tree_v, hidden, w_lm, tokens, parent, cu_nodes, ctx_len,
                      k_cache, v_cache, page_table]
        a.q, a.tree_k, a.tree_v = _ptr(q), _ptr(tree_k), _ptr(tree_v)
        a.hidden, a.w_lm, a.tokens = _ptr(hidden), _ptr(w_lm), _ptr(tokens)
        a.parent, a.cu_nodes, a.ctx_len = _ptr(parent), _ptr(cu_nodes), _ptr(ctx_len)
        a.page_table = _ptr(page_table)
        a.total_nodes = self.T
        a.tau = float(tau)
        a.k_cache, a.v_cache = _ptr(k_cache), _ptr(v_cache)
        for f in self.OUT_FIELDS:
            setattr(a, f, _ptr(self.out[f]))
        for i in range(NUM_STAGE_EVENTS):
            a.stage_events[i] = (events[i].cuda_event if events is not None else None)
        return self

    def run(self, stream=None):
        asd_verify_step(self.dims, self.args, self.workspace, stream)
        return self.out

    def device_status(self, stream=None) -> int:
        return asd_get_device_status(self.workspace, stream)

    def capture(self, copies_in=(), copies_out=()):
        """A CUDA graph of one step: the (device, host) input copies in
        `copies_in`, the verify step, then the (host, device) result copies in
        `copies_out` (host tensors pinned).  It is recorded on a private stream;
        `replay()` runs the whole step on the current stream with one launch
        from the host, as a decode loop replays one graph per tree shape."""
        g = torch.cuda.CUDAGraph()
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.graph(g, stream=side):
            for dst, src in copies_in:
                dst.copy_(src, non_blocking=True)
            self.run(side)
            for dst, src in copies_out:
                dst.copy_(src, non_blocking=True)
        torch.cuda.current_stream().wait_stream(side)
        return g


# ------------------------------------------------------------ tree-shape policy

def asd_policy_triplets(params: PolicyParams) -> list:
    """Every (n_steps, topk, ndt) the policy can select, by increasing DCS
    (host only)."""
    n = int(_lib.asd_policy_triplets(ctypes.byref(params), None, 0))
    if n < 0:
        raise AsdError(-n, "asd_policy_triplets")
    buf = (ctypes.c_int32 * (3 * n))()
    _lib.asd_policy_triplets(ctypes.byref(params), buf, n)
    return [tuple(buf[3 * i:3 * i + 3]) for i in range(n)]


def asd_policy_init(params: PolicyParams, state: torch.Tensor, batch: int, stream=None):
    _check(_lib.asd_policy_init(ctypes.byref(params), _ptr(state), int(batch), _stream(stream)),
           "asd_policy_init")


def asd_policy_update(params: PolicyParams, cu_nodes, path_len, batch: int, state, stream=None):
    _check(_lib.asd_policy_update(ctypes.byref(params), _ptr(cu_nodes), _ptr(path_len),
                                  int(batch), _ptr(state), _stream(stream)), "asd_policy_update")


def asd_policy_select(params: PolicyParams, row_max, row_lse, rows, num_rows: int, batch: int,
                      state, triplet, dcs=None, stream=None):
    _check(_lib.asd_policy_select(ctypes.byref(params), _ptr(row_max), _ptr(row_lse), _ptr(rows),
                                  int(num_rows), int(batch), _ptr(state), _ptr(triplet), _ptr(dcs),
                                  _stream(stream)), "asd_policy_select")


class TreePolicy:
    """Per-request tree-shape policy state in device memory (Sec. 3.3, Eq. 2).

    update() after each verify step (reads path_len and cu_nodes on the
    device); select() after the draft's first forward (reads the draft LM
    head's row_max / row_lse) writes each request's next triplet into
    `self.triplet` [B, 3] and its DCS into `self.dcs` [B].  Nothing here
    synchronises, so the calls can sit inside a captured decode loop."""

    def __init__(self, batch: int, params: Optional[PolicyParams] = None, device="cuda"):
        self.params = params or make_policy_params()
        self.batch = int(batch)
        self.state = torch.empty(max(self.batch, 1) * POLICY_STATE_BYTES, dtype=torch.uint8,
                                 device=device)
        self.triplet = torch.empty(max(self.batch, 1), 3, dtype=torch.int32, device=device)
        self.dcs = torch.empty(max(self.batch, 1), dtype=torch.float64, device=device)
        self.reset()

    def triplets(self) -> list:
        return asd_policy_triplets(self.params)

    def reset(self, stream=None):
        asd_policy_init(self.params, self.state, self.batch, stream)

    def update(self, cu_nodes, path_len, stream=None):
        asd_policy_update(self.params, cu_nodes, path_len, self.batch, self.state, stream)

    def select(self, row_max, row_lse, rows=None, stream=None):
        asd_policy_select(self.params, row_max, row_lse, rows, row_max.numel(), self.batch,
                          self.state, self.triplet, self.dcs, stream)
        return self.triplet

    def state_arrays(self):
        """(rar float64 [B], zero_streak int32 [B], breaks int32 [B]) on the
        device, views of the state array."""
        n = self.batch
        rar = self.state.view(torch.float64)[0:2 * n:2]
        ints = self.state.view(torch.int32).view(-1, 4)[:n]
        return rar, ints[:, 2], ints[:, 3]
