"""The C-ABI library builds, loads, and exports every function declared in
include/asd.h; host-side argument checks answer without touching a GPU."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2609_02897_gb300 import build
    path = build.build()
    return ctypes.CDLL(path)


def _declared():
    src = open(os.path.join(ROOT, "include", "asd.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(asd_[a-z_]+)\s*\(", src)))


def test_every_declared_function_is_exported(lib):
    names = _declared()
    assert len(names) == 19, names
    for n in names:
        assert hasattr(lib, n), n


def test_binding_names_match_header():
    from paper_2609_02897_gb300 import build
    build.build()
    from paper_2609_02897_gb300 import asd
    assert sorted(asd.EXPORTS) == _declared()
    assert asd.abi_version() == 5


def test_host_checks_without_gpu(lib):
    from paper_2609_02897_gb300 import asd
    # null dims / null tensors / tau outside (0, 1] are rejected before any CUDA call
    assert lib.asd_tree_attention(None, *([None] * 9), 0, None, None, ctypes.c_size_t(0), None) == 1
    f = ctypes.c_float
    lib.asd_lmhead_margin.argtypes = asd._lib.asd_lmhead_margin.argtypes
    dims = asd.make_dims(1, 4, 4, 64, 256, 4096, asd.ASD_F32, 0, 320, 0, 8, 5)
    buf = ctypes.c_void_p(16)
    args = [ctypes.byref(dims)] + [buf] * 5 + [8]
    outs = [buf] * 6 + [buf, 1 << 20, None]
    assert lib.asd_lmhead_margin(*args, f(0.0), *outs) == 1
    assert lib.asd_lmhead_margin(*args, f(1.5), *outs) == 1
    assert lib.asd_lmhead_margin(*args, f(float("nan")), *outs) == 1
    lib.asd_status_string.restype = ctypes.c_char_p
    assert lib.asd_status_string(3) == b"malformed draft tree"


def test_packed_lm_head_host_checks(lib):
    """Size of the packed LM-head weight (256 header bytes + W rounded up to
    32 rows and 64 columns) and the packing call's host-side rejections,
    answered before any CUDA call."""
    from paper_2609_02897_gb300 import asd
    V, K = 1000, 200            # 32 groups (1024 rows), 4 k-blocks (256 columns)
    d = asd.make_dims(1, 4, 4, 64, K, V, asd.ASD_BF16, 0, 64, 0, 8, 5)
    assert asd.asd_lm_head_packed_bytes(d) == 256 + 32 * 4 * 4096
    f = asd.make_dims(1, 4, 4, 64, K, V, asd.ASD_F32, 0, 64, 0, 8, 5)
    assert lib.asd_lm_head_packed_bytes(ctypes.byref(f)) == 0
    pk = asd.make_dims(1, 4, 4, 64, K, V, asd.ASD_F32, 0, 64, 0, 8, 5, asd.ASD_LM_PACKED)
    assert lib.asd_workspace_bytes(ctypes.byref(pk), 8) == 0     # packed W is bf16 only
    bad = asd.make_dims(1, 4, 4, 64, K, V, asd.ASD_BF16, 0, 64, 0, 8, 5, 7)
    assert lib.asd_workspace_bytes(ctypes.byref(bad), 8) == 0    # unknown layout
    fn = asd._lib.asd_pack_lm_head
    w, out = ctypes.c_void_p(1 << 20), ctypes.c_void_p(1 << 30)
    assert fn(ctypes.byref(d), None, out, 1 << 30, None) == 1
    assert fn(ctypes.byref(f), w, out, 1 << 30, None) == 2
    assert fn(ctypes.byref(d), w, ctypes.c_void_p((1 << 30) + 16), 1 << 30, None) == 1  # alignment
    assert fn(ctypes.byref(d), w, out, 4096, None) == 6                                 # too small
    assert fn(ctypes.byref(d), w, ctypes.c_void_p((1 << 20) + 256), 1 << 30, None) == 1  # overlap


def test_accept_rule_host_checks(lib):
    """An accept rule outside asd_accept_rule fails the dims check
    (ASD_ERR_SHAPE) and the greedy rules need the ratios
    (ASD_ERR_INVALID_ARG without them); both are answered before any CUDA
    call, so the placeholder pointers are never read."""
    from paper_2609_02897_gb300 import asd
    d = asd.make_dims(1, 4, 4, 64, 256, 4096, asd.ASD_BF16, 0, 64, 0, 8, 5)
    fn = asd._lib.asd_accept_path
    buf = ctypes.c_void_p(1 << 20)

    def call(ratio):
        return fn(ctypes.byref(d), buf, buf, buf, buf, ratio, buf, 8, buf, buf, buf, buf, buf,
                  1 << 20, None)
    for rule in (-1, 4):
        d.accept_rule = rule
        assert call(buf) == 2
        assert lib.asd_workspace_bytes(ctypes.byref(d), 8) == 0
    for rule in (asd.ASD_ACCEPT_GREEDY, asd.ASD_ACCEPT_GREEDY_ONCE):
        d.accept_rule = rule
        assert call(None) == 1


def test_policy_triplets_match_the_oracle():
    """asd_policy_triplets (host C) lists the same triplets, in the same order,
    as the oracle's enumeration, on the paper's range and on random ones."""
    import numpy as np
    from paper_2609_02897_gb300 import build
    build.build()
    from paper_2609_02897_gb300 import asd
    from oracle import policy as P
    rng = np.random.default_rng(5)
    ranges = [((3, 4, 4), (7, 1, 8)), ((7, 1, 8), (3, 4, 4)), ((4, 8, 10), (6, 2, 10)),
              ((3, 1, 4), (3, 1, 4)), ((1, 1, 1), (128, 128, 128))]
    ranges += [(tuple(int(x) for x in rng.integers(1, 33, 3)),
                tuple(int(x) for x in rng.integers(1, 33, 3))) for _ in range(40)]
    for sh, dp in ranges:
        got = asd.asd_policy_triplets(asd.make_policy_params(shallow=sh, deep=dp))
        assert got == P.reachable_triplets(sh, dp), (sh, dp)
    # a short buffer receives the first `cap` triplets and the full count
    import ctypes
    buf = (ctypes.c_int32 * 6)()
    pp = asd.make_policy_params()
    assert asd._lib.asd_policy_triplets(ctypes.byref(pp), buf, 2) == 8
    assert list(buf) == [3, 4, 4, 4, 4, 5]


def test_policy_host_checks(lib):
    """Invalid policy settings and null pointers are rejected before any CUDA
    call (the placeholder pointers are never read)."""
    from paper_2609_02897_gb300 import asd
    buf = ctypes.c_void_p(1 << 20)
    bad = [dict(alpha=0.0), dict(alpha=1.5), dict(alpha=float("nan")), dict(divisor=0.0),
           dict(divisor=float("inf")), dict(rar_init=-0.1), dict(rar_init=1.1),
           dict(shallow=(0, 4, 4)), dict(deep=(7, 1, 129)), dict(breaker=0)]
    for kw in bad:
        pp = asd.make_policy_params(**kw)
        assert asd._lib.asd_policy_triplets(ctypes.byref(pp), None, 0) == -1, kw
        assert asd._lib.asd_policy_init(ctypes.byref(pp), buf, 4, None) == 1, kw
        assert asd._lib.asd_policy_update(ctypes.byref(pp), buf, buf, 4, buf, None) == 1, kw
        assert asd._lib.asd_policy_select(ctypes.byref(pp), buf, buf, None, 4, 4, buf, buf, None,
                                          None) == 1, kw
    pp = asd.make_policy_params()
    pp.reserved = 1
    assert asd._lib.asd_policy_init(ctypes.byref(pp), buf, 4, None) == 1
    pp = asd.make_policy_params()
    assert asd._lib.asd_policy_init(ctypes.byref(pp), None, 4, None) == 1
    assert asd._lib.asd_policy_init(ctypes.byref(pp), buf, -1, None) == 1
    assert asd._lib.asd_policy_update(ctypes.byref(pp), None, buf, 4, buf, None) == 1
    assert asd._lib.asd_policy_select(ctypes.byref(pp), buf, None, None, 4, 4, buf, buf, None,
                                      None) == 1
    assert asd._lib.asd_policy_select(ctypes.byref(pp), buf, buf, None, -1, 4, buf, buf, None,
                                      None) == 1
    # batch 0 enqueues nothing and succeeds
    assert asd._lib.asd_policy_init(ctypes.byref(pp), buf, 0, None) == 0
    assert asd._lib.asd_policy_triplets(None, None, 0) == -1


def test_lm_schedule_host_checks(lib):
    """An unknown LM-head schedule, or the lazy one with fp32, fails the dims
    check (ASD_ERR_SHAPE) before any CUDA call."""
    from paper_2609_02897_gb300 import asd
    buf = ctypes.c_void_p(1 << 20)
    fn = asd._lib.asd_lmhead_margin
    for dtype, sched in ((asd.ASD_BF16, 2), (asd.ASD_BF16, -1), (asd.ASD_F32, asd.ASD_LM_LAZY_LEVELS)):
        d = asd.make_dims(1, 4, 4, 64, 256, 4096, dtype, 0, 64, 0, 8, 5, 0, 0, sched)
        assert fn(ctypes.byref(d), buf, buf, buf, buf, buf, 8, ctypes.c_float(0.5), *([buf] * 6),
                  buf, 1 << 20, None) == 2
        assert lib.asd_workspace_bytes(ctypes.byref(d), 8) == 0


def _struct_members(src, name):
    """Member names, in order, of `typedef struct name {...} name;` in asd.h."""
    body = re.search(r"typedef struct " + name + r" \{(.*?)\} " + name + ";", src, re.S).group(1)
    body = re.sub(r"/\*.*?\*/", "", body, flags=re.S)
    names = []
    for decl in body.split(";"):
        m = re.search(r"(\w+)\s*(\[[^\]]*\])?\s*$", decl.strip())
        if m and decl.strip():
            names.append(m.group(1))
    return names


def _enum_values(src, name):
    body = re.search(r"typedef enum " + name + r" \{(.*?)\} " + name + ";", src, re.S).group(1)
    body = re.sub(r"/\*.*?\*/", "", body, flags=re.S)
    return {k: int(v) for k, v in re.findall(r"(\w+)\s*=\s*(-?\d+)", body)}


def test_binding_structs_and_constants_match_header():
    """The ctypes structs carry the header's members in the header's order,
    their sizes are those of the C layout, and the binding's constants equal
    the header's enumerators."""
    import ctypes
    from paper_2609_02897_gb300 import build
    build.build()
    from paper_2609_02897_gb300 import asd
    src = open(os.path.join(ROOT, "include", "asd.h")).read()
    assert _struct_members(src, "asd_dims") == [f for f, _ in asd.Dims._fields_]
    assert ctypes.sizeof(asd.Dims) == 4 * len(asd.Dims._fields_)
    assert _struct_members(src, "asd_verify_args") == [f for f, _ in asd.VerifyArgs._fields_]
    assert _struct_members(src, "asd_policy_params") == [f for f, _ in asd.PolicyParams._fields_]
    assert ctypes.sizeof(asd.PolicyParams) == 3 * 8 + 8 * 4
    assert _struct_members(src, "asd_policy_state") == ["rar", "zero_streak", "breaks"]
    assert asd.POLICY_STATE_BYTES == 16
    st = _enum_values(src, "asd_status")
    assert {v: k for k, v in st.items()} == asd.STATUS
    assert _enum_values(src, "asd_dtype") == {"ASD_F32": asd.ASD_F32, "ASD_BF16": asd.ASD_BF16}
    assert _enum_values(src, "asd_accept_rule") == {
        "ASD_ACCEPT_LONGEST": asd.ASD_ACCEPT_LONGEST, "ASD_ACCEPT_ONCE": asd.ASD_ACCEPT_ONCE,
        "ASD_ACCEPT_GREEDY": asd.ASD_ACCEPT_GREEDY,
        "ASD_ACCEPT_GREEDY_ONCE": asd.ASD_ACCEPT_GREEDY_ONCE}
    assert _enum_values(src, "asd_lm_layout") == {"ASD_LM_ROWS": asd.ASD_LM_ROWS,
                                                  "ASD_LM_PACKED": asd.ASD_LM_PACKED}
    assert _enum_values(src, "asd_lm_schedule") == {
        "ASD_LM_EVERY_ROW": asd.ASD_LM_EVERY_ROW, "ASD_LM_LAZY_LEVELS": asd.ASD_LM_LAZY_LEVELS}
    defines = dict(re.findall(r"#define (ASD_\w+) \(?(\d+)", src))
    assert int(defines["ASD_MAX_TREE_NODES"]) == asd.MAX_TREE_NODES
    assert int(defines["ASD_NUM_STAGE_EVENTS"]) == asd.NUM_STAGE_EVENTS
    assert int(defines["ASD_ABI_VERSION"]) == asd.abi_version()
    m = re.search(r"#define ASD_NOALLOC_SCRATCH_BYTES \((\d+)u << (\d+)\)", src)
    assert m and int(m.group(1)) << int(m.group(2)) == asd.NOALLOC_SCRATCH_BYTES


def test_wait_budget_hook_checks_its_argument(lib):
    """The failure-path test hook takes a cycle count (0: the default) and
    refuses a negative one; it touches no GPU."""
    lib.asd_debug_set_wait_cycles.restype = ctypes.c_int
    lib.asd_debug_set_wait_cycles.argtypes = [ctypes.c_int64]
    assert lib.asd_debug_set_wait_cycles(-1) == 1
    assert lib.asd_debug_set_wait_cycles(0) == 0
