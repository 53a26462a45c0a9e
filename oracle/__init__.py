"""Plain fp64 CPU oracle for the tree-verification step of margin-based lossy
speculative decoding ("Margins, Not Windows", Sec. 3.2, Eq. 1).

TEST INFRASTRUCTURE ONLY.  Only `tests/`, `__graft_entry__.smoke()` and the
CPU-baseline / reference legs of `bench.py` may import or run anything here.
The CUDA library never calls it and shares no code with it.

Every function is written for clarity, not speed: inputs are widened to
float64, each step follows its definition literally, and library primitives
(numpy matmul, exp, log) are the only building blocks.

Modules
  attention  tree-masked GQA attention over context + tree ancestors (step a1)
  lmhead     logits, row max / argmax / log-sum-exp, drafted logit, Eq. 1 ratio
             and the kappa-threshold rule (step a2)
  accept     longest accepted root-to-node path by literal enumeration (a3)
  compact    copy of the accepted nodes' K/V into the cache (a4)
  verify     the four steps chained
  policy     the dynamic tree-shape policy: DCS, RAR, triplet mapping and
             circuit breaker (Sec. 3.3, Eq. 2)
"""
from .attention import tree_attention, ancestors_of  # noqa: F401
from .lmhead import logits_rows, lmhead_margin, topk_tokens  # noqa: F401
from .accept import accept_path  # noqa: F401
from .compact import kv_compact  # noqa: F401
from .verify import verify_step  # noqa: F401
from . import policy  # noqa: F401
