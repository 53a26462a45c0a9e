// Per-row epilogue of the LM head: consumes logits of one node row in chunks
// of 32 consecutive vocabulary ids (increasing order) and keeps
//   m = running max, a = lowest id attaining it, s = sum of exp(logit - m),
// and records l_draft = logits[row, token] for every child whose drafted token
// falls in the chunk (Eq. 1 needs the parent row's logit of each drafted
// token).  Children come from the tree preparation kernel, grouped by parent
// and sorted by token, so a single forward-moving cursor finds them.
#pragma once

#include <climits>

#include "common.cuh"

namespace asd {

struct RowState {
  float m;
  float s;
  int a;
  int cur;       // next child slot
  int end;       // one past the last child slot
  int next_tok;  // token of child slot `cur` (INT_MAX when done)
};

__device__ __forceinline__ void row_state_init(RowState& st, bool active, int node, int v_begin,
                                               const int32_t* child_start,
                                               const int32_t* child_cnt,
                                               const int32_t* child_tok, int T) {
  st.m = -INFINITY;
  st.s = 0.f;
  st.a = -1;
  st.cur = 0;
  st.end = 0;
  st.next_tok = INT_MAX;
  if (!active) return;
  int cs = child_start[node];
  int cnt = child_cnt[node];
  if (cs < 0 || cnt < 0 || cnt > T || cs > T - cnt) cnt = 0;  // malformed tree: no children
  st.cur = cs;
  st.end = cs + cnt;
  while (st.cur < st.end && child_tok[st.cur] < v_begin) ++st.cur;
  st.next_tok = st.cur < st.end ? child_tok[st.cur] : INT_MAX;
}

// r[j] = logit of vocabulary id c0 + j, valid for j < nvalid.
__device__ __forceinline__ void row_chunk(RowState& st, const float (&r)[32], int c0, int nvalid,
                                          const int32_t* child_tok, const int32_t* child_id,
                                          float* l_draft, int T) {
  float x[32];
  float cm = -INFINITY;
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    x[j] = (j < nvalid) ? r[j] : -INFINITY;
    cm = fmaxf(cm, x[j]);
  }
  if (cm > st.m) {
    int first = 31;
#pragma unroll
    for (int j = 31; j >= 0; --j)
      if (x[j] == cm) first = j;
    st.s *= exp2f((st.m - cm) * kLog2e);
    st.m = cm;
    st.a = c0 + first;
  }
  const float nm = -st.m * kLog2e;
  float acc = 0.f;
  // one special-function-unit instruction per logit (results below 2^-126 of
  // the running max flush to zero: they cannot move the fp32 sum)
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    float e;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(e) : "f"(fmaf(x[j], kLog2e, nm)));
    acc += e;
  }
  st.s += acc;
  while (st.next_tok < c0 + nvalid) {
    const int jj = st.next_tok - c0;
    float v = 0.f;
#pragma unroll
    for (int j = 0; j < 32; ++j)
      if (j == jj) v = r[j];
    const int cid = child_id[st.cur];
    if (static_cast<unsigned>(cid) < static_cast<unsigned>(T)) l_draft[cid] = v;
    ++st.cur;
    st.next_tok = st.cur < st.end ? child_tok[st.cur] : INT_MAX;
  }
}

}  // namespace asd
