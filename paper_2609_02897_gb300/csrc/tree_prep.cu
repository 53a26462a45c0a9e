// Tree preparation: validates each draft tree (parent array, drafted token
// range, context length) into the status word and per-sequence flags, and
// derives what the LM-head epilogue consumes:
//  - children of every node grouped by parent and sorted by (token, node id),
//    so the LM-head epilogue can pick l_draft = logits[parent, token] while it
//    sweeps the vocabulary in increasing order (Eq. 1 needs the parent row's
//    logit of each drafted token).
// One CTA of 128 threads per sequence; thread i owns local node i.
#include "kernels.h"

namespace asd {

__global__ void __launch_bounds__(kMaxNodes) tree_prep_kernel(PrepParams p) {
  __shared__ int s_par[kMaxNodes];
  __shared__ int s_tok[kMaxNodes];
  __shared__ int s_cnt[kMaxNodes];
  __shared__ int s_start[kMaxNodes];
  __shared__ int s_bad;

  pdl_launch_dependents();
  const int b = blockIdx.x;
  const int i = threadIdx.x;
  const int s = p.cu_nodes[b];
  const int e = p.cu_nodes[b + 1];
  if (i == 0) s_bad = 0;
  __syncthreads();

  bool seq_ok = (s >= 0) && (e > s) && (e <= p.T) && (e - s <= p.max_nodes);
  if (b == 0) seq_ok = seq_ok && (s == 0);
  if (b == p.B - 1) seq_ok = seq_ok && (e == p.T);
  if (!seq_ok) {
    if (i == 0) {
      p.seq_flags[b] = kSeqBadTree;
      set_status(p.status, ASD_ERR_TREE);
    }
    return;
  }
  const int n = e - s;

  int par = -1, tok = 0;
  if (i < n) {
    par = p.parent[s + i];
    tok = p.tokens ? p.tokens[s + i] : 0;
    const bool ok = (i == 0) ? (par == -1) : (par >= 0 && par < i);
    if (!ok) atomicOr(&s_bad, kSeqBadTree);
    if (p.tokens && i > 0 && (tok < 0 || tok >= p.vocab)) atomicOr(&s_bad, kSeqBadToken);
    s_par[i] = ok ? par : (i == 0 ? -1 : 0);
    s_tok[i] = tok;
  }
  if (i == 0 && p.ctx_len) {
    const int c = p.ctx_len[b];
    if (c < 0 || c > p.ctx_max) atomicOr(&s_bad, kSeqBadCtx);
  }
  __syncthreads();
  const int bad = s_bad;
  if (i == 0) {
    p.seq_flags[b] = bad;
    if (bad & kSeqBadTree) set_status(p.status, ASD_ERR_TREE);
    else if (bad & kSeqBadToken) set_status(p.status, ASD_ERR_TOKEN_RANGE);
    else if (bad & kSeqBadCtx) set_status(p.status, ASD_ERR_CTX_RANGE);
  }
  const bool tree_ok = !(bad & kSeqBadTree);

  if (i < n) {
    int c = 0;
    if (tree_ok)
      for (int j = 1; j < n; ++j) c += (s_par[j] == i);
    s_cnt[i] = c;
    if (p.l_draft) p.l_draft[s + i] = __int_as_float(0x7fc00000);  // NaN
  }
  __syncthreads();
  if (i < n) {
    int st = 0;
    for (int j = 0; j < i; ++j) st += s_cnt[j];
    s_start[i] = st;
    p.child_start[s + i] = s + st;
    p.child_cnt[s + i] = s_cnt[i];
  }
  __syncthreads();
  if (tree_ok && i > 0 && i < n) {
    const int pp = s_par[i];
    int rank = 0;
    for (int j = 1; j < n; ++j) {
      if (s_par[j] == pp && (s_tok[j] < s_tok[i] || (s_tok[j] == s_tok[i] && j < i))) ++rank;
    }
    const int slot = s + s_start[pp] + rank;
    p.child_tok[slot] = s_tok[i];
    p.child_id[slot] = s + i;
  }
}

cudaError_t launch_tree_prep(const PrepParams& p, cudaStream_t s) {
  tree_prep_kernel<<<p.B, kMaxNodes, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace asd
