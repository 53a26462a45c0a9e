// Per-sequence tail of the verify step, one CTA of 1024 threads per sequence
// (thread i < N owns local node i; all 32 warps share the merge and the copy).  Three stages, selected by TailParams::mode:
//  finalize  merge the LM head's per-range partials of every row into
//            row_max / row_argmax / row_lse and evaluate the margin rule for
//            every drafted node: ratio = exp(l_draft - row_max[parent]) (Eq. 1),
//            accept = strict match of the parent row's top-1 or ratio >= tau
//            (compared as l_draft - row_max >= ln tau);
//  walk      choose the committed path under one of four readings of the
//            paper's first-mismatch rule (Sec. 3.2; TailParams::rule):
//            0 the longest root-to-node path of accepted nodes, ties to the
//              lexicographically smallest node sequence: heights of accepted
//              subtrees bottom-up by depth, then from the root the
//              lowest-index accepted child whose height is one less;
//            1 the same over paths with at most one promoted node (accepted,
//              not a strict match): strict-only and one-promotion heights;
//            2 greedy: a strict child if any (lowest index), else the accepted
//              child of largest ratio (lowest index on ties), else stop;
//            3 greedy with a single promotion;
//  compact   copy the path's tree K/V into cache slots ctx_len .. ctx_len +
//            path_len - 1 (contiguous or through the page table).
#include <climits>

#include "kernels.h"

namespace asd {
namespace {

constexpr int kTailThreads = 1024;     // 32 warps: one node's merge per warp
constexpr int kMaxPartsPerLane = kMaxLmRanges / 32;

__global__ void __launch_bounds__(kTailThreads) tail_kernel(const TailParams p) {
  __shared__ int s_par[kMaxNodes];
  __shared__ int s_tok[kMaxNodes];
  __shared__ int s_arg[kMaxNodes];
  __shared__ float s_max[kMaxNodes];
  __shared__ int s_acc[kMaxNodes];
  __shared__ int s_dep[kMaxNodes];
  __shared__ int s_h[kMaxNodes];
  __shared__ int s_bc[kMaxNodes];
  __shared__ int s_path[kMaxNodes];
  __shared__ int s_h1[kMaxNodes];                    // rule 1: heights with one promotion
  __shared__ int s_bc1[kMaxNodes];                   // rule 1: best child, promotion left
  __shared__ float s_ratio[kMaxNodes];               // rules 2, 3
  __shared__ unsigned long long s_bp[kMaxNodes];     // rules 2, 3: best promoted child key
  __shared__ int s_maxd, s_len, s_skip;

  // Until pdl_wait() this kernel reads only caller inputs (cu_nodes, parent,
  // tokens): no kernel of the call writes them, and every call starts behind
  // a stream-ordered memset, so they are final even before the wait.
  const int b = blockIdx.x;
  const int i = threadIdx.x;
  const int warp = i >> 5, lane = i & 31;
  const int s = p.cu_nodes[b];
  const int e = p.cu_nodes[b + 1];
  const bool seq_ok = (s >= 0) && (e > s) && (e <= p.T) && (e - s <= p.max_nodes);
  if (!seq_ok) {
    pdl_wait();
    if (i == 0) {
      set_status(p.status, ASD_ERR_TREE);
      if (p.mode & kTailWalk) {
        p.path_len[b] = 0;
        p.bonus[b] = -1;
        p.n_promoted[b] = 0;
      }
      if ((p.mode & kTailCompact) && p.ctx_len_out) p.ctx_len_out[b] = p.ctx_len[b];
    }
    return;
  }
  const int n = e - s;

  bool okn = true;
  if (i < n) {
    // the standalone commit has no parent array: it only needs the path
    const int par = p.parent ? p.parent[s + i] : (i == 0 ? -1 : 0);
    okn = (i == 0) ? (par == -1) : (par >= 0 && par < i);
    s_par[i] = okn ? par : -1;
    s_tok[i] = p.tokens ? p.tokens[s + i] : 0;
  }
  if (i == 0) {
    s_maxd = 0;
    s_len = 0;
  }
  const int tree_bad = __syncthreads_or(!okn);
  // node depths for the walk need the tree alone
  if ((p.mode & kTailWalk) && !tree_bad && i < n) {
    int d = 0, u = i;
    while (s_par[u] >= 0) {
      u = s_par[u];
      ++d;
    }
    s_dep[i] = d;
    s_h[i] = 1;
    s_bc[i] = INT_MAX;
    s_h1[i] = 1;
    s_bc1[i] = INT_MAX;
    s_bp[i] = 0ull;
    atomicMax(&s_maxd, d);
  }

  pdl_wait();  // every earlier kernel of the call has completed
  // a bounded wait of an earlier kernel gave up: its statistics or verdicts
  // are incomplete, so no sequence commits anything
  const bool timed_out = reinterpret_cast<const volatile int*>(p.status)[1] != 0;
  const int flags = p.seq_flags ? p.seq_flags[b] : 0;
  // the drafted token's logit, loaded alongside the partials below
  const float l_draft_i =
      ((p.mode & kTailFinalize) && !tree_bad && i > 0 && i < n) ? p.l_draft[s + i] : 0.f;
  if (i == 0) {
    if (tree_bad) set_status(p.status, ASD_ERR_TREE);
    s_skip = (tree_bad || flags || timed_out) ? 1 : 0;
  }

  // ---------------------------------------------------------------- finalize
  if (p.mode & kTailFinalize) {
    if (!tree_bad) {
      // one warp per node: every lane loads its (up to 8) partials before merging
      for (int r = warp; r < n; r += kTailThreads / 32) {
        const size_t node = static_cast<size_t>(s + r);
        const float4* src = reinterpret_cast<const float4*>(p.part + node * p.g_lm);
        float4 q[kMaxPartsPerLane];
#pragma unroll
        for (int k = 0; k < kMaxPartsPerLane; ++k) {
          const int g = lane + 32 * k;
          q[k] = g < p.g_lm ? __ldcg(src + g) : make_float4(-INFINITY, 0.f, 0.f, 0.f);
        }
        float m = -INFINITY, sm = 0.f;
        int a = INT_MAX;
#pragma unroll
        for (int k = 0; k < kMaxPartsPerLane; ++k) merge_part(m, sm, a, q[k].x, q[k].y, __float_as_int(q[k].z));
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
          const float m2 = __shfl_xor_sync(0xffffffffu, m, off);
          const float s2 = __shfl_xor_sync(0xffffffffu, sm, off);
          const int a2 = __shfl_xor_sync(0xffffffffu, a, off);
          merge_part(m, sm, a, m2, s2, a2);
        }
        if (lane == 0) {
          p.row_max[node] = m;
          p.row_argmax[node] = a;
          p.row_lse[node] = m + logf(sm);
          s_max[r] = m;
          s_arg[r] = a;
        }
      }
    }
    __syncthreads();
    if (i < n && !tree_bad) {
      int acc = 1;
      float ratio = __int_as_float(0x7fc00000);
      if (i > 0) {
        const int pp = s_par[i];
        const float d = l_draft_i - s_max[pp];
        const bool strict = s_tok[i] == s_arg[pp];
        ratio = expf(d);
        acc = (strict || d >= p.ln_tau) ? 1 : 0;
      }
      p.ratio[s + i] = ratio;
      p.accept[s + i] = static_cast<uint8_t>(acc);
      s_acc[i] = acc;
      s_ratio[i] = ratio;
    }
  } else if (p.mode & kTailWalk) {
    if (i < n) {
      s_acc[i] = p.accept[s + i] != 0 ? 1 : 0;
      s_arg[i] = p.row_argmax[s + i];
      s_ratio[i] = (p.rule >= 2 && p.ratio) ? p.ratio[s + i] : 0.f;
    }
  }
  __syncthreads();

  // -------------------------------------------------------------------- walk
  if (p.mode & kTailWalk) {
    if (!s_skip) {
      // a node is strict when it drafts its parent row's top-1; root-level
      // quantities are per node below, the walk runs on thread 0
      const bool strict_i = i > 0 && i < n && s_acc[i] && s_tok[i] == s_arg[s_par[i]];
      if (p.rule <= 1) {
        // s_h: heights over accepted (rule 0) or strict-only (rule 1) children;
        // s_h1: heights with at most one promotion below the node (rule 1)
        for (int dd = s_maxd; dd >= 1; --dd) {
          if (i < n && s_dep[i] == dd && s_acc[i]) {
            if (p.rule == 0 || strict_i) atomicMax(&s_h[s_par[i]], s_h[i] + 1);
            if (p.rule == 1) atomicMax(&s_h1[s_par[i]], (strict_i ? s_h1[i] : s_h[i]) + 1);
          }
          __syncthreads();
        }
        if (i > 0 && i < n && s_acc[i]) {
          const int u = s_par[i];
          if ((p.rule == 0 || strict_i) && s_h[i] == s_h[u] - 1) atomicMin(&s_bc[u], i);
          if (p.rule == 1 && (strict_i ? s_h1[i] : s_h[i]) == s_h1[u] - 1) atomicMin(&s_bc1[u], i);
        }
      } else if (i > 0 && i < n && s_acc[i]) {
        const int u = s_par[i];
        if (strict_i) {
          atomicMin(&s_bc[u], i);
        } else {
          // largest ratio first, then the lowest index (ratios are >= 0 here)
          const unsigned long long key =
              (static_cast<unsigned long long>(__float_as_uint(fmaxf(s_ratio[i], 0.f))) << 32) |
              static_cast<unsigned long long>(0xFFFFFFFFu - static_cast<unsigned>(i));
          atomicMax(&s_bp[u], key);
        }
      }
      __syncthreads();
      if (i == 0) {
        int u = 0, len = 0, promoted = 0, budget = 1;
        s_path[len++] = 0;
        while (len < kMaxNodes) {
          int c = INT_MAX;
          if (p.rule == 0) {
            c = s_bc[u];
          } else if (p.rule == 1) {
            c = budget ? s_bc1[u] : s_bc[u];
          } else {
            c = s_bc[u];
            if (c == INT_MAX && s_bp[u] != 0ull && (p.rule == 2 || budget))
              c = static_cast<int>(0xFFFFFFFFu - static_cast<unsigned>(s_bp[u] & 0xFFFFFFFFull));
          }
          if (c == INT_MAX) break;
          if (s_tok[c] != s_arg[u]) {
            ++promoted;
            budget = 0;
          }
          s_path[len++] = c;
          u = c;
        }
        if (len > p.max_path) {
          set_status(p.status, ASD_ERR_SHAPE);
          len = 0;
        }
        s_len = len;
        p.path_len[b] = len;
        p.bonus[b] = len > 0 ? s_arg[u] : -1;
        p.n_promoted[b] = len > 0 ? promoted : 0;
      }
      __syncthreads();
      for (int k = i; k < p.max_path; k += kTailThreads)
        p.path[static_cast<size_t>(b) * p.max_path + k] = k < s_len ? s_path[k] : -1;
    } else {
      for (int k = i; k < p.max_path; k += kTailThreads)
        p.path[static_cast<size_t>(b) * p.max_path + k] = -1;
      if (i == 0) {
        p.path_len[b] = 0;
        p.bonus[b] = -1;
        p.n_promoted[b] = 0;
      }
    }
  } else if (p.mode & kTailCompact) {
    // standalone commit: the path comes from the caller
    if (i == 0) {
      int len = p.path_len[b];
      bool ok = !s_skip && len >= 0 && len <= p.max_path && len <= n;
      for (int k = 0; ok && k < len; ++k) {
        const int u = p.path[static_cast<size_t>(b) * p.max_path + k];
        if (u < 0 || u >= n) ok = false;
        else s_path[k] = u;
      }
      if (!ok) {
        set_status(p.status, ASD_ERR_SHAPE);
        len = 0;
        s_skip = 1;
      }
      s_len = len;
    }
  }
  __syncthreads();

  // ------------------------------------------------------------------ commit
  if (p.mode & kTailCompact) {
    const int ctx = p.ctx_len[b];
    const int len = s_len;
    const bool ctx_ok = ctx >= 0 && ctx + len <= p.ctx_max;
    if (i == 0 && !ctx_ok && !s_skip) set_status(p.status, ASD_ERR_CTX_RANGE);
    if (s_skip || !ctx_ok) {
      if (i == 0) p.ctx_len_out[b] = ctx;
      return;
    }
    const int row_bytes = p.D * p.elem_bytes;
    const int chunks = row_bytes / 16;
    const int per_node = p.Hkv * chunks;
    const uint8_t* tk = static_cast<const uint8_t*>(p.tree_k);
    const uint8_t* tv = static_cast<const uint8_t*>(p.tree_v);
    uint8_t* kc = static_cast<uint8_t*>(p.k_cache);
    uint8_t* vc = static_cast<uint8_t*>(p.v_cache);
    for (int idx = i; idx < len * per_node; idx += kTailThreads) {
      const int k = idx / per_node;
      const int rem = idx - k * per_node;
      const int g = rem / chunks;
      const int ch = rem - g * chunks;
      const size_t src = (static_cast<size_t>(s + s_path[k]) * p.Hkv + g) * row_bytes + ch * 16;
      const int slot = ctx + k;
      size_t dst;
      if (p.page_size == 0) {
        dst = ((static_cast<size_t>(b) * p.Hkv + g) * p.ctx_max + slot) * row_bytes + ch * 16;
      } else {
        const int page = p.page_table[static_cast<size_t>(b) * p.pages_per_seq + slot / p.page_size];
        if (page < 0 || page >= p.num_pages) {
          set_status(p.status, ASD_ERR_CTX_RANGE);
          continue;
        }
        dst = ((static_cast<size_t>(page) * p.Hkv + g) * p.page_size + slot % p.page_size) *
                  row_bytes + ch * 16;
      }
      *reinterpret_cast<uint4*>(kc + dst) = *reinterpret_cast<const uint4*>(tk + src);
      *reinterpret_cast<uint4*>(vc + dst) = *reinterpret_cast<const uint4*>(tv + src);
    }
    if (i == 0) p.ctx_len_out[b] = ctx + len;
  }
}

}  // namespace

cudaError_t launch_tail(const TailParams& p, cudaStream_t s) {
  return launch_pdl(tail_kernel, dim3(p.B), dim3(kTailThreads), 0, s, p);
}

}  // namespace asd
