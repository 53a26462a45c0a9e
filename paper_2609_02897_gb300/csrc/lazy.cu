// Lazy, level-synchronous LM head (asd_lm_schedule ASD_LM_LAZY_LEVELS).
//
// The verify walk only ever reads the accept verdicts of nodes whose every
// ancestor was accepted, and a verdict needs the parent's LM-head row (Eq. 1
// and the kappa rule), so only the rows of the roots and of nodes reached
// through accepted nodes are needed.  They are computed one tree level at a
// time: level d's rows (node ids and a compact copy of their hidden states)
// go through the LM head, then lazy_level_kernel merges the rows' partials,
// judges their children, and appends the accepted children, with their hidden
// rows, to level d + 1.  Every LM-head pass streams W once, so the schedule
// pays when the tree's levels cost fewer passes than its full node count
// costs in flops.
//
// The merge of the partials and the kappa rule are the tail kernel's, in the
// same order, so every computed row and verdict is bit-identical to the
// every-row schedule's.  The order of rows within a level depends on atomic
// appends; no result depends on it.
#include <algorithm>
#include <climits>

#include "kernels.h"

namespace asd {
namespace {

constexpr int kLazyThreads = 256;
constexpr int kMaxPartsPerLane = kMaxLmRanges / 32;

// Copies hidden row `src` (K bf16) to row `dst` of the next level's buffer,
// one warp, 16 bytes per lane and step (K % 8 == 0).
__device__ __forceinline__ void copy_row(const LazyParams& p, int src, int dst, int lane) {
  const uint4* from = reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(p.hidden) +
                                                     static_cast<size_t>(src) * p.K);
  uint4* to = reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(p.h_next) +
                                       static_cast<size_t>(dst) * p.K);
  for (int k = lane; k < p.K / 8; k += 32) to[k] = __ldg(from + k);
}

// Level 0: every unflagged sequence's root, in p.rows_next / p.h_next.
// count[0 .. levels] were zeroed on the stream before this kernel.
__global__ void __launch_bounds__(kLazyThreads) lazy_init_kernel(const LazyParams p) {
  const int tid = blockIdx.x * blockDim.x + threadIdx.x;
  const int nth = gridDim.x * blockDim.x;
  const float nan = __int_as_float(0x7fc00000);
  for (int i = tid; i < p.T; i += nth) {
    p.row_max[i] = nan;
    p.row_argmax[i] = -1;
    p.row_lse[i] = nan;
    p.ratio[i] = nan;
    p.accept[i] = 0;
  }
  const int warp = tid >> 5, lane = threadIdx.x & 31, nwarps = nth >> 5;
  for (int b = warp; b < p.B; b += nwarps) {
    if (p.seq_flags[b] != 0) continue;  // malformed: no row, the walk skips it
    const int root = p.cu_nodes[b];
    int slot = 0;
    if (lane == 0) {
      slot = atomicAdd(&p.count[0], 1);
      p.rows_next[slot] = root;
    }
    slot = __shfl_sync(0xffffffffu, slot, 0);
    copy_row(p, root, slot, lane);
  }
}

// Level `level`: one warp per row of the level.  Merges the row's partials
// into row_max / row_argmax / row_lse of its node, applies the kappa rule to
// the node's children, and appends the accepted ones to the next level.
__global__ void __launch_bounds__(kLazyThreads) lazy_level_kernel(const LazyParams p) {
  const int lane = threadIdx.x & 31;
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int nwarps = (gridDim.x * blockDim.x) >> 5;
  const int nrow = min(max(p.count[p.level], 0), p.T);
  for (int r = warp; r < nrow; r += nwarps) {
    const int node = p.rows_cur[r];
    if (node < 0 || node >= p.T) continue;
    const float4* src = reinterpret_cast<const float4*>(p.part + static_cast<size_t>(r) * p.g_lm);
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
      if (p.level == 0) p.accept[node] = 1;  // the root
    }
    // the node's children, judged by its row (Eq. 1 and the kappa rule)
    const int cs = p.child_start[node];
    const int cn = p.child_cnt[node];
    if (cs < 0 || cn < 0 || cs > p.T - cn) continue;
    for (int j0 = 0; j0 < cn; j0 += 32) {
      const int j = j0 + lane;
      int c = -1;
      bool acc = false;
      if (j < cn) {
        c = p.child_id[cs + j];
        if (c > node && c < p.T) {
          const float d = p.l_draft[c] - m;
          const bool strict = p.tokens[c] == a;
          p.ratio[c] = expf(d);
          acc = strict || d >= p.ln_tau;
          p.accept[c] = static_cast<uint8_t>(acc ? 1 : 0);
        }
      }
      const unsigned taken = __ballot_sync(0xffffffffu, acc);
      if (!taken) continue;
      if (p.level >= p.last_level) {
        // a reached node one level deeper than max_path allows
        if (lane == 0) set_status(p.status, ASD_ERR_SHAPE);
        continue;
      }
      int base = 0;
      if (lane == 0) base = atomicAdd(&p.count[p.level + 1], __popc(taken));
      base = __shfl_sync(0xffffffffu, base, 0);
      if (acc) p.rows_next[base + __popc(taken & ((1u << lane) - 1u))] = c;
      for (unsigned left = taken; left; left &= left - 1u) {
        const int l = __ffs(left) - 1;
        const int cc = __shfl_sync(0xffffffffu, c, l);
        copy_row(p, cc, base + __popc(taken & ((1u << l) - 1u)), lane);
      }
    }
  }
}

}  // namespace

cudaError_t launch_lazy_init(const LazyParams& p, int levels, cudaStream_t s) {
  cudaError_t err = cudaMemsetAsync(p.count, 0, sizeof(int) * static_cast<size_t>(levels + 1), s);
  if (err != cudaSuccess) return err;
  const int blocks = std::max(1, std::min(1024, (std::max(p.T, 32 * p.B) + kLazyThreads - 1) / kLazyThreads));
  lazy_init_kernel<<<blocks, kLazyThreads, 0, s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_lazy_level(const LazyParams& p, int nsm, cudaStream_t s) {
  // enough warps for the largest level (at most T rows), at most 4 CTAs per SM
  const int rows_per_block = kLazyThreads / 32;
  const int blocks = std::max(1, std::min(4 * nsm, (p.T + rows_per_block - 1) / rows_per_block));
  lazy_level_kernel<<<blocks, kLazyThreads, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace asd
