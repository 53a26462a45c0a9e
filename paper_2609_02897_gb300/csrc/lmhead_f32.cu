// LM head fused with the margin-rule statistics (Eq. 1) for fp32 inputs:
// exact fp32 FMA on the CUDA cores (the tensor cores have no fp32-exact mode).
// Same decomposition as the tensor-core kernel: one CTA per vocabulary range,
// one thread per node row, logits consumed in 32-wide chunks by the shared
// per-row epilogue, one (max, argmax, sum-exp) partial per node and range.
#include "kernels.h"
#include "lm_epilogue.cuh"

namespace asd {
namespace {

constexpr int kRows = 128;   // node rows per CTA pass (one per thread)
constexpr int kKc = 32;      // hidden elements staged per step

__global__ void __launch_bounds__(kRows) lmhead_f32_kernel(const LmParams p) {
  __shared__ float s_w[32][kKc + 1];
  __shared__ float s_h[kRows][kKc + 1];
  pdl_wait();
  pdl_launch_dependents();
  const int tid = threadIdx.x;
  const float* hid = static_cast<const float*>(p.hidden);
  const float* w = static_cast<const float*>(p.w);

  const int ngroups = (p.V + 31) / 32;
  const int gs = static_cast<int>(static_cast<long long>(blockIdx.x) * ngroups / p.g_lm);
  const int ge = static_cast<int>(static_cast<long long>(blockIdx.x + 1) * ngroups / p.g_lm);
  const int vs = gs * 32;
  const int ve = min(p.V, ge * 32);

  for (int nt = 0; nt * kRows < p.T; ++nt) {
    const int node = nt * kRows + tid;
    const bool active = node < p.T;
    RowState st;
    row_state_init(st, active, node, vs, p.child_start, p.child_cnt, p.child_tok, p.T);
    for (int v0 = vs; v0 < ve; v0 += 32) {
      const int nv = min(32, ve - v0);
      float acc[32];
#pragma unroll
      for (int j = 0; j < 32; ++j) acc[j] = 0.f;
      for (int k0 = 0; k0 < p.K; k0 += kKc) {
        for (int idx = tid; idx < 32 * kKc; idx += kRows) {
          const int j = idx / kKc, kk = idx % kKc;
          s_w[j][kk] = (j < nv && k0 + kk < p.K) ? w[static_cast<size_t>(v0 + j) * p.K + k0 + kk]
                                                 : 0.f;
        }
        for (int idx = tid; idx < kRows * kKc; idx += kRows) {
          const int r = idx / kKc, kk = idx % kKc;
          const int nd = nt * kRows + r;
          s_h[r][kk] = (nd < p.T && k0 + kk < p.K) ? hid[static_cast<size_t>(nd) * p.K + k0 + kk]
                                                   : 0.f;
        }
        __syncthreads();
#pragma unroll 4
        for (int kk = 0; kk < kKc; ++kk) {
          const float h = s_h[tid][kk];
#pragma unroll
          for (int j = 0; j < 32; ++j) acc[j] = fmaf(h, s_w[j][kk], acc[j]);
        }
        __syncthreads();
      }
      if (active) row_chunk(st, acc, v0, nv, p.child_tok, p.child_id, p.l_draft, p.T);
    }
    if (active) {
      LmPartial part;
      part.m = st.m;
      part.s = st.s;
      part.a = st.a;
      part.pad = 0;
      p.part[static_cast<size_t>(node) * p.g_lm + blockIdx.x] = part;
    }
  }
}

}  // namespace

cudaError_t launch_lmhead_f32(const LmParams& p, cudaStream_t s) {
  return launch_pdl(lmhead_f32_kernel, dim3(p.g_lm), dim3(kRows), 0, s, p);
}

}  // namespace asd
