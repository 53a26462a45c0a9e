// Shared device helpers and the workspace layout of libasd (sm_103a).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "asd.h"

namespace asd {

constexpr int kMaxNodes = ASD_MAX_TREE_NODES;
constexpr int kMaxLmRanges = 256;   // upper bound on LM-head vocabulary ranges (CTAs)
constexpr int kMaxAttnParts = 8;    // attention context splits = cluster size (portable max)
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
// Bounded waits give up after this many SM clock cycles (about 2 s at 2 GHz).
constexpr long long kWaitCycles = 4000000000LL;

// Per-sequence flags written by the tree preparation kernel.
enum SeqFlag : int { kSeqBadTree = 1, kSeqBadToken = 2, kSeqBadCtx = 4 };

// One vocabulary range's running softmax statistics of one LM-head row.
struct LmPartial {
  float m;   // max logit in the range
  float s;   // sum of exp(logit - m) over the range
  int a;     // lowest vocab id attaining m
  int pad;
};

// Offsets (bytes) of the workspace regions; every region is 256-byte aligned.
struct WsLayout {
  size_t status;       // int32[4]: [0] first device error code; [1] a bounded wait gave
                       // up; [2..3] int64 wait budget (0: the default), set for testing
  size_t seq_flags;    // int32[B]
  size_t child_start;  // int32[T]: global slot of the node's first child
  size_t child_cnt;    // int32[T]
  size_t child_tok;    // int32[T]: children tokens, grouped by parent, sorted by (token, id)
  size_t child_id;     // int32[T]: global node id of each slot
  size_t lm_part;      // LmPartial[T][g_lm]
  size_t total;
  int g_lm;            // CTAs of the LM-head kernel (vocabulary ranges)
  int n_splits;        // context splits of the attention kernel
  int split_len;       // keys per context split (multiple of 64)
  int n_parts;         // = n_splits (the tree keys ride with the last split)
  // lazy LM-head schedule only (0 otherwise)
  size_t lz_count;     // int32[max_path + 1]: rows per level
  size_t lz_rows;      // int32[2][T]: node ids of a level's rows (two levels in flight)
  size_t lz_h;         // bf16[2][lz_cap][hidden]: their hidden rows
  int lz_cap;          // T rounded up to 128
  int attn_tc;         // tensor-core attention (attention has the SMs to itself): 1 one
                       // query tile per CTA, 2 two query tiles in ping-pong; 0: the bf16
                       // mma.sync or the fp32 kernel
};

// ---------------------------------------------------------------- device utils

__device__ __forceinline__ void set_status(int* status, int code) {
  atomicCAS(status, 0, code);
}

// A bounded wait gave up: ASD_ERR_TIMEOUT as the call's status (unless an
// earlier error came first) and word 1 of the status block set, which tells
// the later kernels of the call that results of this one are incomplete.
__device__ __forceinline__ void note_timeout(int* status) {
  set_status(status, ASD_ERR_TIMEOUT);
  atomicExch(status + 1, 1);
}

// Folds one vocabulary range's LM-head statistics (max m2, sum of exp(logit -
// m2) s2, lowest argmax a2) into a running (m, s, a); ties in the max keep the
// lowest vocabulary id.  The merge of every row's partials (tail kernel and
// lazy level kernel) uses this, in the same order.
__device__ __forceinline__ void merge_part(float& m, float& s, int& a, float m2, float s2,
                                           int a2) {
  if (m2 == -INFINITY) return;
  if (m == -INFINITY) {
    m = m2;
    s = s2;
    a = a2;
    return;
  }
  const float M = fmaxf(m, m2);
  s = s * exp2f((m - M) * kLog2e) + s2 * exp2f((m2 - M) * kLog2e);
  if (m2 > m) a = a2;
  else if (m2 == m) a = min(a, a2);
  m = M;
}

// Programmatic dependent launch: a kernel launched with programmatic stream
// serialisation may start while its predecessor in the stream still runs;
// pdl_wait() blocks until every predecessor grid has completed and its memory
// is visible, pdl_launch_dependents() lets the next kernel start launching.
// Both are no-ops for kernels launched without the attribute.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void fence_proxy_async() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// Non-blocking test of the phase with the given parity.
__device__ __forceinline__ bool mbar_test_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// Waits until the phase with the given parity has completed.  Gives up after
// `budget` SM clock cycles (kWaitCycles unless the call set another) and
// returns false (the caller records ASD_ERR_TIMEOUT).  try_wait may suspend
// the thread for a while by itself, so a shortened budget (a test making a
// wait give up) polls with the non-blocking test_wait instead.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity,
                                          long long budget = kWaitCycles) {
  if (budget < kWaitCycles) {
    const long long t0 = clock64();
    while (!mbar_test_wait(bar, parity))
      if (clock64() - t0 > budget) return false;
    return true;
  }
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (true) {
#pragma unroll 1
    for (int i = 0; i < 32; ++i)
      if (mbar_try_wait(bar, parity)) return true;
    if (clock64() - t0 > budget) return false;
  }
}

// The wait budget of the kernels of one call: words 2-3 of the workspace
// status block hold it when the host set a shorter one for testing
// (asd_debug_set_wait_cycles), zero otherwise.  Waits for copies and MMAs
// already in flight always use the full kWaitCycles.
__device__ __forceinline__ long long wait_budget(const int* status) {
  const long long b = *reinterpret_cast<const volatile long long*>(status + 2);
  return b > 0 ? b : kWaitCycles;
}

__device__ __forceinline__ uint64_t l2_policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}

__device__ __forceinline__ uint64_t l2_policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}

// 2D tiled TMA load into this CTA's shared memory, completing on `bar`.
// x (innermost coordinate) must be a multiple of 16 bytes / element size.
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* tmap, uint32_t bar,
                                            int x, int y, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      ".L2::cache_hint [%0], [%1, {%3, %4}], [%2], %5;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(bar), "r"(x), "r"(y), "l"(policy)
      : "memory");
}

// 3D tiled TMA load (coordinates x innermost) into shared memory.
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* tmap, uint32_t bar,
                                            int x, int y, int z, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      ".L2::cache_hint [%0], [%1, {%3, %4, %5}], [%2], %6;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(bar), "r"(x), "r"(y), "r"(z), "l"(policy)
      : "memory");
}

// Plain bulk copy global -> shared (both 16-byte aligned, bytes % 16 == 0).
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes,
                                          uint32_t bar, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1], %2, [%3], %4;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(bar), "l"(policy)
      : "memory");
}


__device__ __forceinline__ void prefetch_tmap(const CUtensorMap* tmap) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(tmap)) : "memory");
}

__device__ __forceinline__ float bf16_bits_to_float(uint16_t v) {
  return __uint_as_float(static_cast<uint32_t>(v) << 16);
}

template <typename T>
__device__ __forceinline__ float to_f32(T v);
template <>
__device__ __forceinline__ float to_f32<float>(float v) { return v; }
template <>
__device__ __forceinline__ float to_f32<__nv_bfloat16>(__nv_bfloat16 v) {
  return __bfloat162float(v);
}

template <typename T>
__device__ __forceinline__ T from_f32(float v);
template <>
__device__ __forceinline__ float from_f32<float>(float v) { return v; }
template <>
__device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float v) {
  return __float2bfloat16_rn(v);
}

}  // namespace asd
