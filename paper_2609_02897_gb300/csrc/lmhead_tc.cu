// LM head of the verify pass fused with the margin-rule statistics (Eq. 1),
// bf16 inputs on the sm_103a tensor cores (tcgen05, accumulators in TMEM).
//
// logits[node, v] = hidden[node, :] . W[v, :] are computed as
//   D[128 nodes, up to 256 vocab rows] = hidden_tile[128, K] x W_tile[N, K]^T
// so that TMEM lane i holds node row i and the epilogue thread that owns lane
// i reduces its row over the vocabulary without any cross-thread exchange:
// running max, lowest argmax, sum of exp and the drafted tokens' logits.
// Logits never leave the SM.  Each CTA owns one contiguous vocabulary range
// (one CTA per SM, ranges balanced to 32 rows), streams its slice of W once
// per 128-node tile through a 3-stage TMA ring, and writes one partial
// (max, argmax, sum-exp) per node; the tail kernel merges the ranges.
//
// A stage holds two k-blocks (128 hidden elements) of a 128-row vocabulary
// tile (W, 32 KB: one contiguous bulk copy from the packed weight, or 64-row
// TMA boxes from [V, K] rows) and of the node tile (hidden states, a_rows
// rows).  Reading 256 contiguous bytes of each weight row per stage streams W
// from HBM markedly faster than one k-block of a 256-row tile per stage, and
// the packed order, where every SM's range is one contiguous run, faster
// still.
//
// Warp roles (192 threads): warp 0 TMA producer, warp 1 TMEM allocator and
// MMA issuer, warps 2-5 epilogue (TMEM lane quarters 2, 3, 0, 1).
#include "kernels.h"
#include "lm_epilogue.cuh"
#include "tc.cuh"

namespace asd {
namespace {

constexpr int kM = 128;                        // node rows per MMA = TMEM lanes
constexpr int kKB = 64;                        // hidden elements per k-block (128 B)
constexpr int kKbPerStage = 2;
constexpr int kBTile = kLmTileN * 128;         // W rows of one k-block: 16 KB
constexpr int kGroupBytes = kLmBoxRows * 128;  // one 32-row group of one k-block: 4 KB
constexpr uint32_t kTmemCols = 2 * kLmTileN;   // two accumulators

// Stage slot: the node rows of both k-blocks (a_rows x 128 B each), then W.
// The MMA reads 128 A rows from each k-block's start; rows past a_rows fall
// on the next block of the same slot and only feed accumulator rows that
// no node owns.
__host__ __device__ constexpr int lm_a_bytes(int a_rows) { return kKbPerStage * a_rows * 128; }
__host__ __device__ constexpr int lm_slot_bytes(int a_rows) {
  return lm_a_bytes(a_rows) + kKbPerStage * kBTile;
}

__global__ void __launch_bounds__(192, 1)
    lmhead_tc_kernel(const __grid_constant__ LmMaps maps, const LmParams p) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t s_full[kLmStages];
  __shared__ __align__(8) uint64_t s_empty[kLmStages];
  __shared__ __align__(8) uint64_t s_tfull[2];
  __shared__ __align__(8) uint64_t s_tempty[2];
  __shared__ __align__(8) uint64_t s_mma_done;
  __shared__ uint32_t s_tmem;
  __shared__ volatile int s_abort;
  __shared__ int s_pack_bad;
  __shared__ int s_issued[kLmStages];   // fills issued per stage (drained before exit)

  // W and the hidden states are inputs of the step, not results of earlier
  // kernels: only the epilogue (children lists, l_draft) waits for them
  pdl_launch_dependents();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long budget = wait_budget(p.status);

  // this CTA's vocabulary range, in whole groups of kLmBoxRows rows
  const int ngroups = (p.V + kLmBoxRows - 1) / kLmBoxRows;
  const int gs = lm_range_begin(blockIdx.x, p.g_lm, ngroups);
  const int ge = lm_range_begin(blockIdx.x + 1, p.g_lm, ngroups);
  const int vs = gs * kLmBoxRows;
  const int ve = min(p.V, ge * kLmBoxRows);
  const int nnt = (p.T + kM - 1) / kM;
  const int nkb = (p.K + kKB - 1) / kKB;
  const int nkp = (nkb + kKbPerStage - 1) / kKbPerStage;   // stages per tile
  const int a_blk = p.a_rows * 128;                         // one k-block of node rows
  const int slot = lm_slot_bytes(p.a_rows);

  uint32_t base = smem_u32(smem_raw);
  base += (1024u - (base & 1023u)) & 1023u;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kLmStages; ++s) {
      mbar_init(smem_u32(&s_full[s]), 1);
      mbar_init(smem_u32(&s_empty[s]), 1);
      s_issued[s] = 0;
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(smem_u32(&s_tfull[a]), 1);
      mbar_init(smem_u32(&s_tempty[a]), 4);
    }
    mbar_init(smem_u32(&s_mma_done), 1);
    s_abort = 0;
    // a packed weight must come from asd_pack_lm_head for this vocabulary,
    // width and range count; otherwise nothing is loaded and the error recorded
    int bad = 0;
    if (p.w_packed) {
      const LmPackHeader* h = reinterpret_cast<const LmPackHeader*>(p.w_packed);
      bad = (h->magic != kLmPackMagic || h->version != kLmPackVersion || h->vocab != p.V ||
             h->hidden != p.K || h->ranges != p.g_lm);
      if (bad) set_status(p.status, ASD_ERR_SHAPE);
    }
    s_pack_bad = bad;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&s_tmem), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;
  // vocabulary tiles of this CTA (none when a packed weight does not match)
  const int nvt = (ve > vs && !s_pack_bad) ? (ve - vs + kLmTileN - 1) / kLmTileN : 0;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    uint64_t pol_w = 0, pol_h = 0;
    if (lane == 0) {
      prefetch_tmap(&maps.h);
      if (!p.w_packed) {
        prefetch_tmap(&maps.w64);
        prefetch_tmap(&maps.w32);
      }
      pol_w = l2_policy_evict_first();
      pol_h = l2_policy_evict_last();
    }
    int stage = 0;
    uint32_t ph = 0;
    bool ok = true;
    for (int nt = 0; nt < nnt && ok; ++nt) {
      for (int vt = 0; vt < nvt && ok; ++vt) {
        const int v0 = vs + vt * kLmTileN;
        const int ng = (min(kLmTileN, ve - v0) + kLmBoxRows - 1) / kLmBoxRows;  // 32-row groups
        for (int kp = 0; kp < nkp; ++kp) {
          const uint32_t full = smem_u32(&s_full[stage]);
          ok = __shfl_sync(0xffffffffu, mbar_wait(smem_u32(&s_empty[stage]), ph ^ 1u, budget), 0);
          if (!ok || s_abort) {
            ok = false;
            break;
          }
          if (lane == 0) {
            const uint32_t a_s = base + stage * slot;
            const uint32_t b_s = a_s + lm_a_bytes(p.a_rows);
            const int nk = min(kKbPerStage, nkb - kp * kKbPerStage);
            mbar_expect_tx(full, static_cast<uint32_t>(nk * (a_blk + ng * kGroupBytes)));
            for (int kk = 0; kk < nk; ++kk)
              tma_load_2d(a_s + kk * a_blk, &maps.h, full, (kp * kKbPerStage + kk) * kKB,
                          nt * kM, pol_h);
            if (p.w_packed) {
              // both k-blocks of the stage are one contiguous run of the packed weight
              const size_t off = kLmPackHeader +
                                 static_cast<size_t>(kGroupBytes) *
                                     (static_cast<size_t>(nkb) * (v0 / kLmBoxRows) +
                                      static_cast<size_t>(kp * kKbPerStage) * ng);
              bulk_load(b_s, p.w_packed + off, static_cast<uint32_t>(nk * ng * kGroupBytes), full,
                        pol_w);
            } else {
              for (int kk = 0; kk < nk; ++kk) {
                const int kx = (kp * kKbPerStage + kk) * kKB;
                int j = 0;
                for (; j + 1 < ng; j += 2)
                  tma_load_2d(b_s + kk * kBTile + j * kGroupBytes, &maps.w64, full, kx,
                              v0 + j * kLmBoxRows, pol_w);
                if (j < ng)
                  tma_load_2d(b_s + kk * kBTile + j * kGroupBytes, &maps.w32, full, kx,
                              v0 + j * kLmBoxRows, pol_w);
              }
            }
            ++s_issued[stage];
          }
          __syncwarp();
          if (++stage == kLmStages) {
            stage = 0;
            ph ^= 1u;
          }
        }
      }
    }
    if (!ok && lane == 0) {
      note_timeout(p.status);
      s_abort = 1;
    }
    // every fill this CTA issued has landed before the CTA may leave
    if (lane == 0)
      for (int s = 0; s < kLmStages; ++s)
        if (s_issued[s] > 0)
          mbar_wait(smem_u32(&s_full[s]), static_cast<uint32_t>((s_issued[s] - 1) & 1));
    __syncwarp();
  } else if (warp == 1) {
    // --------------------------------------------------------------- MMA issuer
    int stage = 0;
    uint32_t ph = 0;
    int acc = 0;
    uint32_t aph = 0;
    bool ok = true;
    for (int nt = 0; nt < nnt && ok; ++nt) {
      for (int vt = 0; vt < nvt && ok; ++vt) {
        const int v0 = vs + vt * kLmTileN;
        const int nrows = min(kLmTileN, ve - v0);
        const uint32_t idesc = idesc_bf16(kM, (nrows + 15) & ~15);
        // the second k-block's W rows: a fixed slot, or right behind the first
        // block's ng groups in the packed layout
        const int b_kstride =
            p.w_packed ? ((nrows + kLmBoxRows - 1) / kLmBoxRows) * kGroupBytes : kBTile;
        ok = __shfl_sync(0xffffffffu, mbar_wait(smem_u32(&s_tempty[acc]), aph ^ 1u, budget), 0);
        if (!ok || s_abort) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + static_cast<uint32_t>(acc * kLmTileN);
        for (int kp = 0; kp < nkp; ++kp) {
          ok = __shfl_sync(0xffffffffu, mbar_wait(smem_u32(&s_full[stage]), ph, budget), 0);
          if (!ok || s_abort) {
            ok = false;
            break;
          }
          tc_fence_after();
          if (lane == 0) {
            const uint32_t a_s = base + stage * slot;
            const uint32_t b_s = a_s + lm_a_bytes(p.a_rows);
            const int nk = min(kKbPerStage, nkb - kp * kKbPerStage);
            for (int kk = 0; kk < nk; ++kk) {
#pragma unroll
              for (int k = 0; k < kKB / 16; ++k)
                tc_mma(d, sw128_desc(a_s + kk * a_blk + 32 * k),
                       sw128_desc(b_s + kk * b_kstride + 32 * k), idesc,
                       (kp | kk | k) != 0 ? 1u : 0u);
            }
            tc_commit(smem_u32(&s_empty[stage]));
          }
          __syncwarp();
          if (++stage == kLmStages) {
            stage = 0;
            ph ^= 1u;
          }
        }
        if (!ok) break;
        if (lane == 0) tc_commit(smem_u32(&s_tfull[acc]));
        __syncwarp();
        acc ^= 1;
        if (acc == 0) aph ^= 1u;
      }
    }
    if (!ok && lane == 0) {
      note_timeout(p.status);
      s_abort = 1;
    }
    // every tcgen05 operation of this thread is done before TMEM is released
    if (lane == 0) {
      tc_commit(smem_u32(&s_mma_done));
      mbar_wait(smem_u32(&s_mma_done), 0);
    }
    __syncwarp();
  } else {
    // ----------------------------------------------------------------- epilogue
    const int q = warp & 3;
    const int row = q * 32 + lane;
    pdl_wait();
    int acc = 0;
    uint32_t aph = 0;
    bool ok = true;
    for (int nt = 0; nt < nnt && ok; ++nt) {
      const int node = nt * kM + row;
      const bool active = node < p.T;
      RowState st;
      row_state_init(st, active, node, vs, p.child_start, p.child_cnt, p.child_tok, p.T);
      for (int vt = 0; vt < nvt; ++vt) {
        const int v0 = vs + vt * kLmTileN;
        const int nrows = min(kLmTileN, ve - v0);
        ok = __shfl_sync(0xffffffffu, mbar_wait(smem_u32(&s_tfull[acc]), aph, budget), 0);
        if (!ok || s_abort) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t taddr = tmem + (static_cast<uint32_t>(q * 32) << 16) +
                               static_cast<uint32_t>(acc * kLmTileN);
        const int nchunks = (nrows + 31) / 32;
        for (int c = 0; c < nchunks; ++c) {
          float r[32];
          tmem_ld32(taddr + 32 * c, r);
          if (active)
            row_chunk(st, r, v0 + 32 * c, min(32, nrows - 32 * c), p.child_tok, p.child_id,
                      p.l_draft, p.T);
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&s_tempty[acc]));
        acc ^= 1;
        if (acc == 0) aph ^= 1u;
      }
      if (ok && active) {
        LmPartial part;
        part.m = st.m;
        part.s = st.s;
        part.a = st.a;
        part.pad = 0;
        p.part[static_cast<size_t>(node) * p.g_lm + blockIdx.x] = part;
      }
    }
    if (!ok && lane == 0) {
      note_timeout(p.status);
      s_abort = 1;
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, kTmemCols);
}

// ----------------------------------------------------------------------------
// Wide variant for more than 128 nodes.  Two node tiles share every streamed
// W stage and each MMA covers 256 vocabulary rows, D[128 nodes, 256 vocab
// rows], so that one MMA reads 12 KB of shared memory per 128 x 256 x 16
// product instead of 8 KB per 128 x 128 x 16: with 128-row vocabulary tiles
// the tensor cores wait on shared-memory reads.  A stage holds one k-block of
// the 256 W rows (two packed 128-row tiles, or 64-row TMA boxes) and of the
// CTA's two node tiles; the hidden rows (a few MB) stay in L2 across the
// vocabulary tiles.  TMEM holds one 256-column accumulator per node tile, each
// with its own full / empty barriers, so the MMAs into one resume as soon as
// the epilogue has drained it.
//
// CL = 2: the CTAs come in clusters of two that own two adjacent vocabulary
// ranges together and take alternate node pairs.  Each CTA copies one of the
// two 128-row halves of every W stage and multicasts it to both, so every SM
// pulls 48 KB per stage instead of 64 and W crosses HBM once per four node
// tiles.  A stage is refilled only after both CTAs' MMAs have read it (each
// CTA's commit arrives on both CTAs' empty barriers); both CTAs run the same
// sequence of stages, a CTA without a node pair in the last round still
// copying its half.  Every thread keeps one running state per vocabulary
// range and writes one partial per range, so the statistics are those of
// CTAs that own one range each, bit for bit.
//
// Warp roles (352 threads): warp 0 TMA producer, warp 1 TMEM allocator and
// MMA issuer for node tile 0 of every pair, warp 10 MMA issuer for node tile
// 1 (two issuing threads: a barrier wait costs its thread a few hundred
// cycles, and one thread's waits then overlap the other's MMAs), warps 2-5
// and 6-9 two epilogue groups; group g drains the accumulator of the pair's
// node tile g, so that both accumulators of a vocabulary tile are drained at
// once and the MMAs of the next tile wait for one drain instead of two.
constexpr int kWideN = 2 * kLmTileN;                 // vocabulary rows per MMA
constexpr int kWideG = 2;                            // node tiles per W stage and CTA
constexpr int kWideStages = 3;
constexpr int kWideA = kM * 128;                     // one node tile's k-block: 16 KB
constexpr int kWideSlot = kWideG * kWideA + kWideN * 128;   // 64 KB
constexpr uint32_t kWideTmemCols = kWideG * kWideN;  // 512
constexpr int kTileGroups = kLmTileN / kLmBoxRows;   // range groups per packed tile
constexpr int kWideThreads = 352;                    // producer, 2 MMA issuers, 2 epilogue groups

__device__ __forceinline__ uint32_t cta_rank_in_cluster() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

__device__ __forceinline__ void cluster_barrier() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;"
               ::: "memory");
}

// The shared::cluster address of this CTA's shared variable at `local` in the
// CTA of cluster rank `rank`.
__device__ __forceinline__ uint32_t cluster_addr(uint32_t local, int rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(local), "r"(rank));
  return r;
}
__device__ __forceinline__ void st_cluster_u32(uint32_t addr, uint32_t v) {
  asm volatile("st.shared::cluster.u32 [%0], %1;" ::"r"(addr), "r"(v) : "memory");
}
__device__ __forceinline__ uint32_t ld_cluster_u32(uint32_t addr) {
  uint32_t v;
  asm volatile("ld.shared::cluster.u32 %0, [%1];" : "=r"(v) : "r"(addr) : "memory");
  return v;
}
// Counts `bytes` as arrived on the barrier's current phase without a copy.
__device__ __forceinline__ void mbar_complete_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.complete_tx.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}

// Bulk copy global -> shared of every CTA in `mask` (same offset, each CTA's
// barrier at `bar`'s offset receives the bytes).
__device__ __forceinline__ void bulk_load_mc(uint32_t dst, const void* src, uint32_t bytes,
                                             uint32_t bar, uint16_t mask, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.multicast::cluster"
      ".L2::cache_hint [%0], [%1], %2, [%3], %4, %5;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(bar), "h"(mask), "l"(policy)
      : "memory");
}

__device__ __forceinline__ void tma_load_2d_mc(uint32_t dst, const CUtensorMap* tmap, uint32_t bar,
                                               int x, int y, uint16_t mask, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      ".multicast::cluster.L2::cache_hint [%0], [%1, {%3, %4}], [%2], %5, %6;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(bar), "r"(x), "r"(y), "h"(mask), "l"(policy)
      : "memory");
}

// Arrive on `bar` of every CTA in `mask` once this thread's earlier tcgen05
// operations are done.
__device__ __forceinline__ void tc_commit_mc(uint32_t bar, uint16_t mask) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
      " [%0], %1;" ::"r"(bar), "h"(mask)
      : "memory");
}

// The CTA's (cluster's) vocabulary: CL adjacent ranges, each cut into packed
// 128-row tiles from its start; tile j of the concatenation.
struct WideVocab {
  int gs0, ge0, nt0;         // first range: 32-row groups [gs0, ge0), packed tiles
  int gs1, ge1, nt1;         // second range (CL = 2), else empty
  int ntiles;                // packed tiles of all ranges
  __device__ __forceinline__ void tile(int j, int V, int& q, int& g0, int& ng, int& v0,
                                       int& rows) const {
    q = j < nt0 ? 0 : 1;
    g0 = q ? gs1 + (j - nt0) * kTileGroups : gs0 + j * kTileGroups;
    ng = min(kTileGroups, (q ? ge1 : ge0) - g0);
    v0 = g0 * kLmBoxRows;
    rows = min(ng * kLmBoxRows, V - v0);
  }
};

template <int CL>
__global__ void __launch_bounds__(kWideThreads, 1)
    lmhead_wide_kernel(const __grid_constant__ LmMaps maps, const LmParams p) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t s_full[kWideStages];
  __shared__ __align__(8) uint64_t s_empty[kWideStages];
  __shared__ __align__(8) uint64_t s_tfull[kWideG];
  __shared__ __align__(8) uint64_t s_tempty[kWideG];
  __shared__ __align__(8) uint64_t s_mma_done[kWideG];   // each MMA issuer's own drain
  __shared__ uint32_t s_tmem;
  __shared__ volatile int s_abort;
  __shared__ int s_pack_bad;
  __shared__ int s_issued[kWideStages];   // fills issued per stage (drained before exit)

  pdl_launch_dependents();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long budget = wait_budget(p.status);
  const int rank = CL == 2 ? static_cast<int>(cta_rank_in_cluster()) : 0;
  const uint16_t both = static_cast<uint16_t>((1u << CL) - 1u);
  // hidden rows of this launch: T, or (one level of the lazy schedule) the
  // count and the rows that the previous kernel wrote
  int nrow = p.T;
  if (p.t_dev) {
    pdl_wait();
    nrow = min(max(*p.t_dev, 0), p.T);
  }

  const int ngroups = (p.V + kLmBoxRows - 1) / kLmBoxRows;
  const int cid = blockIdx.x / CL;                       // the ranges cid*CL .. cid*CL+CL-1
  WideVocab voc;
  voc.gs0 = lm_range_begin(cid * CL, p.g_lm, ngroups);
  voc.ge0 = lm_range_begin(cid * CL + 1, p.g_lm, ngroups);
  voc.gs1 = CL == 2 ? voc.ge0 : 0;
  voc.ge1 = CL == 2 ? lm_range_begin(cid * CL + 2, p.g_lm, ngroups) : 0;
  voc.nt0 = (voc.ge0 - voc.gs0 + kTileGroups - 1) / kTileGroups;
  voc.nt1 = (voc.ge1 - voc.gs1 + kTileGroups - 1) / kTileGroups;
  voc.ntiles = voc.nt0 + voc.nt1;
  const int nnt = (nrow + kM - 1) / kM;                  // node tiles
  const int nng = (nnt + kWideG - 1) / kWideG;           // node-tile pairs
  const int nit = (nng + CL - 1) / CL;                   // rounds: pair i*CL + rank in round i
  const int nkb = (p.K + kKB - 1) / kKB;

  uint32_t base = smem_u32(smem_raw);
  base += (1024u - (base & 1023u)) & 1023u;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kWideStages; ++s) {
      mbar_init(smem_u32(&s_full[s]), 1);
      mbar_init(smem_u32(&s_empty[s]), kWideG * CL);   // both issuers of every CTA read it
      s_issued[s] = 0;
    }
    for (int a = 0; a < kWideG; ++a) {
      mbar_init(smem_u32(&s_tfull[a]), 1);
      mbar_init(smem_u32(&s_tempty[a]), 4);
    }
    for (int j = 0; j < kWideG; ++j) mbar_init(smem_u32(&s_mma_done[j]), 1);
    s_abort = 0;
    int bad = 0;
    if (p.w_packed) {
      const LmPackHeader* h = reinterpret_cast<const LmPackHeader*>(p.w_packed);
      bad = (h->magic != kLmPackMagic || h->version != kLmPackVersion || h->vocab != p.V ||
             h->hidden != p.K || h->ranges != p.g_lm);
      if (bad) set_status(p.status, ASD_ERR_SHAPE);
    }
    s_pack_bad = bad;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&s_tmem), kWideTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  if (CL == 2) cluster_barrier();   // the peer's barriers exist before any multicast
  tc_fence_after();
  const uint32_t tmem = s_tmem;
  // 256-row vocabulary tiles (pairs of packed tiles); none when a packed
  // weight does not match (both CTAs of a cluster read the same header)
  const int nvt = s_pack_bad ? 0 : (voc.ntiles + 1) / 2;
  // a wait that gives up stops this CTA and its peer
  auto abort_cta = [&]() {
    note_timeout(p.status);
    s_abort = 1;
    if (CL == 2)
      st_cluster_u32(cluster_addr(smem_u32(const_cast<int*>(&s_abort)), rank ^ 1), 1u);
  };

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    uint64_t pol_w = 0, pol_h = 0;
    if (lane == 0) {
      prefetch_tmap(&maps.h);
      if (!p.w_packed) {
        prefetch_tmap(&maps.w64);
        prefetch_tmap(&maps.w32);
      }
      pol_w = l2_policy_evict_first();
      pol_h = l2_policy_evict_last();
    }
    int stage = 0;
    uint32_t ph = 0;
    bool ok = true;
    for (int it = 0; it < nit && ok; ++it) {
      const int pi = it * CL + rank;                       // this CTA's node pair
      const int gn = pi < nng ? min(kWideG, nnt - pi * kWideG) : 0;
      for (int vt = 0; vt < nvt && ok; ++vt) {
        int q[2], g0[2], ng[2], v0[2], rows[2];
        int wbytes = 0;
#pragma unroll
        for (int hf = 0; hf < 2; ++hf) {
          ng[hf] = 0;
          g0[hf] = 0;
          if (2 * vt + hf < voc.ntiles) {
            voc.tile(2 * vt + hf, p.V, q[hf], g0[hf], ng[hf], v0[hf], rows[hf]);
            wbytes += ng[hf] * kGroupBytes;
          }
        }
        for (int kb = 0; kb < nkb; ++kb) {
          const uint32_t full = smem_u32(&s_full[stage]);
          ok = __shfl_sync(0xffffffffu, mbar_wait(smem_u32(&s_empty[stage]), ph ^ 1u, budget), 0);
          if (!ok || s_abort) {
            ok = false;
            break;
          }
          if (lane == 0) {
            const uint32_t a_s = base + stage * kWideSlot;
            const uint32_t b_s = a_s + kWideG * kWideA;
            // every W byte of the stage lands here (half of it from the peer)
            mbar_expect_tx(full, static_cast<uint32_t>(gn * kWideA + wbytes));
            for (int j = 0; j < gn; ++j)
              tma_load_2d(a_s + j * kWideA, &maps.h, full, kb * kKB, (pi * kWideG + j) * kM,
                          pol_h);
#pragma unroll
            for (int hf = 0; hf < 2; ++hf) {
              if (ng[hf] == 0 || (CL == 2 && hf != rank)) continue;   // the peer's half
              const uint32_t dst = b_s + hf * kBTile;
              if (p.w_packed) {
                const size_t off = kLmPackHeader +
                                   static_cast<size_t>(kGroupBytes) *
                                       (static_cast<size_t>(nkb) * g0[hf] +
                                        static_cast<size_t>(kb) * ng[hf]);
                if (CL == 2)
                  bulk_load_mc(dst, p.w_packed + off, static_cast<uint32_t>(ng[hf] * kGroupBytes),
                               full, both, pol_w);
                else
                  bulk_load(dst, p.w_packed + off, static_cast<uint32_t>(ng[hf] * kGroupBytes),
                            full, pol_w);
              } else {
                const int vh = g0[hf] * kLmBoxRows;
                int j = 0;
                for (; j + 1 < ng[hf]; j += 2) {
                  if (CL == 2)
                    tma_load_2d_mc(dst + j * kGroupBytes, &maps.w64, full, kb * kKB,
                                   vh + j * kLmBoxRows, both, pol_w);
                  else
                    tma_load_2d(dst + j * kGroupBytes, &maps.w64, full, kb * kKB,
                                vh + j * kLmBoxRows, pol_w);
                }
                if (j < ng[hf]) {
                  if (CL == 2)
                    tma_load_2d_mc(dst + j * kGroupBytes, &maps.w32, full, kb * kKB,
                                   vh + j * kLmBoxRows, both, pol_w);
                  else
                    tma_load_2d(dst + j * kGroupBytes, &maps.w32, full, kb * kKB,
                                vh + j * kLmBoxRows, pol_w);
                }
              }
            }
            ++s_issued[stage];
          }
          __syncwarp();
          if (++stage == kWideStages) {
            stage = 0;
            ph ^= 1u;
          }
        }
      }
    }
    if (!ok && lane == 0) abort_cta();
  } else if (warp == 1 || warp == 10) {
    // ------------------------------------------------------------ MMA issuers
    // Two issuing threads, one per node tile of the pair (warp 1: tile 0,
    // warp 10: tile 1), so that the one's barrier waits overlap the other's
    // MMAs.  Both read every stage and both release it.  Accumulator use u
    // (counted over the kernel) goes to TMEM buffer u % 2; its empty barrier
    // completes once per lap.
    const int j = warp == 1 ? 0 : 1;
    int stage = 0;
    uint32_t ph = 0;
    int used = 0;
    bool ok = true;
    for (int it = 0; it < nit && ok; ++it) {
      const int pi = it * CL + rank;
      const int gn = pi < nng ? min(kWideG, nnt - pi * kWideG) : 0;
      for (int vt = 0; vt < nvt && ok; ++vt) {
        // N covers the low half's rows, or all 128 of them and the high half's
        int q, g0, ng, v0, rows_lo, rows_hi = 0;
        voc.tile(2 * vt, p.V, q, g0, ng, v0, rows_lo);
        if (2 * vt + 1 < voc.ntiles) voc.tile(2 * vt + 1, p.V, q, g0, ng, v0, rows_hi);
        const int ncols = rows_hi > 0 ? kLmTileN + rows_hi : rows_lo;
        const uint32_t idesc = idesc_bf16(kM, (ncols + 15) & ~15);
        const int u = used + j;
        const int acc = u % kWideG;
        for (int kb = 0; kb < nkb && ok; ++kb) {
          ok = __shfl_sync(0xffffffffu, mbar_wait(smem_u32(&s_full[stage]), ph, budget), 0);
          if (!ok || s_abort) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_s = base + stage * kWideSlot;
          const uint32_t b_s = a_s + kWideG * kWideA;
          if (j < gn) {
            if (kb == 0) {
              // the epilogue must have drained this buffer's previous tile
              ok = __shfl_sync(
                  0xffffffffu,
                  mbar_wait(smem_u32(&s_tempty[acc]), ((static_cast<uint32_t>(u / kWideG)) & 1u) ^ 1u,
                            budget),
                  0);
              if (!ok || s_abort) {
                ok = false;
                break;
              }
              tc_fence_after();
            }
            if (lane == 0) {
              const uint32_t d = tmem + static_cast<uint32_t>(acc * kWideN);
#pragma unroll
              for (int k = 0; k < kKB / 16; ++k)
                tc_mma(d, sw128_desc(a_s + j * kWideA + 32 * k), sw128_desc(b_s + 32 * k), idesc,
                       (kb | k) != 0 ? 1u : 0u);
              if (kb == nkb - 1) tc_commit(smem_u32(&s_tfull[acc]));
            }
            __syncwarp();
          }
          // the stage is free for refilling once both issuers of every CTA of
          // the cluster have read it
          if (lane == 0) {
            if (CL == 2)
              tc_commit_mc(smem_u32(&s_empty[stage]), both);
            else
              tc_commit(smem_u32(&s_empty[stage]));
          }
          __syncwarp();
          if (++stage == kWideStages) {
            stage = 0;
            ph ^= 1u;
          }
        }
        used += gn;
      }
    }
    if (!ok && lane == 0) abort_cta();
    // every tcgen05 operation of this thread, the commits included, is done
    // before the CTA leaves the cluster
    if (lane == 0) {
      tc_commit(smem_u32(&s_mma_done[j]));
      mbar_wait(smem_u32(&s_mma_done[j]), 0);
    }
    __syncwarp();
  } else {
    // ----------------------------------------------------------------- epilogue
    // Two groups of four warps: group g drains the accumulator of node tile
    // j = g of the current pair, so both accumulators of a vocabulary tile
    // drain at once.  Thread `row` of a group owns TMEM lane `row`: row `row`
    // of its node tile, one running state per vocabulary range.
    const int q4 = warp & 3;
    const int row = q4 * 32 + lane;
    const int g = (warp - 2) >> 2;
    pdl_wait();
    int used = 0;
    bool ok = true;
    for (int it = 0; it < nit && ok; ++it) {
      const int pi = it * CL + rank;
      const int gn = pi < nng ? min(kWideG, nnt - pi * kWideG) : 0;
      const int r = (pi * kWideG + g) * kM + row;
      const int node = (g < gn && r < nrow && p.row_node) ? p.row_node[r] : r;
      const bool act = g < gn && r < nrow && node >= 0 && node < p.T;
      RowState st[CL];
#pragma unroll
      for (int qq = 0; qq < CL; ++qq)
        row_state_init(st[qq], act, node, (qq ? voc.gs1 : voc.gs0) * kLmBoxRows, p.child_start,
                       p.child_cnt, p.child_tok, p.T);
      for (int vt = 0; vt < nvt && ok; ++vt) {
        if (g < gn) {
          const int u = used + g;
          const int acc = u % kWideG;
          ok = __shfl_sync(0xffffffffu,
                           mbar_wait(smem_u32(&s_tfull[acc]), (static_cast<uint32_t>(u / kWideG)) & 1u,
                                     budget),
                           0);
          if (!ok || s_abort) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t taddr = tmem + (static_cast<uint32_t>(q4 * 32) << 16) +
                                 static_cast<uint32_t>(acc * kWideN);
          // the two packed tiles of the 256 columns, each from its own vocabulary base
#pragma unroll
          for (int hf = 0; hf < 2; ++hf) {
            if (2 * vt + hf >= voc.ntiles) break;
            int q, g0, ng, v0, rows;
            voc.tile(2 * vt + hf, p.V, q, g0, ng, v0, rows);
            for (int c = 0; c < rows; c += 64) {
              float x[64];
              tmem_ld64(taddr + hf * kLmTileN + c, x);
              if (act) {
                float (&x0)[32] = *reinterpret_cast<float(*)[32]>(&x[0]);
                float (&x1)[32] = *reinterpret_cast<float(*)[32]>(&x[32]);
                const int n0 = min(32, rows - c), n1 = min(32, rows - c - 32);
                if (CL == 2 && q == 1) {
                  row_chunk(st[CL - 1], x0, v0 + c, n0, p.child_tok, p.child_id, p.l_draft, p.T);
                  if (n1 > 0)
                    row_chunk(st[CL - 1], x1, v0 + c + 32, n1, p.child_tok, p.child_id,
                              p.l_draft, p.T);
                } else {
                  row_chunk(st[0], x0, v0 + c, n0, p.child_tok, p.child_id, p.l_draft, p.T);
                  if (n1 > 0)
                    row_chunk(st[0], x1, v0 + c + 32, n1, p.child_tok, p.child_id, p.l_draft, p.T);
                }
              }
            }
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(smem_u32(&s_tempty[acc]));
        }
        used += gn;
      }
      if (ok && g < gn && r < nrow) {   // partials by row, one per range
#pragma unroll
        for (int qq = 0; qq < CL; ++qq) {
          LmPartial part;
          part.m = st[qq].m;
          part.s = st[qq].s;
          part.a = st[qq].a;
          part.pad = 0;
          p.part[static_cast<size_t>(r) * p.g_lm + cid * CL + qq] = part;
        }
      }
    }
    if (!ok && lane == 0) abort_cta();
  }

  tc_fence_before();
  __syncthreads();
  // From here on neither producer of the cluster issues a copy.  Every copy
  // that lands in this CTA's shared memory (its own and, with CL = 2, the
  // peer's half of W) has landed before the CTA leaves: the producer waits
  // for the last phase of every stage.  The producers of a cluster are at
  // most one phase of a stage apart (a fill needs both CTAs' MMAs to have
  // read the previous one), so a phase that only one of them filled is either
  // armed here for the peer's bytes or has the missing peer bytes completed
  // here, and then waited for like the others.
  if (CL == 2) cluster_barrier();
  if (warp == 0 && lane == 0) {
    for (int s = 0; s < kWideStages; ++s) {
      const uint32_t full = smem_u32(&s_full[s]);
      const int mine = s_issued[s];
      const int peer =
          CL == 2 ? static_cast<int>(ld_cluster_u32(cluster_addr(smem_u32(&s_issued[s]), rank ^ 1)))
                  : mine;
      // bytes of the peer's half of W in fill f of stage s (stage sequence n)
      auto peer_bytes = [&](int f) -> uint32_t {
        const int n = f * kWideStages + s;
        const int vt = (n / nkb) % max(nvt, 1);
        const int t = 2 * vt + (rank ^ 1);
        if (CL != 2 || t >= voc.ntiles) return 0u;
        int q, g0, ng, v0, rows;
        voc.tile(t, p.V, q, g0, ng, v0, rows);
        return static_cast<uint32_t>(ng * kGroupBytes);
      };
      if (peer == mine + 1) {
        if (mine > 0) mbar_wait(full, static_cast<uint32_t>((mine - 1) & 1));
        mbar_expect_tx(full, peer_bytes(mine));
        mbar_wait(full, static_cast<uint32_t>(mine & 1));
      } else if (mine == peer + 1) {
        if (mine > 1) mbar_wait(full, static_cast<uint32_t>((mine - 2) & 1));
        mbar_complete_tx(full, peer_bytes(mine - 1));
        mbar_wait(full, static_cast<uint32_t>((mine - 1) & 1));
      } else if (mine > 0) {
        mbar_wait(full, static_cast<uint32_t>((mine - 1) & 1));
      }
    }
  }
  if (CL == 2) cluster_barrier();   // the peer's copies into this CTA have landed as well
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, kWideTmemCols);
  if (CL == 2) cluster_barrier();   // no multicast or remote arrive targets a CTA that left
}

}  // namespace

// One CTA per (32-row group g, k-block kb): copies that 4 KB block of W into
// its place in the packed layout, swizzled, zeros past V.  Block (0, 0) also
// writes the header.
__global__ void __launch_bounds__(256) lm_pack_kernel(const __nv_bfloat16* w, uint8_t* out,
                                                      int V, int K, int ranges) {
  const int g = blockIdx.x, kb = blockIdx.y;
  const int ngroups = gridDim.x, nkb = gridDim.y;
  // the range holding group g, and its tile
  int c = static_cast<int>(static_cast<long long>(g) * ranges / ngroups);
  while (c + 1 < ranges && lm_range_begin(c + 1, ranges, ngroups) <= g) ++c;
  while (c > 0 && lm_range_begin(c, ranges, ngroups) > g) --c;
  const int gs = lm_range_begin(c, ranges, ngroups), ge = lm_range_begin(c + 1, ranges, ngroups);
  const int tile_groups = kLmTileN / kLmBoxRows;
  const int g0 = gs + ((g - gs) / tile_groups) * tile_groups;
  const int ng = min(tile_groups, ge - g0);
  const size_t blk = kLmPackHeader + static_cast<size_t>(kGroupBytes) *
                                         (static_cast<size_t>(nkb) * g0 + static_cast<size_t>(kb) * ng +
                                          (g - g0));
  const int r = threadIdx.x >> 3, ch = threadIdx.x & 7;
  const int row = g * kLmBoxRows + r, col = kb * kKB + ch * 8;
  uint4 v = make_uint4(0u, 0u, 0u, 0u);
  if (row < V && col < K)  // K % 8 == 0: a chunk is all in or all out
    v = *reinterpret_cast<const uint4*>(w + static_cast<size_t>(row) * K + col);
  *reinterpret_cast<uint4*>(out + blk + r * 128 + ((ch ^ (r & 7)) << 4)) = v;
  if (g == 0 && kb == 0 && threadIdx.x < kLmPackHeader / 4) {
    uint32_t word = 0;
    switch (threadIdx.x) {
      case 0: word = kLmPackMagic; break;
      case 1: word = kLmPackVersion; break;
      case 2: word = static_cast<uint32_t>(V); break;
      case 3: word = static_cast<uint32_t>(K); break;
      case 4: word = static_cast<uint32_t>(ranges); break;
      default: break;
    }
    reinterpret_cast<uint32_t*>(out)[threadIdx.x] = word;
  }
}

size_t lmhead_tc_smem_bytes(int a_rows) {
  return 1024 + static_cast<size_t>(kLmStages) * lm_slot_bytes(a_rows);
}

size_t lm_packed_bytes(int vocab, int hidden) {
  const size_t ngroups = (static_cast<size_t>(vocab) + kLmBoxRows - 1) / kLmBoxRows;
  const size_t nkb = (static_cast<size_t>(hidden) + kKB - 1) / kKB;
  return kLmPackHeader + ngroups * nkb * kGroupBytes;
}

cudaError_t launch_lm_pack(const void* w, void* w_packed, int vocab, int hidden, int ranges,
                           cudaStream_t s) {
  const unsigned ngroups = static_cast<unsigned>((vocab + kLmBoxRows - 1) / kLmBoxRows);
  const unsigned nkb = static_cast<unsigned>((hidden + kKB - 1) / kKB);
  if (nkb > 65535u) return cudaErrorInvalidValue;
  lm_pack_kernel<<<dim3(ngroups, nkb), 256, 0, s>>>(static_cast<const __nv_bfloat16*>(w),
                                                    static_cast<uint8_t*>(w_packed), vocab,
                                                    hidden, ranges);
  return cudaGetLastError();
}

namespace {
template <int CL>
cudaError_t launch_wide(const LmParams& p, const LmMaps& maps, cudaStream_t s) {
  const size_t smem = 1024 + static_cast<size_t>(kWideStages) * kWideSlot;
  cudaError_t err = set_smem_attrs(lmhead_wide_kernel<CL>, smem);
  if (err != cudaSuccess) return err;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.g_lm);
  cfg.blockDim = dim3(kWideThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = CL;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, lmhead_wide_kernel<CL>, maps, p);
}
}  // namespace

int lmhead_bf16_variant(const LmParams& p) {
  if (p.T <= kM && !p.t_dev) return 1;
  // several node tiles, or a row count known on the device only: the wide
  // kernel (full 128-row node boxes).  Clusters of two halve the W traffic
  // (each W stage is read once per cluster) and move their CTAs in lock step
  // through the rounds of node pairs, so they pay unless that lock step leaves
  // one CTA idle for a large share of the work: with three pairs the CTA
  // without a pair in the second round idles for half of it (measured with
  // two MMA-issuing threads: two pairs 430 -> 393 us on the Qwen3-8B B8
  // workload, four and more pairs 10 % faster).  The ranges must pair up, and
  // the W multicast reads this GPU's own memory only: a weight elsewhere
  // (host or another device) runs unclustered.
  const int pairs = (p.T + kWideG * kM - 1) / (kWideG * kM);
  return (p.g_lm % 2 == 0 && !p.t_dev && (pairs == 2 || pairs >= 4) && p.w_local) ? 3 : 2;
}

cudaError_t launch_lmhead_bf16(const LmParams& p, const LmMaps& maps, cudaStream_t s) {
  if (p.a_rows < 8 || p.a_rows > kM || p.a_rows % 8) return cudaErrorInvalidValue;
  const int variant = lmhead_bf16_variant(p);
  if (variant != 1) {
    if (p.a_rows != kM) return cudaErrorInvalidValue;
    return variant == 3 ? launch_wide<2>(p, maps, s) : launch_wide<1>(p, maps, s);
  }
  const size_t smem = lmhead_tc_smem_bytes(p.a_rows);
  cudaError_t err = set_smem_attrs(lmhead_tc_kernel, smem);
  if (err != cudaSuccess) return err;
  return launch_pdl(lmhead_tc_kernel, dim3(p.g_lm), dim3(192), smem, s, maps, p);
}

}  // namespace asd
