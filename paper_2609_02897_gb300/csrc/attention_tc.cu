// Tree attention (Sec. 2 "Verify": the target scores every drafted node in
// one forward pass) on the 5th-generation tensor cores, for steps where the
// attention kernel has the SMs to itself (more than 128 tree nodes: the LM
// head then takes most of an SM's shared memory and runs first).  bf16 in,
// fp32 accumulate.
//
// Work item (one CTA): 128 query rows of one (sequence, KV head) pair, the
// whole context; the CTAs take the sequences in decreasing order of work, so
// the longest items start first.  The rows of a pair are its N nodes times
// the G query heads that share the KV head, node-major (row r -> node r / G,
// head g*G + r % G); row r lives in TMEM lane r.  Keys come in tiles of 128,
// K and V through TMA rings of their own (128-byte swizzle; paged caches one
// box per page; the tree K/V through a 3D map over [T, Hkv, D]), so a K slot
// is refilled as soon as its S MMA is done rather than after the tile's P.V;
// the last tile of a pair holds its tree keys, where a node sees only its
// ancestors (bitmasks derived here from the parent array).
//
//   Q             loaded once into shared memory by one TMA (G dividing 128:
//                 boxes of G heads x 128/G nodes), else by the softmax warps
//   S = Q . K^T   tcgen05.mma, Q and K K-major in shared memory
//   P = exp2(S*c - m), per row by the thread that owns the row, written back
//                 over the tile's S columns as bf16 pairs
//   O += P . V    tcgen05.mma, A (= P) from TMEM, V MN-major straight from its
//                 TMA tile, O in TMEM for the whole item
//
// The softmax keeps a per-row reference max m and rescales O only when the
// running max exceeds m by more than 2^8 in the exp2 domain (P then stays
// below 2^8 and the result equals that with the exact running max).  S/P is triple-buffered: S of tile
// t+1 is ready when the softmax finishes tile t, and S of tile t+2 does not
// wait for O += P V of tile t (with two buffers it did, which put the P.V,
// its commit and the next S on the softmax's path every second tile).
//
// TMEM (512 columns): O [0, D), S/P [128, 256), [256, 384), [384, 512).
// Shared memory: Q, a 3-stage K ring and a V ring (160 KB of rings for D =
// 128).
// Warp roles (384 threads): warp 0 K producer, warp 1 TMEM allocator and
// issuer of the S MMAs, warps 2-9 softmax and epilogue, two per TMEM lane
// quarter, each on one half of every tile's keys, warp 10 issuer of the P.V
// MMAs, warp 11 V producer.
#include "kernels.h"
#include "tc.cuh"

namespace asd {
namespace {

constexpr int kRows = kAttnTcRows;   // query rows per CTA = TMEM lanes
constexpr int kKeys = kAttnTcKeys;   // keys per tile
constexpr int kThreads = 384;   // twelve warps (the roles above; the ping-pong form's below)
constexpr int kSoftmaxThreads = 256;   // eight warps: two per TMEM lane quarter
constexpr float kRescaleLog2 = 8.f;
constexpr uint32_t kTmemCols = 512;
constexpr int kSBufs = 3;              // S/P buffers in TMEM
constexpr uint32_t kSCol0 = 128;       // S/P buffer b at columns [128 (b + 1), 128 (b + 2))

// Dynamic shared memory, 1024-byte aligned: Q [D/64][128 rows][128 B], the K
// ring [stage][D/64][128 keys][128 B], then the V ring likewise (two stages
// for D = 128, where a third does not fit beside Q).
template <int D>
struct TcGeom {
  static constexpr int kNH = D / 64;
  static constexpr int kTileBytes = kNH * kKeys * 128;   // one K or one V tile
  static constexpr int kKStages = 3;
  static constexpr int kVStages = D == 64 ? 3 : 2;
  static constexpr int kQOff = 0;
  static constexpr int kKOff = kNH * kRows * 128;
  static constexpr int kVOff = kKOff + kKStages * kTileBytes;
  static constexpr int kBytes = kVOff + kVStages * kTileBytes;
};

// Named barrier 1 of the eight softmax warps.
__device__ __forceinline__ void softmax_sync() {
  asm volatile("bar.sync 1, %0;" ::"n"(kSoftmaxThreads) : "memory");
}

// AND of `v` over the eight softmax warps (named barrier 1); uniform result.
__device__ __forceinline__ bool softmax_all(bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 q, %1, 0;\n\t"
      "barrier.cta.red.and.pred p, 1, %2, q;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(r)
      : "r"(v ? 1u : 0u), "n"(kSoftmaxThreads)
      : "memory");
  return r != 0;
}

// OR of `v` over the eight softmax warps (named barrier 1); uniform result.
__device__ __forceinline__ bool softmax_any(bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 q, %1, 0;\n\t"
      "barrier.cta.red.or.pred p, 1, %2, q;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(r)
      : "r"(v ? 1u : 0u), "n"(kSoftmaxThreads)
      : "memory");
  return r != 0;
}

// Every lane polls (bounded by `budget` cycles); the result is lane 0's,
// uniform over the warp.
__device__ __forceinline__ bool wait_all(uint64_t* bar, uint32_t parity, long long budget) {
  return __shfl_sync(0xffffffffu, mbar_wait(smem_u32(bar), parity, budget) ? 1 : 0, 0) != 0;
}

__device__ __forceinline__ bool aborted_warp(volatile int* s_abort) {
  return __shfl_sync(0xffffffffu, *s_abort, 0) != 0;
}

struct Item {
  int b, g, s0, n, r0, nrows, R;
  int ctx, nctx, ntree, ntiles;
};

constexpr int kOrderMax = 256;   // batches ordered by work in-kernel (larger ones: index order)

// The sequence of rank r when the B sequences are ordered by decreasing
// attention work (their context and tree key tiles, ties by index): the
// hardware dispatches CTAs in blockIdx order, so the longest items start
// first and the short ones fill the last wave.  Every thread of the CTA calls
// it (it synchronises the CTA); s_work holds kOrderMax ints.
__device__ __forceinline__ int sequence_of_rank(const AttnParams& p, int r, int* s_work,
                                                int* s_b) {
  if (p.B > kOrderMax) return r;
  if (threadIdx.x == 0) *s_b = r;
  for (int q = threadIdx.x; q < p.B; q += blockDim.x) {
    const int c = min(max(p.ctx_len[q], 0), p.ctx_max);
    const int n = min(max(p.cu_nodes[q + 1] - p.cu_nodes[q], 0), kMaxNodes);
    s_work[q] = (c + kKeys - 1) / kKeys + (n + kKeys - 1) / kKeys;
  }
  __syncthreads();
  for (int q = threadIdx.x; q < p.B; q += blockDim.x) {
    const int w = s_work[q];
    int rank = 0;
    for (int j = 0; j < p.B; ++j) {
      const int v = s_work[j];
      rank += (v > w || (v == w && j < q)) ? 1 : 0;
    }
    if (rank == r) *s_b = q;
  }
  __syncthreads();
  return *s_b;
}

// blockIdx.y = (r, g): KV head g of the sequence of rank r (sequence_of_rank);
// blockIdx.x: the item's block of query rows.
__device__ __forceinline__ bool make_item(const AttnParams& p, Item& it, int* s_work, int* s_b) {
  const int rb = blockIdx.x, bg = blockIdx.y;
  const int r = bg / p.Hkv;
  it.b = sequence_of_rank(p, r, s_work, s_b);
  it.g = bg - r * p.Hkv;
  it.s0 = p.cu_nodes[it.b];
  it.n = p.cu_nodes[it.b + 1] - it.s0;
  it.R = it.n * p.G;
  it.r0 = rb * kRows;
  // sequence extents and context lengths are caller inputs (the tree
  // preparation reports bad ones); every access below stays in bounds anyway
  if (it.n <= 0 || it.n > kMaxNodes || it.s0 < 0 || it.s0 + it.n > p.T || it.r0 >= it.R)
    return false;
  it.nrows = min(kRows, it.R - it.r0);
  it.ctx = min(max(p.ctx_len[it.b], 0), p.ctx_max);
  it.nctx = (it.ctx + kKeys - 1) / kKeys;
  it.ntree = (it.n + kKeys - 1) / kKeys;
  it.ntiles = it.nctx + it.ntree;
  return true;
}

__device__ __forceinline__ size_t grow_of(const AttnParams& p, const Item& it, int r) {
  const int rr = it.r0 + r;
  const int i = rr / p.G;
  return static_cast<size_t>(it.s0 + i) * p.Hq + it.g * p.G + (rr - i * p.G);
}

constexpr int kPageChunk = 512;   // page-table entries staged in shared memory

// Issues one K (which = 0) or V (which = 1) tile t into `dst` (producer lane 0;
// contiguous cache or tree keys).
template <int D>
__device__ __forceinline__ void issue_half_tile(const AttnParams& p, const Item& it, int t,
                                                uint32_t dst, uint32_t bar,
                                                const CUtensorMap* tm, const CUtensorMap* tm_tree,
                                                uint64_t pol) {
  using G = TcGeom<D>;
  mbar_expect_tx(bar, G::kTileBytes);
  if (t >= it.nctx) {
    const int key0 = (t - it.nctx) * kKeys;
#pragma unroll
    for (int h = 0; h < G::kNH; ++h)
      tma_load_3d(dst + h * (kKeys * 128), tm_tree, bar, h * 64, it.g, it.s0 + key0, pol);
    return;
  }
  const int row = (it.b * p.Hkv + it.g) * p.ctx_max + t * kKeys;
#pragma unroll
  for (int h = 0; h < G::kNH; ++h) tma_load_2d(dst + h * (kKeys * 128), tm, bar, h * 64, row, pol);
}

// Paged context tile t, K or V (the whole producer warp): one box of
// min(page, 128) rows per page the tile touches, lane j taking page j of the
// tile, its page id read from a chunk of the sequence's page-table row that
// the warp stages in shared memory (`chunk0`: first staged entry, -1 before
// the first chunk).  Pages past the context are not loaded; an out-of-range
// page id is reported and not loaded.
template <int D>
__device__ __forceinline__ void issue_paged_half(const AttnParams& p, const Item& it, int t,
                                                 uint32_t dst, uint32_t bar, const CUtensorMap* tm,
                                                 uint64_t pol, int* s_pages, int& chunk0,
                                                 int lane) {
  using G = TcGeom<D>;
  const int ps = p.page_size;
  const int br = ps < kKeys ? ps : kKeys;
  const int nbox = kKeys / br;
  const int key0 = t * kKeys;
  const int e_first = key0 / ps, e_last = (key0 + (nbox - 1) * br) / ps;
  if (chunk0 < 0 || e_first < chunk0 || e_last >= chunk0 + kPageChunk) {
    chunk0 = e_first;
    const int32_t* row_pt = p.page_table + static_cast<size_t>(it.b) * p.pages_per_seq;
    for (int i = lane; i < kPageChunk; i += 32) {
      const int e = chunk0 + i;
      s_pages[i] = e < p.pages_per_seq ? row_pt[e] : -1;
    }
    __syncwarp();
  }
  int row = -1;
  if (lane < nbox) {
    const int key = key0 + lane * br;
    if (key < it.ctx) {
      const int page = s_pages[key / ps - chunk0];
      if (page < 0 || page >= p.num_pages)
        set_status(p.status, ASD_ERR_CTX_RANGE);
      else
        row = (page * p.Hkv + it.g) * ps + (key % ps);
    }
  }
  const uint32_t valid = __ballot_sync(0xffffffffu, row >= 0);
  if (lane == 0) mbar_expect_tx(bar, static_cast<uint32_t>(__popc(valid) * G::kNH * br * 128));
  __syncwarp();
  if (row >= 0) {
#pragma unroll
    for (int h = 0; h < G::kNH; ++h)
      tma_load_2d(dst + h * (kKeys * 128) + lane * br * 128, tm, bar, h * 64, row, pol);
  }
  __syncwarp();
}

// The query tile of an item by TMA (p.q_tma): a 3D map over q [T, Hq, D]
// with boxes of 64 columns x G heads x 128/G nodes lands as the item's 128
// rows (node-major, head-minor, as grow_of numbers them), 128-byte swizzled;
// rows past the item's hold the next nodes' queries (or zeros past T), which
// no output row reads.
template <int D>
__device__ __forceinline__ void issue_q_tile(const AttnParams& p, const Item& it, uint32_t q_s,
                                             uint32_t bar, const CUtensorMap* tm_q,
                                             uint64_t pol) {
  using G = TcGeom<D>;
  mbar_expect_tx(bar, static_cast<uint32_t>(G::kNH * kRows * 128));
#pragma unroll
  for (int h = 0; h < G::kNH; ++h)
    tma_load_3d(q_s + h * (kRows * 128), tm_q, bar, h * 64, it.g * p.G, it.s0 + it.r0 / p.G,
                pol);
}

// Softmax warps (eight): warp w handles TMEM lane quarter w % 4 (its 32 query
// rows, one thread per row) and half h = (w - 2) / 4 of every tile's 128 keys.
// Per tile: read its 64 S columns, mask, exchange the row's partial max with
// the warp that holds the other half, keep the reference max, and write P
// (bf16 pairs) over the tile's S columns: half h's keys go to P columns
// [32h, 32h + 32), which overlap S columns that both halves have read before
// the exchange.  The row sum stays split between the two threads of a row
// until the end.  Returns false (uniformly over the eight warps) when a
// bounded wait gave up; otherwise inv = 1 / (row sum), with O complete in
// TMEM.
template <int D>
__device__ __forceinline__ bool softmax_role(const AttnParams& p, const Item& it, uint32_t tmem,
                                             uint8_t* gbase, const uint64_t (*s_anc)[2],
                                             float (*s_mx)[2][kRows], float (*s_l)[kRows],
                                             uint64_t* q_ready, uint64_t* s_full,
                                             uint64_t* p_full, uint64_t* pv_done,
                                             uint64_t* v_full, volatile int* s_abort,
                                             long long budget, float& inv) {
  using G = TcGeom<D>;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int hf = (warp - 2) >> 2;              // key half of every tile
  const int row = (warp & 3) * 32 + lane;      // = TMEM lane
  const int tid = threadIdx.x - 64;            // 0..255
  const uint32_t lane_base = tmem + (static_cast<uint32_t>((warp & 3) * 32) << 16);

  // this half of the row's query (16-byte chunks [hf D/16, (hf+1) D/16)) ->
  // shared memory, 128-byte swizzled like a TMA tile; zeros past nrows
  // (unless the query tile comes by TMA)
  if (!p.q_tma) {
    const bool mine = row < it.nrows;
    const uint4* qg = reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(p.q) +
                                                     (mine ? grow_of(p, it, row) : 0) * D);
    uint8_t* qs = gbase + G::kQOff;
#pragma unroll
    for (int k = 0; k < D / 16; ++k) {
      const int c = hf * (D / 16) + k;
      const uint4 v = mine ? qg[c] : make_uint4(0u, 0u, 0u, 0u);
      *reinterpret_cast<uint4*>(qs + (c >> 3) * (kRows * 128) + row * 128 +
                                (((c & 7) ^ (row & 7)) << 4)) = v;
    }
  }
  if (!p.q_tma) {
    fence_proxy_async();   // the tensor cores read these rows
    __syncwarp();
    if (lane == 0) mbar_arrive(smem_u32(q_ready));
  }

  uint64_t alo = 0, ahi = 0;
  if (row < it.nrows) {
    const int node = (it.r0 + row) / p.G;
    alo = s_anc[node][0];
    ahi = s_anc[node][1];
  }
  const float c = p.scale_log2;
  float m_ref = -INFINITY, l = 0.f;
  bool ok = true, bad = false;
  bool s_seen = false;   // S of tile t already seen complete (probed during tile t-1)
  for (int t = 0; t < it.ntiles; ++t) {
    const int b = t % kSBufs, e = t & 1;
    const uint32_t sb = lane_base + kSCol0 + b * kKeys;
    const bool tree = t >= it.nctx;
    const int key0 = tree ? (t - it.nctx) * kKeys : t * kKeys;
    const int valid = min(kKeys, (tree ? it.n : it.ctx) - key0);
    float x[64];
    float mt = -INFINITY;
    const bool here = !bad && (s_seen || wait_all(&s_full[b], (t / kSBufs) & 1, budget)) &&
                      !aborted_warp(s_abort);
    if (here) {
      tc_fence_after();
      tmem_ld64(sb + 64 * hf, x);
      if (tree || valid < kKeys) {
        // the tree tile holds every node of the sequence (at most 128) from
        // key 0: key k of this half is bit k of the half's ancestor word
        const uint64_t am = tree ? (hf ? ahi : alo) : ~0ull;
#pragma unroll
        for (int k = 0; k < 64; ++k) {
          const bool v = (64 * hf + k < valid) && ((am >> k) & 1ull);
          x[k] = v ? x[k] : -INFINITY;
        }
      }
#pragma unroll
      for (int k = 0; k < 64; ++k) mt = fmaxf(mt, x[k]);
      s_mx[e][hf][row] = mt;
    }
    // probe S of the next tile now (non-blocking), so that the barrier's
    // latency passes under this tile's exponentials; once complete, that
    // phase stays complete until this warp has consumed the tile
    s_seen = __all_sync(0xffffffffu,
                        t + 1 < it.ntiles &&
                            mbar_test_wait(smem_u32(&s_full[(t + 1) % kSBufs]),
                                           static_cast<uint32_t>(((t + 1) / kSBufs) & 1)));
    // every softmax warp decides together whether to go on (no warp may be
    // left waiting at a barrier), and the partial maxima become visible
    ok = softmax_all(here);
    if (!ok) break;
    // the row's max over both halves (raw scores; the scale is positive)
    mt = fmaxf(mt, s_mx[e][hf ^ 1][row]) * c;
    const float mn = fmaxf(m_ref, mt);
    const bool had = m_ref != -INFINITY;
    const bool need = had ? (mn > m_ref + kRescaleLog2) : (mn != -INFINITY);
    if (__any_sync(0xffffffffu, need && had)) {
      // O holds earlier tiles of this row: rescale this half of it once
      // O += P V of tile t-1 is done
      // (a wait that gives up marks the thread; all leave at the next tile)
      if (!wait_all(&pv_done[(t - 1) % kSBufs], ((t - 1) / kSBufs) & 1, budget)) {
        bad = true;
      } else {
        tc_fence_after();
        const float alpha = (need && had) ? exp2f(m_ref - mn) : 1.f;
#pragma unroll 1
        for (int cc = 0; cc < D / 64; ++cc) {
          float o[32];
          const uint32_t oc = lane_base + hf * (D / 2) + 32 * cc;
          tmem_ld32(oc, o);
#pragma unroll
          for (int i = 0; i < 32; ++i) o[i] *= alpha;
          tmem_st32(oc, o);
        }
      }
    }
    if (need) {
      l = had ? l * exp2f(m_ref - mn) : 0.f;
      m_ref = mn;
    }
    const float mu = (m_ref == -INFINITY) ? 0.f : m_ref;
    uint32_t pk[32];
#pragma unroll
    for (int k = 0; k < 64; k += 2) {
      const float p0 = ex2_approx(fmaf(x[k], c, -mu)), p1 = ex2_approx(fmaf(x[k + 1], c, -mu));
      l += p0 + p1;
      __nv_bfloat162 h = __floats2bfloat162_rn(p0, p1);
      pk[k / 2] = *reinterpret_cast<uint32_t*>(&h);
    }
    tmem_st32u(sb + 32 * hf, pk);
    if (valid < kKeys) {
      // ragged tile: V rows past the last valid key may hold anything; zero
      // them so that 0 * V stays 0, once the V tile has landed (it comes
      // through its own ring and may still be in flight)
      if (!bad && wait_all(&v_full[t % G::kVStages], (t / G::kVStages) & 1, budget)) {
        uint8_t* vt = gbase + G::kVOff + (t % G::kVStages) * G::kTileBytes;
        constexpr int kChunksPerRow = G::kNH * 8;
        for (int i = tid; i < (kKeys - valid) * kChunksPerRow; i += kSoftmaxThreads) {
          const int r = valid + i / kChunksPerRow, rem = i % kChunksPerRow;
          *reinterpret_cast<uint4*>(vt + (rem >> 3) * (kKeys * 128) + r * 128 + (rem & 7) * 16) =
              make_uint4(0u, 0u, 0u, 0u);
        }
        fence_proxy_async();  // the zeroed rows are read by the tensor cores
      } else {
        bad = true;
      }
    }
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive(smem_u32(&p_full[b]));
  }
  if (ok) {
    // O is complete once the last P.V is done (S of the last tile waited for
    // the P.V three tiles back, so that buffer's pending phase is the last's)
    const int last = it.ntiles - 1;
    ok = !bad && wait_all(&pv_done[last % kSBufs], (last / kSBufs) & 1, budget) &&
         !aborted_warp(s_abort);
    if (ok) tc_fence_after();
  }
  if (softmax_any(!ok)) {
    if (tid == 0) {
      note_timeout(p.status);
      *s_abort = 1;
    }
    return false;
  }
  // the row sum over both halves
  s_l[hf][row] = l;
  softmax_sync();
  l += s_l[hf ^ 1][row];
  inv = l > 0.f ? 1.f / l : 0.f;
  return true;
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v,
                   const __grid_constant__ CUtensorMap tm_tk,
                   const __grid_constant__ CUtensorMap tm_tv,
                   const __grid_constant__ CUtensorMap tm_q, const AttnParams p) {
  using G = TcGeom<D>;
  extern __shared__ uint8_t smem_raw[];
  constexpr int KS = G::kKStages, VS = G::kVStages;
  __shared__ __align__(8) uint64_t s_k_full[KS], s_k_empty[KS];
  __shared__ __align__(8) uint64_t s_v_full[VS], s_v_empty[VS];
  __shared__ __align__(8) uint64_t s_s_full[kSBufs];    // S of a tile in TMEM (MMA -> softmax)
  __shared__ __align__(8) uint64_t s_p_full[kSBufs];    // P of a tile in TMEM (softmax -> MMA)
  __shared__ __align__(8) uint64_t s_pv_done[kSBufs];   // O += P V of a tile done (MMA -> softmax)
  __shared__ __align__(8) uint64_t s_q_ready;
  __shared__ __align__(8) uint64_t s_mma_done[2];   // each MMA issuer's own drain
  __shared__ uint32_t s_tmem;
  __shared__ volatile int s_abort;
  __shared__ int s_par[kMaxNodes];
  __shared__ uint64_t s_anc[kMaxNodes][2];
  __shared__ float s_mx[2][2][kRows];   // [tile parity][key half][row]: partial row max
  __shared__ float s_l[2][kRows];       // [key half][row]: partial row sum
  __shared__ int s_pages[2][kPageChunk];   // K / V producer: staged page-table entries
  __shared__ int s_issued[2][KS > VS ? KS : VS];  // producer: K (0) / V (1) fills per stage

  pdl_launch_dependents();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long budget = wait_budget(p.status);
  __shared__ int s_work[kOrderMax];
  __shared__ int s_seq;
  Item it;
  if (!make_item(p, it, s_work, &s_seq)) {  // no query rows here (uniform over the CTA)
    pdl_wait();
    return;
  }

  uint32_t base = smem_u32(smem_raw);
  const uint32_t pad = (1024u - (base & 1023u)) & 1023u;
  uint8_t* gbase = smem_raw + pad;
  base += pad;
  const uint32_t q_s = base + G::kQOff, k_s0 = base + G::kKOff, v_s0 = base + G::kVOff;

  if (threadIdx.x == 0) {
    for (int s = 0; s < KS; ++s) {
      mbar_init(smem_u32(&s_k_full[s]), 1);
      mbar_init(smem_u32(&s_k_empty[s]), 1);
      s_issued[0][s] = 0;
    }
    for (int s = 0; s < VS; ++s) {
      mbar_init(smem_u32(&s_v_full[s]), 1);
      mbar_init(smem_u32(&s_v_empty[s]), 1);
      s_issued[1][s] = 0;
    }
    for (int b = 0; b < kSBufs; ++b) {
      mbar_init(smem_u32(&s_s_full[b]), 1);
      mbar_init(smem_u32(&s_p_full[b]), kSoftmaxThreads / 32);
      mbar_init(smem_u32(&s_pv_done[b]), 1);
    }
    // the query: one TMA (p.q_tma) or the eight softmax warps' stores
    mbar_init(smem_u32(&s_q_ready), p.q_tma ? 1 : kSoftmaxThreads / 32);
    mbar_init(smem_u32(&s_mma_done[0]), 1);
    mbar_init(smem_u32(&s_mma_done[1]), 1);
    s_abort = 0;
    fence_mbar_init();
    // The item's first copies go out before the rest of the set-up: its
    // query tile (TMA form), then the first fill of both rings on a
    // contiguous cache (the producers go on from there).  What the first S
    // MMA waits for then lands while the CTA allocates TMEM and builds the
    // ancestor masks.
    const uint64_t pol = l2_policy_evict_first();
    if (p.q_tma) issue_q_tile<D>(p, it, q_s, smem_u32(&s_q_ready), &tm_q, pol);
    if (p.page_size == 0) {
      for (int t = 0; t < KS && t < it.ntiles; ++t) {
        issue_half_tile<D>(p, it, t, k_s0 + t * G::kTileBytes, smem_u32(&s_k_full[t]), &tm_k,
                           &tm_tk, pol);
        s_issued[0][t] = 1;
        if (t < VS) {
          issue_half_tile<D>(p, it, t, v_s0 + t * G::kTileBytes, smem_u32(&s_v_full[t]), &tm_v,
                             &tm_tv, pol);
          s_issued[1][t] = 1;
        }
      }
    }
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&s_tmem), kTmemCols);
    tmem_relinquish();
  }
  // ancestor bitmasks (self included) of the sequence's nodes for the tree
  // tile; a malformed parent ends the walk, so it is bounded
  for (int i = threadIdx.x; i < it.n; i += kThreads) s_par[i] = p.parent[it.s0 + i];
  __syncthreads();
  for (int i = threadIdx.x; i < it.n; i += kThreads) {
    uint64_t lo = 0, hi = 0;
    int u = i;
    while (true) {
      if (u < 64) lo |= 1ull << u; else hi |= 1ull << (u - 64);
      const int pu = s_par[u];
      if (pu < 0 || pu >= u) break;
      u = pu;
    }
    s_anc[i][0] = lo;
    s_anc[i][1] = hi;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;

  bool ok = false;           // softmax warps: O complete in TMEM
  float inv = 0.f;
  if (warp == 0 || warp == 11) {
    // ----------------------------------------------------------- TMA producers
    // K and V come through rings of their own, each filled by its own warp
    // (warp 0 K, warp 11 V), so that neither ring waits behind the other: a K
    // slot is free again once the S MMA of its tile is done, a V slot once the
    // P.V MMA is.
    const int which = warp == 0 ? 0 : 1;
    const int ns = which ? VS : KS;
    if (lane == 0) {
      prefetch_tmap(which ? &tm_v : &tm_k);
      prefetch_tmap(which ? &tm_tv : &tm_tk);
    }
    const uint64_t pol = l2_policy_evict_first();
    int chunk0 = -1;
    bool pok = true;
    // on a contiguous cache the first fill of the ring went out with the set-up
    for (int t = p.page_size == 0 ? ns : 0; pok && t < it.ntiles; ++t) {
      const int stage = t % ns;
      uint64_t* empty = which ? &s_v_empty[stage] : &s_k_empty[stage];
      uint64_t* full = which ? &s_v_full[stage] : &s_k_full[stage];
      if (!wait_all(empty, ((t / ns) & 1) ^ 1u, budget) || aborted_warp(&s_abort)) {
        pok = false;
        break;
      }
      const uint32_t dst = base + (which ? G::kVOff : G::kKOff) + stage * G::kTileBytes;
      if (p.page_size != 0 && t < it.nctx)
        issue_paged_half<D>(p, it, t, dst, smem_u32(full), which ? &tm_v : &tm_k, pol,
                            s_pages[which], chunk0, lane);
      else if (lane == 0)
        issue_half_tile<D>(p, it, t, dst, smem_u32(full), which ? &tm_v : &tm_k,
                           which ? &tm_tv : &tm_tk, pol);
      if (lane == 0) ++s_issued[which][stage];
      __syncwarp();
    }
    if (!pok && lane == 0) {
      note_timeout(p.status);
      s_abort = 1;
    }
    // every copy issued has landed before the buffers are reused or left
    // (the query tile's too, which a wait that gave up may have left in flight)
    if (lane == 0) {
      for (int st = 0; st < ns; ++st)
        if (s_issued[which][st] > 0)
          mbar_wait(smem_u32(which ? &s_v_full[st] : &s_k_full[st]),
                    static_cast<uint32_t>((s_issued[which][st] - 1) & 1));
      if (which == 0 && p.q_tma) mbar_wait(smem_u32(&s_q_ready), 0);
    }
    __syncwarp();
  } else if (warp == 1 || warp == 10) {
    // ------------------------------------------------------------ MMA issuers
    // Two issuing threads, so that the one's barrier waits (each a few hundred
    // cycles even on a completed phase) overlap the other's MMAs: warp 1
    // issues S = Q K^T of every tile, warp 10 O += P V.  Each commit tracks the
    // issuing thread's own MMAs.
    if (lane == 0) {
      bool mok = true;
      if (warp == 1) {
        const uint32_t idesc_s = idesc_bf16(kRows, kKeys);   // S = Q K^T
        mok = mbar_wait(smem_u32(&s_q_ready), 0, budget);
        if (mok) tc_fence_after();
        for (int t = 0; mok && t < it.ntiles; ++t) {
          const int stage = t % KS, b = t % kSBufs;
          mok = mbar_wait(smem_u32(&s_k_full[stage]), (t / KS) & 1, budget);
          // the S/P buffer is free once O += P V of tile t-3 is done
          if (mok && t >= kSBufs)
            mok = mbar_wait(smem_u32(&s_pv_done[b]), ((t / kSBufs) - 1) & 1, budget);
          if (!mok || s_abort) break;
          tc_fence_after();
          const uint32_t kst = k_s0 + stage * G::kTileBytes;
#pragma unroll
          for (int ks = 0; ks < D / 16; ++ks) {
            const int h = ks >> 2, kk = ks & 3;
            tc_mma(tmem + kSCol0 + b * kKeys, sw128_desc(q_s + h * (kRows * 128) + 32 * kk),
                   sw128_desc(kst + h * (kKeys * 128) + 32 * kk), idesc_s, ks > 0 ? 1u : 0u);
          }
          tc_commit(smem_u32(&s_s_full[b]));
          tc_commit(smem_u32(&s_k_empty[stage]));
        }
      } else {
        const uint32_t idesc_o = idesc_bf16(kRows, D, true);   // O += P V, V MN-major
        for (int j = 0; mok && j < it.ntiles; ++j) {
          // O += P_j V_j once tile j's softmax has written P_j
          const int stage = j % VS, b = j % kSBufs;
          mok = mbar_wait(smem_u32(&s_p_full[b]), (j / kSBufs) & 1, budget) &&
                mbar_wait(smem_u32(&s_v_full[stage]), (j / VS) & 1, budget);
          if (!mok || s_abort) break;
          tc_fence_after();
          const uint32_t vst = v_s0 + stage * G::kTileBytes;
#pragma unroll
          for (int kk = 0; kk < kKeys / 16; ++kk)
            tc_mma_ts(tmem, tmem + kSCol0 + b * kKeys + kk * 8,
                      sw128_desc_mn(vst + kk * 2048, kKeys * 128, 1024), idesc_o,
                      (j > 0 || kk > 0) ? 1u : 0u);
          tc_commit(smem_u32(&s_pv_done[b]));
          tc_commit(smem_u32(&s_v_empty[stage]));
        }
      }
      if (!mok) {
        note_timeout(p.status);
        s_abort = 1;
      }
      // every MMA this thread issued has finished before TMEM or the buffers
      // are reused
      uint64_t* done = &s_mma_done[warp == 1 ? 0 : 1];
      tc_commit(smem_u32(done));
      mbar_wait(smem_u32(done), 0);
    }
    __syncwarp();
  } else {
    ok = softmax_role<D>(p, it, tmem, gbase, s_anc, s_mx, s_l, &s_q_ready, s_s_full, s_p_full,
                         s_pv_done, s_v_full, &s_abort, budget, inv);
  }

  // ------------------------------------------------------------------ finish
  tc_fence_before();
  __syncthreads();   // the tile buffers and the tensor cores are idle from here on
  tc_fence_after();
  if (warp >= 2 && warp < 10 && ok) {
    // each thread writes its key half's share of the row: D/2 output columns
    const int hf = (warp - 2) >> 2;
    const int row = (warp & 3) * 32 + lane;   // TMEM lane = query row
    const uint32_t lane_base = tmem + (static_cast<uint32_t>((warp & 3) * 32) << 16) +
                               static_cast<uint32_t>(hf * (D / 2));
    const bool mine = row < it.nrows;
    __nv_bfloat16* out = static_cast<__nv_bfloat16*>(p.out) +
                         (mine ? grow_of(p, it, row) : 0) * D + hf * (D / 2);
#pragma unroll 1
    for (int c = 0; c < D / 64; ++c) {
      float o[32];
      tmem_ld32(lane_base + 32 * c, o);   // every lane takes part in the warp-wide load
      if (mine) {
#pragma unroll
        for (int k = 0; k < 32; k += 8) {
          uint4 pk;
          __nv_bfloat162 h0 = __floats2bfloat162_rn(o[k] * inv, o[k + 1] * inv);
          __nv_bfloat162 h1 = __floats2bfloat162_rn(o[k + 2] * inv, o[k + 3] * inv);
          __nv_bfloat162 h2 = __floats2bfloat162_rn(o[k + 4] * inv, o[k + 5] * inv);
          __nv_bfloat162 h3 = __floats2bfloat162_rn(o[k + 6] * inv, o[k + 7] * inv);
          pk.x = *reinterpret_cast<uint32_t*>(&h0);
          pk.y = *reinterpret_cast<uint32_t*>(&h1);
          pk.z = *reinterpret_cast<uint32_t*>(&h2);
          pk.w = *reinterpret_cast<uint32_t*>(&h3);
          *reinterpret_cast<uint4*>(out + 32 * c + k) = pk;
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, kTmemCols);
  pdl_wait();   // the next kernel's wait covers every earlier kernel
}

// ----------------------------------------------------------------------------
// Ping-pong variant: one CTA per (256 query rows, sequence x KV head) = two
// 128-row query tiles A and B that see the same keys.  Every K/V tile serves
// both: S_A = Q_A.K^T and S_B = Q_B.K^T, then O_A += P_A.V and O_B += P_B.V, so
// the MMAs of one tile run while the other tile's softmax works, and a K/V
// byte feeds twice the products.  Q stays in shared memory (both tiles, 128-byte
// swizzled, by TMA or written by the softmax threads); TMEM holds O_A [0, D),
// O_B [D, 2D) and S/P_A [256, 384), S/P_B [384, 512).  K and V come through
// separate rings with their own barriers, so a K slot is refilled as soon as
// both S MMAs have read it.  Warps: 0 K producer, 1 S-MMA issuer (lane 0),
// 2-5 softmax of tile A, 6-9 softmax of tile B, 10 P.V-MMA issuer (lane 0),
// 11 V producer; a softmax thread owns one row
// of its tile and all 128 keys of every key tile, so no exchange between warps
// is needed: per key tile it reads S twice (the row max, then the
// exponentials) and writes P as bf16 pairs over the S columns already read.
constexpr int kPPRows = 2 * kRows;   // query rows per CTA

template <int D>
struct PPGeom {
  static constexpr int kNH = D / 64;
  static constexpr int kStages = D == 64 ? 3 : 2;
  static constexpr int kQTile = kNH * kRows * 128;    // one query tile
  static constexpr int kKVTile = kNH * kKeys * 128;   // one K or one V tile
  static constexpr int kQOff = 0;
  static constexpr int kKOff = 2 * kQTile;
  static constexpr int kVOff = kKOff + kStages * kKVTile;
  static constexpr int kBytes = kVOff + kStages * kKVTile;
};

__device__ __forceinline__ bool make_item_pp(const AttnParams& p, Item& it, int* s_work,
                                             int* s_b) {
  const int rb = blockIdx.x, bg = blockIdx.y;
  const int r = bg / p.Hkv;
  it.b = sequence_of_rank(p, r, s_work, s_b);
  it.g = bg - r * p.Hkv;
  it.s0 = p.cu_nodes[it.b];
  it.n = p.cu_nodes[it.b + 1] - it.s0;
  it.R = it.n * p.G;
  it.r0 = rb * kPPRows;
  if (it.n <= 0 || it.n > kMaxNodes || it.s0 < 0 || it.s0 + it.n > p.T || it.r0 >= it.R)
    return false;
  it.nrows = min(kPPRows, it.R - it.r0);
  it.ctx = min(max(p.ctx_len[it.b], 0), p.ctx_max);
  it.nctx = (it.ctx + kKeys - 1) / kKeys;
  it.ntree = (it.n + kKeys - 1) / kKeys;
  it.ntiles = it.nctx + it.ntree;
  return true;
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    attn_pp_kernel(const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v,
                   const __grid_constant__ CUtensorMap tm_tk,
                   const __grid_constant__ CUtensorMap tm_tv,
                   const __grid_constant__ CUtensorMap tm_q, const AttnParams p) {
  using G = PPGeom<D>;
  constexpr int S = G::kStages;
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t s_k_full[S], s_k_empty[S], s_v_full[S], s_v_empty[S];
  __shared__ __align__(8) uint64_t s_s_full[2];    // S of tile X computed (MMA -> softmax X)
  __shared__ __align__(8) uint64_t s_p_full[2];    // P of tile X written (softmax X -> MMA)
  __shared__ __align__(8) uint64_t s_pv_done[2];   // O_X += P_X V done (MMA -> softmax X)
  __shared__ __align__(8) uint64_t s_q_ready;
  __shared__ __align__(8) uint64_t s_mma_done[2];   // each MMA issuer's own drain
  __shared__ uint32_t s_tmem;
  __shared__ volatile int s_abort;
  __shared__ int s_par[kMaxNodes];
  __shared__ uint64_t s_anc[kMaxNodes][2];
  __shared__ int s_pages[2][kPageChunk];   // K / V producer: staged page-table entries
  __shared__ int s_issued[2][S];   // producer: K (0) and V (1) fills issued per stage

  pdl_launch_dependents();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long budget = wait_budget(p.status);
  __shared__ int s_work[kOrderMax];
  __shared__ int s_seq;
  Item it;
  if (!make_item_pp(p, it, s_work, &s_seq)) {  // no query rows here (uniform over the CTA)
    pdl_wait();
    return;
  }
  const int nx = it.nrows > kRows ? 2 : 1;   // query tiles present

  uint32_t base = smem_u32(smem_raw);
  const uint32_t pad = (1024u - (base & 1023u)) & 1023u;
  uint8_t* gbase = smem_raw + pad;
  base += pad;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(smem_u32(&s_k_full[s]), 1);
      mbar_init(smem_u32(&s_k_empty[s]), 1);
      mbar_init(smem_u32(&s_v_full[s]), 1);
      mbar_init(smem_u32(&s_v_empty[s]), 1);
      s_issued[0][s] = s_issued[1][s] = 0;
    }
    for (int x = 0; x < 2; ++x) {
      mbar_init(smem_u32(&s_s_full[x]), 1);
      mbar_init(smem_u32(&s_p_full[x]), 4);
      mbar_init(smem_u32(&s_pv_done[x]), 1);
    }
    // the query tiles: one TMA per present tile (p.q_tma), issued before the
    // rest of the set-up, or the eight softmax warps' stores
    mbar_init(smem_u32(&s_q_ready), p.q_tma ? 1 : 8);
    mbar_init(smem_u32(&s_mma_done[0]), 1);
    mbar_init(smem_u32(&s_mma_done[1]), 1);
    s_abort = 0;
    fence_mbar_init();
    if (p.q_tma) {
      const uint64_t pol = l2_policy_evict_first();
      const uint32_t bar = smem_u32(&s_q_ready);
      mbar_expect_tx(bar, static_cast<uint32_t>(nx * G::kQTile));
      for (int x = 0; x < nx; ++x)
#pragma unroll
        for (int h = 0; h < G::kNH; ++h)
          tma_load_3d(base + G::kQOff + x * G::kQTile + h * (kRows * 128), &tm_q, bar, h * 64,
                      it.g * p.G, it.s0 + (it.r0 + x * kRows) / p.G, pol);
    }
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&s_tmem), kTmemCols);
    tmem_relinquish();
  }
  for (int i = threadIdx.x; i < it.n; i += kThreads) s_par[i] = p.parent[it.s0 + i];
  __syncthreads();
  for (int i = threadIdx.x; i < it.n; i += kThreads) {
    uint64_t lo = 0, hi = 0;
    int u = i;
    while (true) {
      if (u < 64) lo |= 1ull << u; else hi |= 1ull << (u - 64);
      const int pu = s_par[u];
      if (pu < 0 || pu >= u) break;
      u = pu;
    }
    s_anc[i][0] = lo;
    s_anc[i][1] = hi;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;

  if (warp == 0 || warp == 11) {
    // ----------------------------------------------------------- TMA producers
    // K (warp 0) and V (warp 11), each into its own ring; K slots free up as
    // soon as both S MMAs of their tile are done, V slots after both P.V MMAs
    const int which = warp == 0 ? 0 : 1;
    if (lane == 0) {
      prefetch_tmap(which ? &tm_v : &tm_k);
      prefetch_tmap(which ? &tm_tv : &tm_tk);
    }
    const uint64_t pol = l2_policy_evict_first();
    int chunk0 = -1;
    bool pok = true;
    for (int t = 0; t < it.ntiles; ++t) {
      const int stage = t % S;
      uint64_t* empty = which ? &s_v_empty[stage] : &s_k_empty[stage];
      uint64_t* full = which ? &s_v_full[stage] : &s_k_full[stage];
      if (!wait_all(empty, ((t / S) & 1) ^ 1u, budget) || aborted_warp(&s_abort)) {
        pok = false;
        break;
      }
      const uint32_t dst = base + (which ? G::kVOff : G::kKOff) + stage * G::kKVTile;
      if (p.page_size != 0 && t < it.nctx)
        issue_paged_half<D>(p, it, t, dst, smem_u32(full), which ? &tm_v : &tm_k, pol,
                            s_pages[which], chunk0, lane);
      else if (lane == 0)
        issue_half_tile<D>(p, it, t, dst, smem_u32(full), which ? &tm_v : &tm_k,
                           which ? &tm_tv : &tm_tk, pol);
      if (lane == 0) ++s_issued[which][stage];
      __syncwarp();
    }
    if (!pok && lane == 0) {
      note_timeout(p.status);
      s_abort = 1;
    }
    // every copy issued has landed before the buffers are reused or left
    // (the query tiles' too, which a wait that gave up may have left in flight)
    if (lane == 0) {
      for (int st = 0; st < S; ++st)
        if (s_issued[which][st] > 0)
          mbar_wait(smem_u32(which ? &s_v_full[st] : &s_k_full[st]),
                    static_cast<uint32_t>((s_issued[which][st] - 1) & 1));
      if (which == 0 && p.q_tma) mbar_wait(smem_u32(&s_q_ready), 0);
    }
    __syncwarp();
  } else if (warp == 1 || warp == 10) {
    // ------------------------------------------------------------ MMA issuers
    // Two issuing threads, so that the one's barrier waits overlap the other's
    // MMAs: warp 1 issues S_x(t) = Q_x K(t)^T, warp 10 O_x += P_x(t) V(t).
    // While tile A's softmax works on key tile t, the tensor cores run
    // O_B += P_B V(t-1) and S_B(t); while B's works, O_A += P_A V(t) and
    // S_A(t+1).  Each commit tracks the issuing thread's own MMAs.
    if (lane == 0) {
      bool mok = true;
      if (warp == 1) {
        const uint32_t idesc_s = idesc_bf16(kRows, kKeys);   // S = Q K^T
        mok = mbar_wait(smem_u32(&s_q_ready), 0, budget);
        if (mok) tc_fence_after();
        for (int t = 0; mok && t < it.ntiles; ++t) {
          const int stage = t % S;
          mok = mbar_wait(smem_u32(&s_k_full[stage]), (t / S) & 1, budget);
          for (int x = 0; mok && x < nx; ++x) {
            // tile x's S/P columns are free once O_x += P_x V of tile t-1 is done
            if (t > 0) mok = mbar_wait(smem_u32(&s_pv_done[x]), (t - 1) & 1, budget);
            if (!mok || s_abort) {
              mok = false;
              break;
            }
            tc_fence_after();
            const uint32_t kst = base + G::kKOff + stage * G::kKVTile;
            const uint32_t qst = base + G::kQOff + x * G::kQTile;
#pragma unroll
            for (int ks = 0; ks < D / 16; ++ks) {
              const int h = ks >> 2, kk = ks & 3;
              tc_mma(tmem + (256u + 128u * static_cast<uint32_t>(x)),
                     sw128_desc(qst + h * (kRows * 128) + 32 * kk),
                     sw128_desc(kst + h * (kKeys * 128) + 32 * kk), idesc_s, ks > 0 ? 1u : 0u);
            }
            tc_commit(smem_u32(&s_s_full[x]));
          }
          // the last S of tile t releases K(t)
          if (mok) tc_commit(smem_u32(&s_k_empty[stage]));
        }
      } else {
        const uint32_t idesc_o = idesc_bf16(kRows, D, true);   // O += P V, V MN-major
        for (int t = 0; mok && t < it.ntiles; ++t) {
          const int stage = t % S;
          mok = mbar_wait(smem_u32(&s_v_full[stage]), (t / S) & 1, budget);
          for (int x = 0; mok && x < nx; ++x) {
            // O_x += P_x(t) V(t) once tile x's softmax of key tile t is done
            mok = mbar_wait(smem_u32(&s_p_full[x]), t & 1, budget);
            if (!mok || s_abort) {
              mok = false;
              break;
            }
            tc_fence_after();
            const uint32_t vst = base + G::kVOff + stage * G::kKVTile;
#pragma unroll
            for (int kk = 0; kk < kKeys / 16; ++kk)
              tc_mma_ts(tmem + static_cast<uint32_t>(x * D),
                        tmem + (256u + 128u * static_cast<uint32_t>(x)) + kk * 8,
                        sw128_desc_mn(vst + kk * 2048, kKeys * 128, 1024), idesc_o,
                        (t > 0 || kk > 0) ? 1u : 0u);
            tc_commit(smem_u32(&s_pv_done[x]));
          }
          // the last P.V of tile t releases V(t)
          if (mok) tc_commit(smem_u32(&s_v_empty[stage]));
        }
      }
      if (!mok) {
        note_timeout(p.status);
        s_abort = 1;
      }
      // every MMA this thread issued has finished before TMEM or the buffers
      // are reused
      uint64_t* done = &s_mma_done[warp == 1 ? 0 : 1];
      tc_commit(smem_u32(done));
      mbar_wait(smem_u32(done), 0);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ softmax of tile x
    const int x = (warp - 2) >> 2;
    const int row = (warp & 3) * 32 + lane;    // = TMEM lane = row of the tile
    const int rr = x * kRows + row;            // row of the item
    const bool mine = rr < it.nrows;
    const uint32_t lane_base = tmem + (static_cast<uint32_t>((warp & 3) * 32) << 16);
    const uint32_t sb = lane_base + (256u + 128u * static_cast<uint32_t>(x));
    // the row's query -> shared memory, 128-byte swizzled like a TMA tile
    // (unless the query tiles come by TMA)
    if (!p.q_tma) {
      const int q_row = it.r0 + rr;
      const int node = q_row / p.G;
      const uint4* qg = reinterpret_cast<const uint4*>(
          static_cast<const __nv_bfloat16*>(p.q) +
          (mine ? (static_cast<size_t>(it.s0 + node) * p.Hq + it.g * p.G + (q_row - node * p.G)) : 0) *
              D);
      uint8_t* qs = gbase + G::kQOff + x * G::kQTile;
#pragma unroll
      for (int c = 0; c < D / 8; ++c) {
        const uint4 v = mine ? qg[c] : make_uint4(0u, 0u, 0u, 0u);
        *reinterpret_cast<uint4*>(qs + (c >> 3) * (kRows * 128) + row * 128 +
                                  (((c & 7) ^ (row & 7)) << 4)) = v;
      }
      fence_proxy_async();   // the tensor cores read these rows
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&s_q_ready));
    }
    uint64_t alo = 0, ahi = 0;
    if (mine) {
      const int node = (it.r0 + rr) / p.G;
      alo = s_anc[node][0];
      ahi = s_anc[node][1];
    }
    // a second query tile with no rows: its warps only staged the zero rows
    if (x < nx) {
    const float c = p.scale_log2;
    float m_ref = -INFINITY, l = 0.f;
    bool ok = true;
    for (int t = 0; t < it.ntiles; ++t) {
      const bool tree = t >= it.nctx;
      const int key0 = tree ? (t - it.nctx) * kKeys : t * kKeys;
      const int valid = min(kKeys, (tree ? it.n : it.ctx) - key0);
      ok = wait_all(&s_s_full[x], t & 1, budget) && !aborted_warp(&s_abort);
      if (!ok) break;
      tc_fence_after();
      // pass 1: the row's max over the tile's keys (raw scores); only a
      // ragged context tile and the tree tile need the key mask
      const bool masked = tree || valid < kKeys;
      float mt = -INFINITY;
#pragma unroll
      for (int hf = 0; hf < 2; ++hf) {
        float xs[64];
        tmem_ld64(sb + 64 * hf, xs);
        if (masked) {
          // the tree tile holds every node of the sequence (at most 128) from
          // key 0: key k of this half is bit k of the half's ancestor word
          const uint64_t am = tree ? (hf ? ahi : alo) : ~0ull;
#pragma unroll
          for (int k = 0; k < 64; ++k) {
            const bool v = (64 * hf + k < valid) && ((am >> k) & 1ull);
            xs[k] = v ? xs[k] : -INFINITY;
          }
        }
#pragma unroll
        for (int k = 0; k < 64; ++k) mt = fmaxf(mt, xs[k]);
      }
      mt *= c;
      const float mn = fmaxf(m_ref, mt);
      const bool had = m_ref != -INFINITY;
      const bool need = had ? (mn > m_ref + kRescaleLog2) : (mn != -INFINITY);
      if (__any_sync(0xffffffffu, need && had)) {
        // O holds earlier tiles of this row: rescale it once O += P V of tile
        // t-1 is done
        if (!wait_all(&s_pv_done[x], (t - 1) & 1, budget)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const float alpha = (need && had) ? exp2f(m_ref - mn) : 1.f;
#pragma unroll 1
        for (int cc = 0; cc < D / 32; ++cc) {
          float o[32];
          const uint32_t oc = lane_base + static_cast<uint32_t>(x * D) + 32 * cc;
          tmem_ld32(oc, o);
#pragma unroll
          for (int i = 0; i < 32; ++i) o[i] *= alpha;
          tmem_st32(oc, o);
        }
      }
      if (need) {
        l = had ? l * exp2f(m_ref - mn) : 0.f;
        m_ref = mn;
      }
      const float mu = (m_ref == -INFINITY) ? 0.f : m_ref;
      // pass 2: P = exp2(s c - m) as bf16 pairs over the S columns already read
#pragma unroll
      for (int hf = 0; hf < 2; ++hf) {
        float xs[64];
        tmem_ld64(sb + 64 * hf, xs);
        if (masked) {
          // the tree tile holds every node of the sequence (at most 128) from
          // key 0: key k of this half is bit k of the half's ancestor word
          const uint64_t am = tree ? (hf ? ahi : alo) : ~0ull;
#pragma unroll
          for (int k = 0; k < 64; ++k) {
            const bool v = (64 * hf + k < valid) && ((am >> k) & 1ull);
            xs[k] = v ? xs[k] : -INFINITY;
          }
        }
        uint32_t pk[32];
#pragma unroll
        for (int k = 0; k < 64; k += 2) {
          const float p0 = ex2_approx(fmaf(xs[k], c, -mu)), p1 = ex2_approx(fmaf(xs[k + 1], c, -mu));
          l += p0 + p1;
          __nv_bfloat162 h = __floats2bfloat162_rn(p0, p1);
          pk[k / 2] = *reinterpret_cast<uint32_t*>(&h);
        }
        tmem_st32u(sb + 32 * hf, pk);
      }
      if (valid < kKeys && x == 0) {
        // ragged tile: V rows past the last valid key may hold anything; zero
        // them (once the tile has landed) so that 0 * V stays 0 for both tiles
        const int stage = t % S;
        if (!wait_all(&s_v_full[stage], (t / S) & 1, budget)) {
          ok = false;
          break;
        }
        uint8_t* vt = gbase + G::kVOff + stage * G::kKVTile;
        constexpr int kChunksPerRow = G::kNH * 8;
        for (int i = threadIdx.x - 64; i < (kKeys - valid) * kChunksPerRow; i += 128) {
          const int r = valid + i / kChunksPerRow, rem = i % kChunksPerRow;
          *reinterpret_cast<uint4*>(vt + (rem >> 3) * (kKeys * 128) + r * 128 + (rem & 7) * 16) =
              make_uint4(0u, 0u, 0u, 0u);
        }
        fence_proxy_async();
        // the four warps of tile A zero disjoint rows; each arrives for itself
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&s_p_full[x]));
    }
    if (ok) {
      const int last = it.ntiles - 1;
      ok = wait_all(&s_pv_done[x], last & 1, budget) && !aborted_warp(&s_abort);
      if (ok) tc_fence_after();
    }
    if (!ok) {
      if (lane == 0) {
        note_timeout(p.status);
        s_abort = 1;
      }
    } else {
      // O_x / l -> the row's output, D columns
      const float inv = l > 0.f ? 1.f / l : 0.f;
      __nv_bfloat16* out = nullptr;
      if (mine) {
        const int q_row = it.r0 + rr;
        const int node = q_row / p.G;
        out = static_cast<__nv_bfloat16*>(p.out) +
              (static_cast<size_t>(it.s0 + node) * p.Hq + it.g * p.G + (q_row - node * p.G)) * D;
      }
#pragma unroll 1
      for (int cc = 0; cc < D / 32; ++cc) {
        float o[32];
        tmem_ld32(lane_base + static_cast<uint32_t>(x * D) + 32 * cc, o);
        if (mine) {
#pragma unroll
          for (int k = 0; k < 32; k += 8) {
            uint4 pk;
            __nv_bfloat162 h0 = __floats2bfloat162_rn(o[k] * inv, o[k + 1] * inv);
            __nv_bfloat162 h1 = __floats2bfloat162_rn(o[k + 2] * inv, o[k + 3] * inv);
            __nv_bfloat162 h2 = __floats2bfloat162_rn(o[k + 4] * inv, o[k + 5] * inv);
            __nv_bfloat162 h3 = __floats2bfloat162_rn(o[k + 6] * inv, o[k + 7] * inv);
            pk.x = *reinterpret_cast<uint32_t*>(&h0);
            pk.y = *reinterpret_cast<uint32_t*>(&h1);
            pk.z = *reinterpret_cast<uint32_t*>(&h2);
            pk.w = *reinterpret_cast<uint32_t*>(&h3);
            *reinterpret_cast<uint4*>(out + 32 * cc + k) = pk;
          }
        }
      }
    }
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, kTmemCols);
  pdl_wait();   // the next kernel's wait covers every earlier kernel
}

}  // namespace

size_t attention_tc_smem_bytes(int head_dim, bool pingpong) {
  if (pingpong)
    return 1024 + static_cast<size_t>(head_dim == 64 ? PPGeom<64>::kBytes : PPGeom<128>::kBytes);
  return 1024 + static_cast<size_t>(head_dim == 64 ? TcGeom<64>::kBytes : TcGeom<128>::kBytes);
}

bool attention_pingpong(int batch, int num_kv_heads, int G, int total_nodes, int nsm) {
  // the ping-pong kernel does two query tiles per CTA: it pays once its items
  // fill at least two waves of CTAs (measured: 1.2x the single-tile kernel's
  // work per SM; with fewer items the single-tile kernel keeps more SMs busy)
  const long long rows = static_cast<long long>(total_nodes) * G;
  const long long items = static_cast<long long>(num_kv_heads) * ((rows + kPPRows - 1) / kPPRows);
  return batch > 0 && items >= 2LL * nsm;
}

bool attention_q_tma_ok(int G) { return G >= 1 && kRows % G == 0; }

cudaError_t launch_attention_tc(const AttnParams& p, const CUtensorMap& tm_k,
                                const CUtensorMap& tm_v, const CUtensorMap& tm_tk,
                                const CUtensorMap& tm_tv, const CUtensorMap& tm_q, bool pingpong,
                                cudaStream_t s) {
  const size_t smem = attention_tc_smem_bytes(p.D, pingpong);
  if (p.D != 64 && p.D != 128) return cudaErrorInvalidValue;
  cudaError_t err;
  if (pingpong) {
    const dim3 grid((p.max_nodes * p.G + kPPRows - 1) / kPPRows, p.B * p.Hkv, 1);
    auto* k = p.D == 64 ? attn_pp_kernel<64> : attn_pp_kernel<128>;
    err = set_smem_attrs(k, smem);
    if (err != cudaSuccess) return err;
    return launch_pdl(k, grid, dim3(kThreads), smem, s, tm_k, tm_v, tm_tk, tm_tv, tm_q, p);
  }
  const dim3 grid((p.max_nodes * p.G + kRows - 1) / kRows, p.B * p.Hkv, 1);
  auto* k = p.D == 64 ? attn_tc_kernel<64> : attn_tc_kernel<128>;
  err = set_smem_attrs(k, smem);
  if (err != cudaSuccess) return err;
  return launch_pdl(k, grid, dim3(kThreads), smem, s, tm_k, tm_v, tm_tk, tm_tv, tm_q, p);
}

}  // namespace asd
