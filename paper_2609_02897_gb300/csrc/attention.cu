// Tree attention of the verify pass (Sec. 2 "Verify": the target scores every
// drafted node of the tree in one forward pass): the bf16 kernel that shares
// the SMs with the LM head (steps of up to 128 nodes; more go to the
// tensor-core kernel in attention_tc.cu) and the exact fp32 kernel.
//
// Work unit: one CTA per (row block, sequence x KV head, context split).  The
// query rows of a (sequence, KV head) pair are its N nodes times the G query
// heads that share the KV head (grouped-query attention), packed node-major:
// row r -> node r / G, head g*G + r % G.  Split z covers context keys
// [z*L, (z+1)*L) (flash-decoding split-KV); the CTA of the sequence's last
// non-empty split also covers the tree keys, where a node only sees its
// ancestors (bitmasks derived in-kernel from the parent array).  The splits of one
// (row block, sequence x KV head) form a thread-block cluster: each CTA keeps
// its softmax-normalised partial output and log-sum-exp in shared memory, and
// after a cluster barrier every CTA merges a slice of the rows by reading its
// peers' partials through distributed shared memory.  No partial leaves the
// cluster.
#include "kernels.h"

namespace asd {
namespace {

constexpr int kRowsPerCta = 64;   // 4 warps x 16 query rows
constexpr int kKeysPerTile = 32;  // keys per K/V tile (TMA box rows)
constexpr int kAttnStages = 2;
// With D = 128 a CTA takes 1 KB + 16 KB (Q) + 32 KB (K/V ring) of dynamic
// shared memory, small enough to share an SM with an LM-head CTA.

// ---------------------------------------------------------------- mma helpers
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr)
               : "memory");
}

__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                          uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr)
               : "memory");
}

__device__ __forceinline__ void mma_bf16(float (&c)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// Tile layout in shared memory (the TMA 128-byte swizzle): [D/64 halves]
// [ROWS rows][128 bytes]; 16-byte chunk c of row r sits at chunk c ^ (r & 7).
template <int ROWS>
__device__ __forceinline__ uint32_t sw_off(int row, int chunk) {
  return static_cast<uint32_t>((chunk >> 3) * (ROWS * 128) + row * 128 +
                               (((chunk & 7) ^ (row & 7)) << 4));
}

__device__ __forceinline__ bool anc_bit(uint64_t lo, uint64_t hi, int j) {
  return j < 64 ? ((lo >> j) & 1ull) : ((hi >> (j - 64)) & 1ull);
}

// Ancestor bitmasks (self included) of the nodes of one tree, computed by
// walking the parent array in shared memory.  Malformed entries (the tree
// preparation kernel reports them) end the walk, so the loop is bounded.
__device__ __forceinline__ void tree_ancestors(const int32_t* parent, int s0, int n, int* s_par,
                                               uint64_t (*s_anc)[2]) {
  for (int i = threadIdx.x; i < n; i += blockDim.x) s_par[i] = parent[s0 + i];
  __syncthreads();
  for (int i = threadIdx.x; i < n; i += blockDim.x) {
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
  __syncthreads();
}

struct RowMap {
  int s0, G, Hq, g, r0;
  __device__ __forceinline__ size_t grow(int r) const {
    const int rr = r0 + r;
    const int i = rr / G;
    return static_cast<size_t>(s0 + i) * Hq + g * G + (rr - i * G);
  }
};

// Key range of one CTA: context keys [kbeg, kend) and, for the sequence's
// last non-empty split (split 0 when the context is empty), the tree keys.
struct KeyRange {
  int kbeg, kend, nctx, ntree;
  __device__ KeyRange(int z, int split_len, int ctx, int n) {
    kbeg = z * split_len;
    kend = min(kbeg + split_len, ctx);
    nctx = kend > kbeg ? (kend - kbeg + kKeysPerTile - 1) / kKeysPerTile : 0;
    const int last = ctx > 0 ? (ctx - 1) / split_len : 0;
    ntree = (z == last) ? (n + kKeysPerTile - 1) / kKeysPerTile : 0;
  }
};

__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;"
               ::: "memory");
}

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

// Address of the same shared-memory location in cluster CTA `rank`.
__device__ __forceinline__ uint32_t peer_addr(uint32_t local, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(local), "r"(rank));
  return r;
}

__device__ __forceinline__ float ld_peer_f32(uint32_t addr) {
  float v;
  asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(addr) : "memory");
  return v;
}

__device__ __forceinline__ float4 ld_peer_f4(uint32_t addr) {
  float4 v;
  asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "r"(addr)
               : "memory");
  return v;
}

// Merge of the cluster's splits.  Every CTA of the cluster holds, for its
// rows, the split output normalised by its own softmax sum in s_o[r][D]
// (fp32) and the split's log2-domain log-sum-exp in s_lse[r] (-inf for an
// empty split, whose rows are zero).  After a cluster barrier, CTA `rank`
// merges rows [rank*per, (rank+1)*per):
//   out = sum_z 2^(lse_z - M) O_z / sum_z 2^(lse_z - M),
// reading its peers' shared memory; a second barrier keeps every CTA alive
// until its peers are done reading.
template <typename OutT, int D>
__device__ __forceinline__ void cluster_merge(const AttnParams& p, const RowMap& rm, int nrows,
                                              uint32_t s_o, uint32_t s_lse) {
  constexpr int kC4 = D / 4;
  __shared__ float s_w[kRowsPerCta][kMaxAttnParts];
  __shared__ float s_inv[kRowsPerCta];
  cluster_sync();
  const int P = p.n_parts;
  const uint32_t rank = cluster_rank();
  const int per = (nrows + P - 1) / P;
  const int rbeg = static_cast<int>(rank) * per;
  const int rend = min(nrows, rbeg + per);
  for (int r = rbeg + static_cast<int>(threadIdx.x); r < rend; r += blockDim.x) {
    float l[kMaxAttnParts];
    float M = -INFINITY;
#pragma unroll
    for (int zz = 0; zz < kMaxAttnParts; ++zz) {
      l[zz] = zz < P ? ld_peer_f32(peer_addr(s_lse + 4 * r, zz)) : -INFINITY;
      M = fmaxf(M, l[zz]);
    }
    float sum = 0.f;
#pragma unroll
    for (int zz = 0; zz < kMaxAttnParts; ++zz) {
      const float w = (l[zz] == -INFINITY) ? 0.f : exp2f(l[zz] - M);
      s_w[r - rbeg][zz] = w;
      sum += w;
    }
    s_inv[r - rbeg] = sum > 0.f ? 1.f / sum : 0.f;
  }
  __syncthreads();
  for (int it = threadIdx.x; it < (rend - rbeg) * kC4; it += blockDim.x) {
    const int rl = it / kC4, c4 = it - rl * kC4;
    const uint32_t off = s_o + static_cast<uint32_t>(((rbeg + rl) * D + 4 * c4) * 4);
    float4 v[kMaxAttnParts];
#pragma unroll
    for (int zz = 0; zz < kMaxAttnParts; ++zz)
      if (zz < P) v[zz] = ld_peer_f4(peer_addr(off, zz));
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int zz = 0; zz < kMaxAttnParts; ++zz) {
      if (zz < P) {
        const float w = s_w[rl][zz];
        acc.x = fmaf(w, v[zz].x, acc.x);
        acc.y = fmaf(w, v[zz].y, acc.y);
        acc.z = fmaf(w, v[zz].z, acc.z);
        acc.w = fmaf(w, v[zz].w, acc.w);
      }
    }
    const float inv = s_inv[rl];
    OutT* out = static_cast<OutT*>(p.out) + rm.grow(rbeg + rl) * D + 4 * c4;
    out[0] = from_f32<OutT>(acc.x * inv);
    out[1] = from_f32<OutT>(acc.y * inv);
    out[2] = from_f32<OutT>(acc.z * inv);
    out[3] = from_f32<OutT>(acc.w * inv);
  }
  cluster_sync();
}

// ----------------------------------------------------------- bf16 tensor path
template <int D>
__global__ void __launch_bounds__(128) attn_bf16_kernel(const __grid_constant__ CUtensorMap tm_k,
                                                        const __grid_constant__ CUtensorMap tm_v,
                                                        const AttnParams p) {
  constexpr int kTileBytes = kKeysPerTile * D * 2;   // one K or V tile
  constexpr int kQBytes = kRowsPerCta * D * 2;
  constexpr int kHalf = kKeysPerTile * 128;           // one 64-column half of a tile
  constexpr int kNH = D / 64;
  constexpr int kChunks = D / 8;
  constexpr int kNT = kKeysPerTile / 8;               // 8-key n-tiles of S per tile
  static_assert(2 * kAttnStages * kTileBytes >= kRowsPerCta * D * 4,
                "the K/V ring must hold the fp32 output rows");
  extern __shared__ uint8_t smem_raw[];
  __shared__ int s_abort;
  __shared__ int s_abort_tile;   // the tile whose wait gave up
  __shared__ float s_lse[kRowsPerCta];
  __shared__ int s_par[kMaxNodes];
  __shared__ uint64_t s_anc[kMaxNodes][2];

  pdl_launch_dependents();  // nothing downstream reads this kernel's output early
  const long long budget = wait_budget(p.status);

  // This kernel does not depend on the tree preparation: it derives the
  // ancestor masks itself and keeps every access inside the caller's arrays
  // whatever the inputs hold (the preparation kernel reports malformed ones;
  // the outputs of such a sequence are then unspecified).
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int rb = blockIdx.x, bg = blockIdx.y, z = blockIdx.z;
  const int b = bg / p.Hkv, g = bg - b * p.Hkv;
  const int s0 = p.cu_nodes[b];
  const int n = p.cu_nodes[b + 1] - s0;
  const int R = n * p.G;
  const int r0 = rb * kRowsPerCta;
  if (n <= 0 || n > kMaxNodes || s0 < 0 || s0 + n > p.T || r0 >= R) {
    pdl_wait();
    return;
  }
  const int nrows = min(kRowsPerCta, R - r0);
  const KeyRange kr(z, p.split_len, min(p.ctx_len[b], p.ctx_max), n);
  const RowMap rm{s0, p.G, p.Hq, g, r0};

  uint32_t base = smem_u32(smem_raw);
  const uint32_t pad = (1024u - (base & 1023u)) & 1023u;
  uint8_t* smem = smem_raw + pad;
  base += pad;
  const uint32_t sQ = base;
  const uint32_t sK = sQ + kQBytes;
  const uint32_t sV = sK + kAttnStages * kTileBytes;
  const uint32_t sBar = sV + kAttnStages * kTileBytes;
  uint8_t* gQ = smem;
  uint8_t* gK = smem + kQBytes;
  uint8_t* gV = gK + kAttnStages * kTileBytes;

  const int ps = p.page_size;
  uint64_t pol = 0;

  auto issue = [&](int t) {
    const int stage = t % kAttnStages;
    const int key0 = kr.kbeg + t * kKeysPerTile;
    const uint32_t dK = sK + stage * kTileBytes, dV = sV + stage * kTileBytes;
    const uint32_t bar = sBar + 8 * stage;
    if (ps == 0) {
      const int row = (b * p.Hkv + g) * p.ctx_max + key0;
      mbar_expect_tx(bar, 2 * kTileBytes);
#pragma unroll
      for (int h = 0; h < kNH; ++h) {
        tma_load_2d(dK + h * kHalf, &tm_k, bar, h * 64, row, pol);
        tma_load_2d(dV + h * kHalf, &tm_v, bar, h * 64, row, pol);
      }
    } else {
      const int br = ps < kKeysPerTile ? ps : kKeysPerTile;  // rows per box
      const int nbox = kKeysPerTile / br;
      int rows[kKeysPerTile / 8];        // page_size >= 8
      int cnt = 0;
      for (int j = 0; j < nbox; ++j) {
        const int key = key0 + j * br;
        rows[j] = -1;
        if (key >= kr.kend) continue;
        const int page = p.page_table[static_cast<size_t>(b) * p.pages_per_seq + key / ps];
        if (page < 0 || page >= p.num_pages) {
          set_status(p.status, ASD_ERR_CTX_RANGE);
          continue;
        }
        rows[j] = (page * p.Hkv + g) * ps + (key % ps);
        ++cnt;
      }
      mbar_expect_tx(bar, static_cast<uint32_t>(cnt * 2 * kNH * br * 128));
      for (int j = 0; j < nbox; ++j) {
        if (rows[j] < 0) continue;
#pragma unroll
        for (int h = 0; h < kNH; ++h) {
          tma_load_2d(dK + h * kHalf + j * br * 128, &tm_k, bar, h * 64, rows[j], pol);
          tma_load_2d(dV + h * kHalf + j * br * 128, &tm_v, bar, h * 64, rows[j], pol);
        }
      }
    }
  };

  // the producer thread sets up the barriers and starts the first K/V tiles
  // before waiting for the tree preparation and staging the query rows
  if (tid == 0) {
    s_abort = 0;
    if (kr.nctx > 0) {
      for (int s = 0; s < kAttnStages; ++s) mbar_init(sBar + 8 * s, 1);
      fence_mbar_init();
      pol = l2_policy_evict_first();
      prefetch_tmap(&tm_k);
      prefetch_tmap(&tm_v);
      for (int t = 0; t < kr.nctx && t < kAttnStages; ++t) issue(t);
    }
  }

  // after the tile loop the K/V ring holds this split's fp32 output rows
  float* s_o = reinterpret_cast<float*>(gK);
  if (kr.nctx + kr.ntree == 0) {
    // empty split: weight-zero log-sum-exp and finite (zero) rows for the merge
    for (int r = tid; r < kRowsPerCta; r += 128) s_lse[r] = -INFINITY;
    for (int idx = tid; idx < kRowsPerCta * D; idx += 128) s_o[idx] = 0.f;
    cluster_merge<__nv_bfloat16, D>(p, rm, nrows, sK, smem_u32(s_lse));
    pdl_wait();
    return;
  }
  if (kr.ntree > 0) tree_ancestors(p.parent, s0, n, s_par, s_anc);

  // query rows -> shared memory (swizzled like the TMA tiles)
  const __nv_bfloat16* q = static_cast<const __nv_bfloat16*>(p.q);
  for (int c = tid; c < kRowsPerCta * kChunks; c += 128) {
    const int r = c / kChunks, ch = c - r * kChunks;
    uint4 v = make_uint4(0u, 0u, 0u, 0u);
    if (r < nrows) v = *reinterpret_cast<const uint4*>(q + rm.grow(r) * D + ch * 8);
    *reinterpret_cast<uint4*>(gQ + sw_off<kRowsPerCta>(r, ch)) = v;
  }
  __syncthreads();

  // Q fragments stay in registers for the whole kernel
  uint32_t qa[D / 16][4];
#pragma unroll
  for (int ks = 0; ks < D / 16; ++ks) {
    const int row = warp * 16 + (lane & 7) + (((lane >> 3) & 1) << 3);
    const int chunk = 2 * ks + (lane >> 4);
    ldsm_x4(sQ + sw_off<kRowsPerCta>(row, chunk), qa[ks][0], qa[ks][1], qa[ks][2], qa[ks][3]);
  }

  // ancestor masks of this thread's two rows (tree tiles only)
  const int rowA = warp * 16 + (lane >> 2), rowB = rowA + 8;
  uint64_t aAlo = 0, aAhi = 0, aBlo = 0, aBhi = 0;
  if (kr.ntree > 0) {
    if (rowA < nrows) {
      const int node = (r0 + rowA) / p.G;
      aAlo = s_anc[node][0];
      aAhi = s_anc[node][1];
    }
    if (rowB < nrows) {
      const int node = (r0 + rowB) / p.G;
      aBlo = s_anc[node][0];
      aBhi = s_anc[node][1];
    }
  }

  float mA = -INFINITY, mB = -INFINITY, lA = 0.f, lB = 0.f;
  float o[D / 8][4];
#pragma unroll
  for (int j = 0; j < D / 8; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
  const float c = p.scale_log2;
  const int kq = lane & 3;
  const __nv_bfloat16* tk = static_cast<const __nv_bfloat16*>(p.tree_k);
  const __nv_bfloat16* tv = static_cast<const __nv_bfloat16*>(p.tree_v);

  const int ntiles = kr.nctx + kr.ntree;
  for (int t = 0; t < ntiles; ++t) {
    const int stage = t % kAttnStages;
    const bool tree_tile = t >= kr.nctx;
    const int key0 = tree_tile ? (t - kr.nctx) * kKeysPerTile : kr.kbeg + t * kKeysPerTile;
    const int valid = min(kKeysPerTile, (tree_tile ? n : kr.kend) - key0);
    uint8_t* gKs = gK + stage * kTileBytes;
    uint8_t* gVs = gV + stage * kTileBytes;
    if (tree_tile) {
      for (int cidx = tid; cidx < kKeysPerTile * kChunks; cidx += 128) {
        const int r = cidx / kChunks, ch = cidx - r * kChunks;
        uint4 kv = make_uint4(0u, 0u, 0u, 0u), vv = kv;
        if (r < valid) {
          const size_t off = (static_cast<size_t>(s0 + key0 + r) * p.Hkv + g) * D + ch * 8;
          kv = *reinterpret_cast<const uint4*>(tk + off);
          vv = *reinterpret_cast<const uint4*>(tv + off);
        }
        *reinterpret_cast<uint4*>(gKs + sw_off<kKeysPerTile>(r, ch)) = kv;
        *reinterpret_cast<uint4*>(gVs + sw_off<kKeysPerTile>(r, ch)) = vv;
      }
    } else {
      const bool ok = mbar_wait(sBar + 8 * stage, (t / kAttnStages) & 1, budget);
      if (!ok) {
        note_timeout(p.status);
        s_abort = 1;
        s_abort_tile = t;
      } else if (valid < kKeysPerTile) {
        // rows past the context may hold anything: zero V so that 0 * V stays 0
        for (int cidx = tid; cidx < (kKeysPerTile - valid) * kChunks; cidx += 128) {
          const int r = valid + cidx / kChunks, ch = cidx % kChunks;
          *reinterpret_cast<uint4*>(gVs + sw_off<kKeysPerTile>(r, ch)) = make_uint4(0u, 0u, 0u, 0u);
        }
      }
    }
    __syncthreads();
    if (s_abort) break;

    const uint32_t aK = sK + stage * kTileBytes, aV = sV + stage * kTileBytes;
    float sc[kNT][4];
#pragma unroll
    for (int j = 0; j < kNT; ++j) sc[j][0] = sc[j][1] = sc[j][2] = sc[j][3] = 0.f;
#pragma unroll
    for (int ks = 0; ks < D / 16; ++ks) {
#pragma unroll
      for (int nj = 0; nj < kNT / 2; ++nj) {
        uint32_t b0, b1, b2, b3;
        const int key = 16 * nj + (lane & 7) + ((lane >> 4) << 3);
        const int chunk = 2 * ks + ((lane >> 3) & 1);
        ldsm_x4(aK + sw_off<kKeysPerTile>(key, chunk), b0, b1, b2, b3);
        mma_bf16(sc[2 * nj], qa[ks], b0, b1);
        mma_bf16(sc[2 * nj + 1], qa[ks], b2, b3);
      }
    }
    // mask and online softmax (scores in raw units; exp2 with the folded scale)
    float mxA = -INFINITY, mxB = -INFINITY;
#pragma unroll
    for (int j = 0; j < kNT; ++j) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int local = 8 * j + 2 * kq + e;
        bool vA = local < valid, vB = vA;
        if (tree_tile) {
          vA = vA && anc_bit(aAlo, aAhi, key0 + local);
          vB = vB && anc_bit(aBlo, aBhi, key0 + local);
        }
        sc[j][e] = vA ? sc[j][e] : -INFINITY;
        sc[j][2 + e] = vB ? sc[j][2 + e] : -INFINITY;
        mxA = fmaxf(mxA, sc[j][e]);
        mxB = fmaxf(mxB, sc[j][2 + e]);
      }
    }
    mxA = fmaxf(mxA, __shfl_xor_sync(0xffffffffu, mxA, 1));
    mxA = fmaxf(mxA, __shfl_xor_sync(0xffffffffu, mxA, 2));
    mxB = fmaxf(mxB, __shfl_xor_sync(0xffffffffu, mxB, 1));
    mxB = fmaxf(mxB, __shfl_xor_sync(0xffffffffu, mxB, 2));
    const float mnA = fmaxf(mA, mxA), mnB = fmaxf(mB, mxB);
    const float muA = (mnA == -INFINITY) ? 0.f : mnA;
    const float muB = (mnB == -INFINITY) ? 0.f : mnB;
    const float alA = exp2f((mA - muA) * c), alB = exp2f((mB - muB) * c);
    mA = mnA;
    mB = mnB;
    lA *= alA;
    lB *= alB;
#pragma unroll
    for (int j = 0; j < D / 8; ++j) {
      o[j][0] *= alA;
      o[j][1] *= alA;
      o[j][2] *= alB;
      o[j][3] *= alB;
    }
    const float nA = -muA * c, nB = -muB * c;
#pragma unroll
    for (int j = 0; j < kNT; ++j) {
      sc[j][0] = exp2f(fmaf(sc[j][0], c, nA));
      sc[j][1] = exp2f(fmaf(sc[j][1], c, nA));
      sc[j][2] = exp2f(fmaf(sc[j][2], c, nB));
      sc[j][3] = exp2f(fmaf(sc[j][3], c, nB));
      lA += sc[j][0] + sc[j][1];
      lB += sc[j][2] + sc[j][3];
    }
    // O += P V
#pragma unroll
    for (int kk = 0; kk < kKeysPerTile / 16; ++kk) {
      uint32_t pa[4];
      pa[0] = pack_bf16(sc[2 * kk][0], sc[2 * kk][1]);
      pa[1] = pack_bf16(sc[2 * kk][2], sc[2 * kk][3]);
      pa[2] = pack_bf16(sc[2 * kk + 1][0], sc[2 * kk + 1][1]);
      pa[3] = pack_bf16(sc[2 * kk + 1][2], sc[2 * kk + 1][3]);
#pragma unroll
      for (int dp = 0; dp < D / 16; ++dp) {
        uint32_t b0, b1, b2, b3;
        const int key = 16 * kk + (lane & 7) + (((lane >> 3) & 1) << 3);
        const int chunk = 2 * dp + (lane >> 4);
        ldsm_x4_t(aV + sw_off<kKeysPerTile>(key, chunk), b0, b1, b2, b3);
        mma_bf16(o[2 * dp], pa, b0, b1);
        mma_bf16(o[2 * dp + 1], pa, b2, b3);
      }
    }
    __syncthreads();  // every warp is done with this stage
    if (tid == 0 && t + kAttnStages < kr.nctx) {
      fence_proxy_async();
      issue(t + kAttnStages);
    }
  }
  if (s_abort) {  // a bounded wait gave up: contribute nothing, still meet the cluster
    mA = mB = -INFINITY;
    lA = lB = 0.f;
    // the tiles issued from the one that was not waited for on are still in
    // flight: they land before the stage buffers serve the merge
    if (tid == 0)
      for (int tt = s_abort_tile; tt < kr.nctx && tt < s_abort_tile + kAttnStages; ++tt)
        mbar_wait(sBar + 8 * (tt % kAttnStages), (tt / kAttnStages) & 1);
    __syncthreads();
  }

  lA += __shfl_xor_sync(0xffffffffu, lA, 1);
  lA += __shfl_xor_sync(0xffffffffu, lA, 2);
  lB += __shfl_xor_sync(0xffffffffu, lB, 1);
  lB += __shfl_xor_sync(0xffffffffu, lB, 2);
  const float iA = lA > 0.f ? 1.f / lA : 0.f, iB = lB > 0.f ? 1.f / lB : 0.f;
#pragma unroll
  for (int j = 0; j < D / 8; ++j) {
    *reinterpret_cast<float2*>(s_o + rowA * D + 8 * j + 2 * kq) = make_float2(o[j][0] * iA, o[j][1] * iA);
    *reinterpret_cast<float2*>(s_o + rowB * D + 8 * j + 2 * kq) = make_float2(o[j][2] * iB, o[j][3] * iB);
  }
  if (kq == 0) {
    s_lse[rowA] = (mA == -INFINITY) ? -INFINITY : mA * c + log2f(lA);
    s_lse[rowB] = (mB == -INFINITY) ? -INFINITY : mB * c + log2f(lB);
  }
  cluster_merge<__nv_bfloat16, D>(p, rm, nrows, sK, smem_u32(s_lse));
  // complete only after the previous kernel in the stream has: a later
  // kernel's wait on this one then covers that kernel's outputs as well
  pdl_wait();
}

// ----------------------------------------------------------- fp32 SIMT path
// One warp per query row, 32 keys at a time: lane j scores key j of the chunk
// over the whole head dimension (its K row loads in flight with the other
// lanes'), the warp folds the chunk into the running softmax, and each lane
// accumulates P V for D/32 output columns.  Exact fp32 math for the fp32
// workloads (no reduced-precision tensor path).
template <int D>
__global__ void __launch_bounds__(128) attn_f32_kernel(const AttnParams p) {
  constexpr int kPer = D / 32;
  extern __shared__ __align__(16) uint8_t smem_raw[];
  __shared__ float s_lse[kRowsPerCta];
  __shared__ int s_par[kMaxNodes];
  __shared__ uint64_t s_anc[kMaxNodes][2];
  __shared__ __align__(16) float s_q[4][D];          // each warp's current query row
  float* s_o = reinterpret_cast<float*>(smem_raw);   // [64][D] split output rows
  pdl_launch_dependents();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int rb = blockIdx.x, bg = blockIdx.y, z = blockIdx.z;
  const int b = bg / p.Hkv, g = bg - b * p.Hkv;
  const int s0 = p.cu_nodes[b];
  const int n = p.cu_nodes[b + 1] - s0;
  const int R = n * p.G;
  const int r0 = rb * kRowsPerCta;
  if (n <= 0 || n > kMaxNodes || s0 < 0 || s0 + n > p.T || r0 >= R) {
    pdl_wait();
    return;
  }
  const int nrows = min(kRowsPerCta, R - r0);
  const KeyRange kr(z, p.split_len, min(p.ctx_len[b], p.ctx_max), n);
  const RowMap rm{s0, p.G, p.Hq, g, r0};
  const float* qp = static_cast<const float*>(p.q);
  const float* kc = static_cast<const float*>(p.k_cache);
  const float* vc = static_cast<const float*>(p.v_cache);
  const float* tk = static_cast<const float*>(p.tree_k);
  const float* tv = static_cast<const float*>(p.tree_v);
  const float c = p.scale_log2;
  const int ps = p.page_size;
  const int nctx_keys = max(0, kr.kend - kr.kbeg);
  const int ntree_keys = kr.ntree > 0 ? n : 0;
  if (ntree_keys) tree_ancestors(p.parent, s0, n, s_par, s_anc);

  // element offset of key t's K / V row for this (sequence, KV head), or -1
  // when the key does not take part (not an ancestor, or a bad page)
  auto key_off = [&](int t, uint64_t alo, uint64_t ahi) -> long long {
    if (t >= nctx_keys) {
      const int key = t - nctx_keys;
      if (!anc_bit(alo, ahi, key)) return -1;
      return (static_cast<long long>(s0 + key) * p.Hkv + g) * D;
    }
    const int key = kr.kbeg + t;
    if (ps == 0) return ((static_cast<long long>(b) * p.Hkv + g) * p.ctx_max + key) * D;
    const int page = p.page_table[static_cast<size_t>(b) * p.pages_per_seq + key / ps];
    if (page < 0 || page >= p.num_pages) {
      set_status(p.status, ASD_ERR_CTX_RANGE);
      return -1;
    }
    return ((static_cast<long long>(page) * p.Hkv + g) * ps + key % ps) * D;
  };
  const int nkeys = nctx_keys + ntree_keys;
  float* s_qw = s_q[warp];

  for (int r = warp; r < nrows; r += 4) {
    const size_t gr = rm.grow(r);
    if (nkeys == 0) {
      // empty split: weight-zero log-sum-exp and a finite (zero) row
      if (lane == 0) s_lse[r] = -INFINITY;
#pragma unroll
      for (int k = 0; k < kPer; ++k) s_o[r * D + lane + 32 * k] = 0.f;
      continue;
    }
    __syncwarp();
#pragma unroll
    for (int k = 0; k < kPer; ++k) s_qw[lane + 32 * k] = qp[gr * D + lane + 32 * k];
    __syncwarp();
    uint64_t alo = 0, ahi = 0;
    if (ntree_keys) {
      const int node = (r0 + r) / p.G;
      alo = s_anc[node][0];
      ahi = s_anc[node][1];
    }
    float ov[kPer];
#pragma unroll
    for (int k = 0; k < kPer; ++k) ov[k] = 0.f;
    float m = -INFINITY, l = 0.f;
    // 32 keys at a time: lane j scores key t0 + j over the whole head
    // dimension, then the warp folds the chunk into the running softmax and
    // every lane adds p_j V_j to its D/32 output columns
    for (int t0 = 0; t0 < nkeys; t0 += 32) {
      const int t = t0 + lane;
      const long long off = t < nkeys ? key_off(t, alo, ahi) : -1;
      float dot = -INFINITY;
      if (off >= 0) {
        const float4* kr4 = reinterpret_cast<const float4*>((t >= nctx_keys ? tk : kc) + off);
        const float4* q4 = reinterpret_cast<const float4*>(s_qw);
        float acc = 0.f;
#pragma unroll 8
        for (int d = 0; d < D / 4; ++d) {
          const float4 kk = kr4[d], qq = q4[d];
          acc = fmaf(qq.x, kk.x, acc);
          acc = fmaf(qq.y, kk.y, acc);
          acc = fmaf(qq.z, kk.z, acc);
          acc = fmaf(qq.w, kk.w, acc);
        }
        dot = acc;
      }
      float cm = dot;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) cm = fmaxf(cm, __shfl_xor_sync(0xffffffffu, cm, o));
      if (cm == -INFINITY) continue;          // nothing visible in this chunk (uniform)
      const float mn = fmaxf(m, cm);
      const float al = m == -INFINITY ? 0.f : exp2f((m - mn) * c);
      const float pe = dot == -INFINITY ? 0.f : exp2f((dot - mn) * c);
      float ps_ = pe;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) ps_ += __shfl_xor_sync(0xffffffffu, ps_, o);
      l = l * al + ps_;
#pragma unroll
      for (int k = 0; k < kPer; ++k) ov[k] *= al;
      const int nj = min(32, nkeys - t0);
#pragma unroll 4
      for (int j = 0; j < nj; ++j) {
        const float pj = __shfl_sync(0xffffffffu, pe, j);
        const long long oj = __shfl_sync(0xffffffffu, off, j);
        if (pj == 0.f || oj < 0) continue;    // uniform over the warp
        const float* vr = (t0 + j >= nctx_keys ? tv : vc) + oj;
#pragma unroll
        for (int k = 0; k < kPer; ++k) ov[k] = fmaf(pj, vr[lane + 32 * k], ov[k]);
      }
      m = mn;
    }
    const float inv = l > 0.f ? 1.f / l : 0.f;
#pragma unroll
    for (int k = 0; k < kPer; ++k) s_o[r * D + lane + 32 * k] = ov[k] * inv;
    if (lane == 0) s_lse[r] = (m == -INFINITY) ? -INFINITY : m * c + log2f(l);
  }
  cluster_merge<float, D>(p, rm, nrows, smem_u32(s_o), smem_u32(s_lse));
  pdl_wait();
}

}  // namespace

size_t attn_bf16_smem_bytes(int D) {
  const size_t tile = static_cast<size_t>(kKeysPerTile) * D * 2;
  const size_t q = static_cast<size_t>(kRowsPerCta) * D * 2;
  return 1024 + q + tile * 2 * kAttnStages + 8 * kAttnStages;
}

int attention_keys_per_tile() { return kKeysPerTile; }

int attention_row_blocks(int max_nodes, int G) {
  return (max_nodes * G + kRowsPerCta - 1) / kRowsPerCta;
}

static dim3 attn_grid(const AttnParams& p) {
  return dim3(attention_row_blocks(p.max_nodes, p.G), p.B * p.Hkv, p.n_parts);
}

// The n_parts splits of one (row block, sequence x KV head) form a cluster.
template <typename... KArgs, typename... Args>
static cudaError_t launch_attn(void (*kernel)(KArgs...), const AttnParams& p, size_t smem,
                               cudaStream_t s, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = attn_grid(p);
  cfg.blockDim = dim3(128);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 1;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = static_cast<unsigned>(p.n_parts);
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

cudaError_t launch_attention_bf16(const AttnParams& p, const CUtensorMap& tm_k,
                                  const CUtensorMap& tm_v, cudaStream_t s) {
  const size_t smem = attn_bf16_smem_bytes(p.D);
  if (p.D == 128) {
    cudaError_t err = set_smem_attrs(attn_bf16_kernel<128>, smem);
    if (err != cudaSuccess) return err;
    return launch_attn(attn_bf16_kernel<128>, p, smem, s, tm_k, tm_v, p);
  }
  cudaError_t err = set_smem_attrs(attn_bf16_kernel<64>, smem);
  if (err != cudaSuccess) return err;
  return launch_attn(attn_bf16_kernel<64>, p, smem, s, tm_k, tm_v, p);
}

cudaError_t launch_attention_f32(const AttnParams& p, cudaStream_t s) {
  const size_t smem = static_cast<size_t>(kRowsPerCta) * p.D * sizeof(float);
  if (p.D == 128) return launch_attn(attn_f32_kernel<128>, p, smem, s, p);
  return launch_attn(attn_f32_kernel<64>, p, smem, s, p);
}

}  // namespace asd
