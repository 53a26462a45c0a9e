// Internal interface between the C-ABI layer (asd_api.cu) and the kernels.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>

#include "common.cuh"

namespace asd {

// Launches `kernel` with programmatic stream serialisation, so it may begin
// while the previous kernel in the stream finishes (see pdl_wait()).
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t s, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// Dynamic shared memory limit of `kernel`, and the whole unified L1 as shared
// memory, so that an LM-head CTA and an attention CTA fit on one SM together
// (the default carveout is sized for one kernel's CTAs alone).
template <typename K>
cudaError_t set_smem_attrs(K* kernel, size_t smem) {
  cudaError_t err = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
  if (err != cudaSuccess) return err;
  return cudaFuncSetAttribute(kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                              cudaSharedmemCarveoutMaxShared);
}

// ------------------------------------------------------------ tree preparation
struct PrepParams {
  const int32_t* parent;
  const int32_t* tokens;    // may be null (attention-only call)
  const int32_t* cu_nodes;
  const int32_t* ctx_len;   // may be null
  int* status;
  int* seq_flags;
  int32_t* child_start;
  int32_t* child_cnt;
  int32_t* child_tok;
  int32_t* child_id;
  float* l_draft;           // may be null; set to NaN
  int B, T, vocab, max_nodes, ctx_max;
};
cudaError_t launch_tree_prep(const PrepParams& p, cudaStream_t s);

// ------------------------------------------------------------------ attention
struct AttnParams {
  const void* q;            // [T, Hq, D]
  const void* k_cache;      // contiguous [B,Hkv,ctx_max,D] / paged [P,Hkv,ps,D]
  const void* v_cache;
  const void* tree_k;       // [T, Hkv, D]
  const void* tree_v;
  const int32_t* cu_nodes;
  const int32_t* ctx_len;
  const int32_t* page_table;  // [B, ctx_max / ps] or null
  const int32_t* parent;      // local parent ids (ancestor masks are derived in-kernel)
  int* status;
  void* out;                // [T, Hq, D]
  int B, T, Hq, Hkv, G, D;
  int ctx_max, page_size, pages_per_seq, num_pages;
  int n_splits, split_len, n_parts, max_nodes;
  float scale_log2;         // log2(e) / sqrt(D)
  int q_tma;                // tensor-core kernels: the query tiles by TMA (tm_q)
};
// bf16 path: tensor-core (mma.sync) split-KV kernel fed by TMA; tm_k / tm_v are
// 2D tensor maps over the context cache rows (box 64 columns x
// min(attention_keys_per_tile(), rows per page) rows).
// Both paths merge the splits of a group inside its thread-block cluster.
cudaError_t launch_attention_bf16(const AttnParams& p, const CUtensorMap& tm_k,
                                  const CUtensorMap& tm_v, cudaStream_t s);
cudaError_t launch_attention_f32(const AttnParams& p, cudaStream_t s);
int attention_row_blocks(int max_nodes, int G);
int attention_keys_per_tile();   // context keys per K/V tile = TMA box rows
// bf16 path on the 5th-generation tensor cores, for steps where attention has
// the SMs to itself (more than 128 tree nodes): one CTA per (128 query rows,
// sequence x KV head), the whole context, no splits (p.n_parts == 1).  tm_k /
// tm_v: 2D maps over the cache rows with boxes of 64 columns x
// min(kAttnTcKeys, rows per page) rows; tm_tk / tm_tv: 3D maps over the tree
// K/V [T, Hkv, D] with boxes of 64 columns x 1 head x kAttnTcKeys nodes;
// tm_q (with p.q_tma, where attention_q_tma_ok(G)): a 3D map over
// q [T, Hq, D] with boxes of 64 columns x G heads x kAttnTcRows / G nodes.
// pingpong: the two-query-tile form (256 rows per CTA: one tile's MMAs run
// during the other's softmax), chosen by attention_pingpong() when its items
// fill at least two waves of CTAs.
constexpr int kAttnTcRows = 128;   // query rows per CTA (per tile of the ping-pong form)
constexpr int kAttnTcKeys = 128;   // keys per tile
size_t attention_tc_smem_bytes(int head_dim, bool pingpong);
bool attention_pingpong(int batch, int num_kv_heads, int G, int total_nodes, int nsm);
bool attention_q_tma_ok(int G);   // G divides kAttnTcRows: a query box of whole nodes
cudaError_t launch_attention_tc(const AttnParams& p, const CUtensorMap& tm_k,
                                const CUtensorMap& tm_v, const CUtensorMap& tm_tk,
                                const CUtensorMap& tm_tv, const CUtensorMap& tm_q, bool pingpong,
                                cudaStream_t s);

// -------------------------------------------------------------------- LM head
struct LmParams {
  const void* hidden;       // [T, K]
  const void* w;            // [V, K]
  const int32_t* child_start;
  const int32_t* child_cnt;
  const int32_t* child_tok;
  const int32_t* child_id;
  LmPartial* part;          // [T][g_lm]
  float* l_draft;           // [T]
  int* status;
  int T, K, V, g_lm;
  int a_rows;               // node rows per hidden-state TMA box: min(128, T rounded to 8);
                            // accumulator rows past it belong to no node
  const uint8_t* w_packed;  // W in the packed streaming layout, or null ([V, K] rows via TMA)
  // Lazy LM head (one tree level per launch): the number of hidden rows is
  // read from *t_dev (at most T), written by the previous kernel; row r
  // belongs to node row_node[r].  Both null: T rows, row r = node r.
  const int* t_dev;
  const int32_t* row_node;
  // 1: W is memory of the launching device, so the wide kernel may run in
  // clusters of two that multicast W between their SMs (set by the host)
  int w_local;
};
constexpr int kLmStages = 3;       // 3 x 48 KB (a_rows <= 64): room for an attention CTA
constexpr int kLmTileN = 128;      // vocabulary rows per MMA tile
constexpr int kLmBoxRows = 32;     // vocabulary rows per range group (and per small TMA box)
size_t lmhead_tc_smem_bytes(int a_rows);
// Tensor maps of the bf16 LM head (128-byte swizzle, 64-element inner boxes):
// h: hidden [T, K], box a_rows rows; w64 / w32: W [V, K], boxes of 64 and 32
// rows (unused with a packed weight).
struct LmMaps {
  CUtensorMap h, w64, w32;
};
// bf16 path: tcgen05/TMEM GEMM with the fused max/argmax/sum-exp/l_draft epilogue.
cudaError_t launch_lmhead_bf16(const LmParams& p, const LmMaps& maps, cudaStream_t s);
// Which bf16 LM-head kernel launch_lmhead_bf16 runs for these parameters
// (asd_lm_head_variant values: 1 weight-streaming, 2 wide, 3 wide in clusters).
int lmhead_bf16_variant(const LmParams& p);

// Vocabulary ranges of the LM head: range c of g covers the 32-row groups
// [c * ngroups / g, (c + 1) * ngroups / g); each range is cut into tiles of
// up to kLmTileN rows starting at its first group.
__host__ __device__ inline int lm_range_begin(int c, int g, int ngroups) {
  return static_cast<int>(static_cast<long long>(c) * ngroups / g);
}
int lm_ranges(int vocab, int nsm);

// Packed streaming layout of the LM-head weight (asd_pack_lm_head): a header
// of kLmPackHeader bytes, then for every tile in range order and every
// k-block kb, the tile's rows (ng whole 32-row groups, zeros past V and past
// K) x 128 bytes with the 128-byte swizzle applied (16-byte chunk c of row r
// at chunk c ^ (r & 7)).  The block of a tile starting at group g0 for
// k-block kb begins at byte kLmPackHeader + 4096 * (nkb * g0 + kb * ng), so a
// stage's two k-blocks are one contiguous run.
constexpr uint32_t kLmPackMagic = 0x57445341u;  // "ASDW"
constexpr uint32_t kLmPackVersion = 1;
constexpr int kLmPackHeader = 256;
struct LmPackHeader {
  uint32_t magic, version;
  int32_t vocab, hidden, ranges;
};
size_t lm_packed_bytes(int vocab, int hidden);
cudaError_t launch_lm_pack(const void* w, void* w_packed, int vocab, int hidden, int ranges,
                           cudaStream_t s);
cudaError_t launch_lmhead_f32(const LmParams& p, cudaStream_t s);

// --------------------------------------- finalize / accepted path / K/V commit
enum TailMode : int { kTailFinalize = 1, kTailWalk = 2, kTailCompact = 4 };
struct TailParams {
  int mode;
  const int32_t* parent;
  const int32_t* tokens;
  const int32_t* cu_nodes;
  const int* seq_flags;       // from tree preparation, or null
  // finalize
  const LmPartial* part;
  int g_lm;
  float ln_tau;
  float* row_max;
  int32_t* row_argmax;        // written by finalize, read by walk
  float* row_lse;
  const float* l_draft;
  float* ratio;               // written by finalize; read by the greedy walks otherwise
  uint8_t* accept;            // written by finalize, read by walk
  // walk
  int32_t* path;              // [B, max_path]
  int32_t* path_len;
  int32_t* bonus;
  int32_t* n_promoted;
  // compact
  const void* tree_k;
  const void* tree_v;
  void* k_cache;
  void* v_cache;
  const int32_t* ctx_len;
  const int32_t* page_table;
  int32_t* ctx_len_out;
  int* status;
  int rule;                   // accepted-path reading (asd_accept_rule)
  int B, T, Hkv, D, elem_bytes, max_nodes, max_path;
  int ctx_max, page_size, pages_per_seq, num_pages;
};
cudaError_t launch_tail(const TailParams& p, cudaStream_t s);

// Lazy, level-synchronous LM head: rows are computed for the roots and for
// nodes reached through accepted nodes only, one tree level per LM-head pass.
struct LazyParams {
  const int32_t* parent;
  const int32_t* tokens;
  const int32_t* cu_nodes;
  const int* seq_flags;
  const int32_t* child_start;
  const int32_t* child_cnt;
  const int32_t* child_id;
  const void* hidden;         // [T, K] bf16
  const LmPartial* part;      // [rows of the level][g_lm]
  float* row_max;
  int32_t* row_argmax;
  float* row_lse;
  const float* l_draft;
  float* ratio;
  uint8_t* accept;
  int* count;                 // [levels + 1] rows per level
  int32_t* rows_cur;          // node ids of this level's rows
  int32_t* rows_next;
  void* h_next;               // [cap, K] bf16: hidden rows of the next level
  int* status;
  int B, T, K, g_lm, level, last_level;
  float ln_tau;
};
cudaError_t launch_lazy_init(const LazyParams& p, int levels, cudaStream_t s);
cudaError_t launch_lazy_level(const LazyParams& p, int nsm, cudaStream_t s);

}  // namespace asd
