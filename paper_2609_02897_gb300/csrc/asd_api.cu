// C-ABI entry points of libasd (declared in include/asd.h): host-side argument
// checks, workspace layout, TMA descriptors and kernel launches.  Nothing here
// allocates device memory or synchronises, except asd_get_device_status.
#include <atomic>
#include <cmath>
#include <cstring>
#include <mutex>

#include "kernels.h"

using namespace asd;

namespace {

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  });
  return fn;
}

// 2D bf16 tensor map over a row-major [rows, cols] matrix with a 128-byte
// swizzled box of [box_rows, 64] (64 bf16 = 128 bytes per box row).
bool make_tmap_bf16(CUtensorMap* tm, const void* base, uint64_t cols, uint64_t rows,
                    uint32_t box_rows) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return false;
  const cuuint64_t dims[2] = {cols, rows};
  const cuuint64_t strides[1] = {cols * 2};
  const cuuint32_t box[2] = {64, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return enc(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
             estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Tree K/V [T, Hkv, D] bf16 as a 3D map {D, Hkv, T}: a box of 64 columns x 1
// head x box_nodes nodes lands as box_nodes rows of 128 bytes (128-byte swizzle).
bool make_tree_tmap_bf16(CUtensorMap* tm, const void* base, uint64_t d, uint64_t hkv,
                         uint64_t t, uint32_t box_nodes) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return false;
  const cuuint64_t dims[3] = {d, hkv, t};
  const cuuint64_t strides[2] = {d * 2, hkv * d * 2};
  const cuuint32_t box[3] = {64, 1, box_nodes};
  const cuuint32_t estr[3] = {1, 1, 1};
  return enc(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box,
             estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// q [T, Hq, D] bf16 as a 3D map {D, Hq, T}: a box of 64 columns x G heads x
// kAttnTcRows / G nodes lands as the kAttnTcRows query rows of one KV head's
// block (node-major, head-minor), 128-byte swizzled.
bool make_q_tmap_bf16(CUtensorMap* tm, const void* base, uint64_t d, uint64_t hq, uint64_t t,
                      int g) {
  EncodeTiledFn enc = encode_fn();
  if (!enc || g < 1 || kAttnTcRows % g != 0) return false;
  const cuuint64_t dims[3] = {d, hq, t};
  const cuuint64_t strides[2] = {d * 2, hq * d * 2};
  const cuuint32_t box[3] = {64, static_cast<cuuint32_t>(g),
                             static_cast<cuuint32_t>(kAttnTcRows / g)};
  const cuuint32_t estr[3] = {1, 1, 1};
  return enc(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box,
             estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

int asd::lm_ranges(int vocab, int nsm) {
  return std::max(1, std::min(std::min(nsm, kMaxLmRanges), (vocab + kLmBoxRows - 1) / kLmBoxRows));
}

namespace {

int device_sm_count() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  static int cache[128] = {0};
  if (dev < 0 || dev >= 128) return 0;
  if (cache[dev] == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    cache[dev] = n;
  }
  return cache[dev];
}

size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

bool is_pow2(int x) { return x > 0 && (x & (x - 1)) == 0; }

bool dims_ok(const asd_dims* d) {
  if (!d) return false;
  if (d->batch < 1 || d->num_q_heads < 1 || d->num_kv_heads < 1) return false;
  if (d->num_q_heads % d->num_kv_heads) return false;
  if (d->head_dim != 64 && d->head_dim != 128) return false;
  if (d->hidden < 1 || d->vocab < 1) return false;
  if (d->dtype != ASD_F32 && d->dtype != ASD_BF16) return false;
  if (d->dtype == ASD_BF16 && d->hidden % 8) return false;
  if (d->page_size != 0 && !(is_pow2(d->page_size) && d->page_size >= 8 && d->page_size <= 256))
    return false;
  if (d->ctx_max < 0) return false;
  if (d->page_size) {
    if (d->ctx_max % d->page_size || d->num_pages < 1) return false;
  }
  if (d->max_nodes < 1 || d->max_nodes > ASD_MAX_TREE_NODES) return false;
  if (d->max_path < 1) return false;
  if (d->lm_head_layout != ASD_LM_ROWS && d->lm_head_layout != ASD_LM_PACKED) return false;
  if (d->lm_head_layout == ASD_LM_PACKED && d->dtype != ASD_BF16) return false;
  if (d->accept_rule < ASD_ACCEPT_LONGEST || d->accept_rule > ASD_ACCEPT_GREEDY_ONCE) return false;
  if (d->lm_head_schedule != ASD_LM_EVERY_ROW && d->lm_head_schedule != ASD_LM_LAZY_LEVELS)
    return false;
  if (d->lm_head_schedule == ASD_LM_LAZY_LEVELS && d->dtype != ASD_BF16) return false;
  return true;
}

bool nodes_ok(const asd_dims* d, int32_t total_nodes) {
  return total_nodes >= d->batch &&
         static_cast<int64_t>(total_nodes) <= static_cast<int64_t>(d->batch) * d->max_nodes;
}

WsLayout layout(const asd_dims& d, int T, int nsm) {
  WsLayout L{};
  const int G = d.num_q_heads / d.num_kv_heads;
  L.g_lm = lm_ranges(d.vocab, nsm);
  // context splits: at most one attention CTA per SM (in a verify step each
  // shares its SM with an LM-head CTA), at most kMaxAttnParts (the splits of a
  // row block form one thread-block cluster); the last non-empty split of a
  // sequence also takes its tree keys
  const int rblocks = attention_row_blocks(d.max_nodes, G);
  const long long base = static_cast<long long>(rblocks) * d.batch * d.num_kv_heads;
  const int max_splits = std::max(1, std::min(kMaxAttnParts, (d.ctx_max + 63) / 64));
  long long ns = nsm / base;
  ns = std::max(1LL, std::min(ns, static_cast<long long>(max_splits)));
  const int per = static_cast<int>((std::max(d.ctx_max, 1) + ns - 1) / ns);
  L.split_len = ((per + 63) / 64) * 64;
  L.n_splits = std::max(1, (d.ctx_max + L.split_len - 1) / L.split_len);
  L.n_parts = L.n_splits;
  // more than one 128-node tile: the LM head (wide kernel) leaves no room on
  // its SMs, attention runs after it on the tensor-core kernel, unsplit
  L.attn_tc = (d.dtype == ASD_BF16 && T > kAttnTcRows) ? 1 : 0;
  if (L.attn_tc && attention_pingpong(d.batch, d.num_kv_heads, G, T, nsm)) L.attn_tc = 2;
  if (L.attn_tc) {
    L.n_splits = L.n_parts = 1;
    L.split_len = std::max(d.ctx_max, 1);
  }
  size_t off = 0;
  L.status = off;      off = align256(off + 16);
  L.seq_flags = off;   off = align256(off + 4 * static_cast<size_t>(d.batch));
  L.child_start = off; off = align256(off + 4 * static_cast<size_t>(T));
  L.child_cnt = off;   off = align256(off + 4 * static_cast<size_t>(T));
  L.child_tok = off;   off = align256(off + 4 * static_cast<size_t>(T));
  L.child_id = off;    off = align256(off + 4 * static_cast<size_t>(T));
  L.lm_part = off;     off = align256(off + sizeof(LmPartial) * static_cast<size_t>(T) * L.g_lm);
  if (d.lm_head_schedule == ASD_LM_LAZY_LEVELS) {
    L.lz_cap = (T + 127) / 128 * 128;
    L.lz_count = off;  off = align256(off + 4 * (static_cast<size_t>(d.max_path) + 1));
    L.lz_rows = off;   off = align256(off + 4 * 2 * static_cast<size_t>(T));
    L.lz_h = off;      off = align256(off + 2 * 2 * static_cast<size_t>(L.lz_cap) * d.hidden);
  }
  L.total = off;
  return L;
}

template <typename T>
T* ws_at(void* ws, size_t off) {
  return reinterpret_cast<T*>(static_cast<uint8_t*>(ws) + off);
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

struct Ctx {
  asd_dims d;
  WsLayout L;
  int T;
  cudaStream_t st;
  void* ws;
};

// Wait budget (SM clock cycles) that asd_debug_set_wait_cycles set for the
// kernels of later calls; 0: the kernels' default.
std::atomic<long long> g_wait_cycles{0};

// Common checks of every workspace-taking call; fills ctx on success.
asd_status begin_call(const asd_dims* dims, int32_t total_nodes, void* ws, size_t ws_bytes,
                      void* stream, Ctx* c) {
  if (!dims_ok(dims)) return dims ? ASD_ERR_SHAPE : ASD_ERR_INVALID_ARG;
  if (!nodes_ok(dims, total_nodes)) return ASD_ERR_SHAPE;
  if (!ws) return ASD_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(ws) & 255u) return ASD_ERR_WORKSPACE;
  const int nsm = device_sm_count();
  if (nsm <= 0) return ASD_ERR_CUDA;
  c->d = *dims;
  c->T = total_nodes;
  c->L = layout(*dims, total_nodes, nsm);
  if (ws_bytes < c->L.total) return ASD_ERR_WORKSPACE;
  c->st = static_cast<cudaStream_t>(stream);
  c->ws = ws;
  if (cudaMemsetAsync(ws_at<int>(ws, c->L.status), 0, 16, c->st) != cudaSuccess)
    return ASD_ERR_CUDA;
  // a test's shorter wait budget rides in words 2-3 of the status block
  static thread_local long long budget;
  budget = g_wait_cycles.load();
  if (budget != 0 && cudaMemcpyAsync(ws_at<int>(ws, c->L.status) + 2, &budget, sizeof(budget),
                                     cudaMemcpyHostToDevice, c->st) != cudaSuccess)
    return ASD_ERR_CUDA;
  return ASD_OK;
}

PrepParams prep_params(const Ctx& c, const int32_t* parent, const int32_t* tokens,
                       const int32_t* cu, const int32_t* ctx_len, float* l_draft) {
  PrepParams p{};
  p.parent = parent;
  p.tokens = tokens;
  p.cu_nodes = cu;
  p.ctx_len = ctx_len;
  p.status = ws_at<int>(c.ws, c.L.status);
  p.seq_flags = ws_at<int>(c.ws, c.L.seq_flags);
  p.child_start = ws_at<int32_t>(c.ws, c.L.child_start);
  p.child_cnt = ws_at<int32_t>(c.ws, c.L.child_cnt);
  p.child_tok = ws_at<int32_t>(c.ws, c.L.child_tok);
  p.child_id = ws_at<int32_t>(c.ws, c.L.child_id);
  p.l_draft = l_draft;
  p.B = c.d.batch;
  p.T = c.T;
  p.vocab = c.d.vocab;
  p.max_nodes = c.d.max_nodes;
  p.ctx_max = c.d.ctx_max;
  return p;
}

asd_status run_attention(const Ctx& c, const void* q, const void* k_cache, const void* v_cache,
                         const int32_t* page_table, const int32_t* ctx_len, const void* tree_k,
                         const void* tree_v, const int32_t* parent, const int32_t* cu,
                         void* out) {
  const asd_dims& d = c.d;
  AttnParams a{};
  a.q = q;
  a.k_cache = k_cache;
  a.v_cache = v_cache;
  a.tree_k = tree_k;
  a.tree_v = tree_v;
  a.cu_nodes = cu;
  a.ctx_len = ctx_len;
  a.page_table = page_table;
  a.parent = parent;
  a.status = ws_at<int>(c.ws, c.L.status);
  a.out = out;
  a.B = d.batch;
  a.T = c.T;
  a.Hq = d.num_q_heads;
  a.Hkv = d.num_kv_heads;
  a.G = d.num_q_heads / d.num_kv_heads;
  a.D = d.head_dim;
  a.ctx_max = d.ctx_max;
  a.page_size = d.page_size;
  a.pages_per_seq = d.page_size ? d.ctx_max / d.page_size : 0;
  a.num_pages = d.num_pages;
  a.n_splits = c.L.n_splits;
  a.split_len = c.L.split_len;
  a.n_parts = c.L.n_parts;
  a.max_nodes = d.max_nodes;
  a.scale_log2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(d.head_dim)));
  cudaError_t err;
  if (c.L.attn_tc) {
    CUtensorMap tk, tv, ttk, ttv, tq;
    uint64_t rows;
    uint32_t box_rows;
    if (d.page_size == 0) {
      rows = static_cast<uint64_t>(d.batch) * d.num_kv_heads * static_cast<uint64_t>(d.ctx_max);
      box_rows = static_cast<uint32_t>(kAttnTcKeys);
    } else {
      rows = static_cast<uint64_t>(d.num_pages) * d.num_kv_heads * d.page_size;
      box_rows = static_cast<uint32_t>(std::min(d.page_size, kAttnTcKeys));
    }
    if (rows == 0) rows = 1;  // no context at all: the map is never used
    if (!make_tmap_bf16(&tk, k_cache, d.head_dim, rows, box_rows) ||
        !make_tmap_bf16(&tv, v_cache, d.head_dim, rows, box_rows) ||
        !make_tree_tmap_bf16(&ttk, tree_k, d.head_dim, d.num_kv_heads, c.T, kAttnTcKeys) ||
        !make_tree_tmap_bf16(&ttv, tree_v, d.head_dim, d.num_kv_heads, c.T, kAttnTcKeys))
      return ASD_ERR_CUDA;
    // the tensor-core kernels load the query tiles by TMA where G divides
    // their 128 rows (otherwise the softmax warps stage them; tq goes unused)
    tq = ttk;
    if (attention_q_tma_ok(a.G)) {
      if (!make_q_tmap_bf16(&tq, q, d.head_dim, d.num_q_heads, c.T, a.G)) return ASD_ERR_CUDA;
      a.q_tma = 1;
    }
    err = launch_attention_tc(a, tk, tv, ttk, ttv, tq, c.L.attn_tc == 2, c.st);
  } else if (d.dtype == ASD_BF16) {
    CUtensorMap tk, tv;
    uint64_t rows;
    uint32_t box_rows;
    if (d.page_size == 0) {
      rows = static_cast<uint64_t>(d.batch) * d.num_kv_heads * static_cast<uint64_t>(d.ctx_max);
      box_rows = static_cast<uint32_t>(attention_keys_per_tile());
    } else {
      rows = static_cast<uint64_t>(d.num_pages) * d.num_kv_heads * d.page_size;
      box_rows = static_cast<uint32_t>(std::min(d.page_size, attention_keys_per_tile()));
    }
    if (rows == 0) rows = 1;  // no context at all: the map is never used
    if (!make_tmap_bf16(&tk, k_cache, d.head_dim, rows, box_rows) ||
        !make_tmap_bf16(&tv, v_cache, d.head_dim, rows, box_rows))
      return ASD_ERR_CUDA;
    err = launch_attention_bf16(a, tk, tv, c.st);
  } else {
    err = launch_attention_f32(a, c.st);
  }
  return err == cudaSuccess ? ASD_OK : ASD_ERR_CUDA;
}

// True when `w` is device memory of the current device (the only memory the
// clustered LM head may multicast from).
bool on_this_device(const void* w) {
  int dev = 0;
  cudaPointerAttributes a{};
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  if (cudaPointerGetAttributes(&a, w) != cudaSuccess) {
    cudaGetLastError();   // an unregistered host pointer: clear the sticky-free error
    return false;
  }
  return a.type == cudaMemoryTypeDevice && a.device == dev;
}

asd_status run_lmhead(const Ctx& c, const void* hidden, const void* w, float* l_draft) {
  const asd_dims& d = c.d;
  LmParams p{};
  p.w_local = on_this_device(w) ? 1 : 0;
  p.hidden = hidden;
  p.w = w;
  p.child_start = ws_at<int32_t>(c.ws, c.L.child_start);
  p.child_cnt = ws_at<int32_t>(c.ws, c.L.child_cnt);
  p.child_tok = ws_at<int32_t>(c.ws, c.L.child_tok);
  p.child_id = ws_at<int32_t>(c.ws, c.L.child_id);
  p.part = ws_at<LmPartial>(c.ws, c.L.lm_part);
  p.l_draft = l_draft;
  p.status = ws_at<int>(c.ws, c.L.status);
  p.T = c.T;
  p.K = d.hidden;
  p.V = d.vocab;
  p.g_lm = c.L.g_lm;
  p.a_rows = std::min(128, (c.T + 7) / 8 * 8);
  cudaError_t err;
  if (d.dtype == ASD_BF16) {
    LmMaps m{};
    if (!make_tmap_bf16(&m.h, hidden, d.hidden, c.T, static_cast<uint32_t>(p.a_rows)))
      return ASD_ERR_CUDA;
    if (d.lm_head_layout == ASD_LM_PACKED) {
      p.w_packed = static_cast<const uint8_t*>(w);
    } else if (!make_tmap_bf16(&m.w64, w, d.hidden, d.vocab, 2 * kLmBoxRows) ||
               !make_tmap_bf16(&m.w32, w, d.hidden, d.vocab, kLmBoxRows)) {
      return ASD_ERR_CUDA;
    }
    err = launch_lmhead_bf16(p, m, c.st);
  } else {
    err = launch_lmhead_f32(p, c.st);
  }
  return err == cudaSuccess ? ASD_OK : ASD_ERR_CUDA;
}

float ln_tau(float tau);

// The lazy schedule (asd_lm_schedule): level 0 holds the roots; each level's
// rows go through the wide LM head, then the level kernel merges them,
// judges their children and lists the accepted ones for the next level.
// Writes every output of the finalize stage for the rows it computes.
asd_status run_lmhead_lazy(const Ctx& c, const void* hidden, const void* w,
                           const int32_t* parent, const int32_t* tokens,
                           const int32_t* cu_nodes, float tau, float* row_max,
                           int32_t* row_argmax, float* row_lse, float* l_draft, float* ratio,
                           uint8_t* accept) {
  const asd_dims& d = c.d;
  const int levels = d.max_path;
  const size_t hbytes = 2 * static_cast<size_t>(c.L.lz_cap) * d.hidden;
  void* h[2] = {ws_at<uint8_t>(c.ws, c.L.lz_h), ws_at<uint8_t>(c.ws, c.L.lz_h) + hbytes};
  int32_t* rows[2] = {ws_at<int32_t>(c.ws, c.L.lz_rows), ws_at<int32_t>(c.ws, c.L.lz_rows) + c.T};
  int* count = ws_at<int>(c.ws, c.L.lz_count);

  LmParams p{};
  p.w = w;
  p.w_local = on_this_device(w) ? 1 : 0;
  p.child_start = ws_at<int32_t>(c.ws, c.L.child_start);
  p.child_cnt = ws_at<int32_t>(c.ws, c.L.child_cnt);
  p.child_tok = ws_at<int32_t>(c.ws, c.L.child_tok);
  p.child_id = ws_at<int32_t>(c.ws, c.L.child_id);
  p.part = ws_at<LmPartial>(c.ws, c.L.lm_part);
  p.l_draft = l_draft;
  p.status = ws_at<int>(c.ws, c.L.status);
  p.T = c.T;
  p.K = d.hidden;
  p.V = d.vocab;
  p.g_lm = c.L.g_lm;
  p.a_rows = 128;
  LmMaps maps[2] = {};
  for (int k = 0; k < 2; ++k) {
    if (!make_tmap_bf16(&maps[k].h, h[k], d.hidden, c.L.lz_cap, 128)) return ASD_ERR_CUDA;
    if (d.lm_head_layout == ASD_LM_ROWS &&
        (!make_tmap_bf16(&maps[k].w64, w, d.hidden, d.vocab, 2 * kLmBoxRows) ||
         !make_tmap_bf16(&maps[k].w32, w, d.hidden, d.vocab, kLmBoxRows)))
      return ASD_ERR_CUDA;
  }
  if (d.lm_head_layout == ASD_LM_PACKED) p.w_packed = static_cast<const uint8_t*>(w);

  LazyParams z{};
  z.parent = parent;
  z.tokens = tokens;
  z.cu_nodes = cu_nodes;
  z.seq_flags = ws_at<int>(c.ws, c.L.seq_flags);
  z.child_start = p.child_start;
  z.child_cnt = p.child_cnt;
  z.child_id = p.child_id;
  z.hidden = hidden;
  z.part = p.part;
  z.row_max = row_max;
  z.row_argmax = row_argmax;
  z.row_lse = row_lse;
  z.l_draft = l_draft;
  z.ratio = ratio;
  z.accept = accept;
  z.count = count;
  z.status = p.status;
  z.B = d.batch;
  z.T = c.T;
  z.K = d.hidden;
  z.g_lm = c.L.g_lm;
  z.last_level = levels - 1;
  z.ln_tau = ln_tau(tau);
  z.rows_next = rows[0];
  z.h_next = h[0];
  if (launch_lazy_init(z, levels, c.st) != cudaSuccess) return ASD_ERR_CUDA;
  const int nsm = device_sm_count();
  for (int lv = 0; lv < levels; ++lv) {
    p.hidden = h[lv & 1];
    p.t_dev = count + lv;
    p.row_node = rows[lv & 1];
    if (launch_lmhead_bf16(p, maps[lv & 1], c.st) != cudaSuccess) return ASD_ERR_CUDA;
    z.level = lv;
    z.rows_cur = rows[lv & 1];
    z.rows_next = rows[(lv + 1) & 1];
    z.h_next = h[(lv + 1) & 1];
    if (launch_lazy_level(z, nsm, c.st) != cudaSuccess) return ASD_ERR_CUDA;
  }
  return ASD_OK;
}

TailParams tail_params(const Ctx& c, int mode) {
  TailParams t{};
  t.mode = mode;
  t.rule = c.d.accept_rule;
  t.part = ws_at<LmPartial>(c.ws, c.L.lm_part);
  t.g_lm = c.L.g_lm;
  t.status = ws_at<int>(c.ws, c.L.status);
  t.B = c.d.batch;
  t.T = c.T;
  t.Hkv = c.d.num_kv_heads;
  t.D = c.d.head_dim;
  t.elem_bytes = c.d.dtype == ASD_BF16 ? 2 : 4;
  t.max_nodes = c.d.max_nodes;
  t.max_path = c.d.max_path;
  t.ctx_max = c.d.ctx_max;
  t.page_size = c.d.page_size;
  t.pages_per_seq = c.d.page_size ? c.d.ctx_max / c.d.page_size : 0;
  t.num_pages = c.d.num_pages;
  return t;
}

bool tau_ok(float tau) { return std::isfinite(tau) && tau > 0.f && tau <= 1.f; }

float ln_tau(float tau) { return static_cast<float>(std::log(static_cast<double>(tau))); }

void record(void* ev, cudaStream_t st) {
  if (ev) cudaEventRecord(static_cast<cudaEvent_t>(ev), st);
}

}  // namespace

extern "C" {

int32_t asd_abi_version(void) { return ASD_ABI_VERSION; }

int32_t asd_attention_variant(const asd_dims* dims, int32_t total_nodes) {
  if (!dims_ok(dims) || !nodes_ok(dims, total_nodes)) return 0;
  if (dims->dtype != ASD_BF16) return 4;
  const int nsm = device_sm_count();
  if (nsm <= 0) return 0;
  const WsLayout L = layout(*dims, total_nodes, nsm);
  return L.attn_tc == 2 ? 3 : (L.attn_tc == 1 ? 2 : 1);
}

int32_t asd_lm_head_variant(const asd_dims* dims, int32_t total_nodes, const void* w_lm) {
  if (!dims_ok(dims) || !nodes_ok(dims, total_nodes) || !w_lm) return 0;
  if (dims->dtype != ASD_BF16) return 4;
  const int nsm = device_sm_count();
  if (nsm <= 0) return 0;
  LmParams p{};
  p.T = total_nodes;
  p.g_lm = lm_ranges(dims->vocab, nsm);
  p.w_local = on_this_device(w_lm) ? 1 : 0;
  p.t_dev = nullptr;
  if (dims->lm_head_schedule == ASD_LM_LAZY_LEVELS) return 2;   // one level per launch
  return lmhead_bf16_variant(p);
}

asd_status asd_debug_set_wait_cycles(int64_t cycles) {
  if (cycles < 0) return ASD_ERR_INVALID_ARG;
  g_wait_cycles.store(cycles);
  return ASD_OK;
}

const char* asd_status_string(int32_t s) {
  switch (s) {
    case ASD_OK: return "ok";
    case ASD_ERR_INVALID_ARG: return "invalid argument";
    case ASD_ERR_SHAPE: return "unsupported or inconsistent shape";
    case ASD_ERR_TREE: return "malformed draft tree";
    case ASD_ERR_TOKEN_RANGE: return "token id outside the vocabulary";
    case ASD_ERR_CTX_RANGE: return "context length or page id outside the cache";
    case ASD_ERR_WORKSPACE: return "workspace too small or misaligned";
    case ASD_ERR_CUDA: return "CUDA error";
    case ASD_ERR_TIMEOUT: return "a bounded wait inside a kernel gave up";
    case ASD_ERR_UNSUPPORTED: return "unsupported device or feature";
    default: return "unknown status";
  }
}

size_t asd_lm_head_packed_bytes(const asd_dims* dims) {
  if (!dims_ok(dims) || dims->dtype != ASD_BF16) return 0;
  return lm_packed_bytes(dims->vocab, dims->hidden);
}

asd_status asd_pack_lm_head(const asd_dims* dims, const void* w, void* w_packed,
                            size_t packed_bytes, void* stream) {
  if (!dims || !w || !w_packed) return ASD_ERR_INVALID_ARG;
  if (!dims_ok(dims) || dims->dtype != ASD_BF16) return ASD_ERR_SHAPE;
  if (!aligned16(w) || (reinterpret_cast<uintptr_t>(w_packed) & 255u)) return ASD_ERR_INVALID_ARG;
  const size_t need = lm_packed_bytes(dims->vocab, dims->hidden);
  if (packed_bytes < need) return ASD_ERR_WORKSPACE;
  const uintptr_t a0 = reinterpret_cast<uintptr_t>(w), a1 = a0 + 2ull * dims->vocab * dims->hidden;
  const uintptr_t b0 = reinterpret_cast<uintptr_t>(w_packed), b1 = b0 + need;
  if (a0 < b1 && b0 < a1) return ASD_ERR_INVALID_ARG;
  const int nsm = device_sm_count();
  if (nsm <= 0) return ASD_ERR_CUDA;
  return launch_lm_pack(w, w_packed, dims->vocab, dims->hidden, lm_ranges(dims->vocab, nsm),
                        static_cast<cudaStream_t>(stream)) == cudaSuccess
             ? ASD_OK
             : ASD_ERR_CUDA;
}

size_t asd_workspace_bytes(const asd_dims* dims, int32_t total_nodes) {
  if (!dims_ok(dims) || !nodes_ok(dims, total_nodes)) return 0;
  const int nsm = device_sm_count();
  if (nsm <= 0) return 0;
  return layout(*dims, total_nodes, nsm).total;
}

asd_status asd_tree_attention(const asd_dims* dims, const void* q, const void* k_cache,
                              const void* v_cache, const int32_t* page_table,
                              const int32_t* ctx_len, const void* tree_k, const void* tree_v,
                              const int32_t* parent, const int32_t* cu_nodes,
                              int32_t total_nodes, void* out, void* workspace,
                              size_t workspace_bytes, void* stream) {
  if (!q || !k_cache || !v_cache || !ctx_len || !tree_k || !tree_v || !parent || !cu_nodes ||
      !out)
    return ASD_ERR_INVALID_ARG;
  if (dims && dims->page_size && !page_table) return ASD_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(k_cache) || !aligned16(v_cache) || !aligned16(tree_k) ||
      !aligned16(tree_v) || !aligned16(out))
    return ASD_ERR_INVALID_ARG;
  Ctx c;
  asd_status st = begin_call(dims, total_nodes, workspace, workspace_bytes, stream, &c);
  if (st != ASD_OK) return st;
  if (launch_tree_prep(prep_params(c, parent, nullptr, cu_nodes, ctx_len, nullptr), c.st) !=
      cudaSuccess)
    return ASD_ERR_CUDA;
  return run_attention(c, q, k_cache, v_cache, page_table, ctx_len, tree_k, tree_v, parent,
                       cu_nodes, out);
}

asd_status asd_lmhead_margin(const asd_dims* dims, const void* hidden, const void* w_lm,
                             const int32_t* tokens, const int32_t* parent,
                             const int32_t* cu_nodes, int32_t total_nodes, float tau,
                             float* row_max, int32_t* row_argmax, float* row_lse,
                             float* l_draft, float* ratio, uint8_t* accept, void* workspace,
                             size_t workspace_bytes, void* stream) {
  if (!hidden || !w_lm || !tokens || !parent || !cu_nodes || !row_max || !row_argmax ||
      !row_lse || !l_draft || !ratio || !accept)
    return ASD_ERR_INVALID_ARG;
  if (!tau_ok(tau)) return ASD_ERR_INVALID_ARG;
  if (!aligned16(hidden) || !aligned16(w_lm)) return ASD_ERR_INVALID_ARG;
  Ctx c;
  asd_status st = begin_call(dims, total_nodes, workspace, workspace_bytes, stream, &c);
  if (st != ASD_OK) return st;
  if (launch_tree_prep(prep_params(c, parent, tokens, cu_nodes, nullptr, l_draft), c.st) !=
      cudaSuccess)
    return ASD_ERR_CUDA;
  if (c.d.lm_head_schedule == ASD_LM_LAZY_LEVELS)
    return run_lmhead_lazy(c, hidden, w_lm, parent, tokens, cu_nodes, tau, row_max, row_argmax,
                           row_lse, l_draft, ratio, accept);
  st = run_lmhead(c, hidden, w_lm, l_draft);
  if (st != ASD_OK) return st;
  TailParams t = tail_params(c, kTailFinalize);
  t.parent = parent;
  t.tokens = tokens;
  t.cu_nodes = cu_nodes;
  t.seq_flags = ws_at<int>(c.ws, c.L.seq_flags);
  t.ln_tau = ln_tau(tau);
  t.row_max = row_max;
  t.row_argmax = row_argmax;
  t.row_lse = row_lse;
  t.l_draft = l_draft;
  t.ratio = ratio;
  t.accept = accept;
  return launch_tail(t, c.st) == cudaSuccess ? ASD_OK : ASD_ERR_CUDA;
}

asd_status asd_accept_path(const asd_dims* dims, const int32_t* parent, const int32_t* tokens,
                           const uint8_t* accept, const int32_t* row_argmax, const float* ratio,
                           const int32_t* cu_nodes, int32_t total_nodes, int32_t* path,
                           int32_t* path_len, int32_t* bonus, int32_t* n_promoted,
                           void* workspace, size_t workspace_bytes, void* stream) {
  if (!parent || !tokens || !accept || !row_argmax || !cu_nodes || !path || !path_len || !bonus ||
      !n_promoted)
    return ASD_ERR_INVALID_ARG;
  if (dims && dims->accept_rule >= ASD_ACCEPT_GREEDY && !ratio) return ASD_ERR_INVALID_ARG;
  Ctx c;
  asd_status st = begin_call(dims, total_nodes, workspace, workspace_bytes, stream, &c);
  if (st != ASD_OK) return st;
  TailParams t = tail_params(c, kTailWalk);
  t.ratio = const_cast<float*>(ratio);
  t.parent = parent;
  t.tokens = tokens;
  t.cu_nodes = cu_nodes;
  t.accept = const_cast<uint8_t*>(accept);
  t.row_argmax = const_cast<int32_t*>(row_argmax);
  t.path = path;
  t.path_len = path_len;
  t.bonus = bonus;
  t.n_promoted = n_promoted;
  return launch_tail(t, c.st) == cudaSuccess ? ASD_OK : ASD_ERR_CUDA;
}

asd_status asd_kv_compact(const asd_dims* dims, const void* tree_k, const void* tree_v,
                          const int32_t* cu_nodes, int32_t total_nodes, const int32_t* path,
                          const int32_t* path_len, const int32_t* ctx_len,
                          const int32_t* page_table, void* k_cache, void* v_cache,
                          int32_t* ctx_len_out, void* workspace, size_t workspace_bytes,
                          void* stream) {
  if (!tree_k || !tree_v || !cu_nodes || !path || !path_len || !ctx_len || !k_cache || !v_cache ||
      !ctx_len_out)
    return ASD_ERR_INVALID_ARG;
  if (dims && dims->page_size && !page_table) return ASD_ERR_INVALID_ARG;
  if (!aligned16(tree_k) || !aligned16(tree_v) || !aligned16(k_cache) || !aligned16(v_cache))
    return ASD_ERR_INVALID_ARG;
  Ctx c;
  asd_status st = begin_call(dims, total_nodes, workspace, workspace_bytes, stream, &c);
  if (st != ASD_OK) return st;
  TailParams t = tail_params(c, kTailCompact);
  t.parent = nullptr;  // path entries are checked against the tree sizes only
  t.cu_nodes = cu_nodes;
  t.path = const_cast<int32_t*>(path);
  t.path_len = const_cast<int32_t*>(path_len);
  t.tree_k = tree_k;
  t.tree_v = tree_v;
  t.k_cache = k_cache;
  t.v_cache = v_cache;
  t.ctx_len = ctx_len;
  t.page_table = page_table;
  t.ctx_len_out = ctx_len_out;
  return launch_tail(t, c.st) == cudaSuccess ? ASD_OK : ASD_ERR_CUDA;
}

asd_status asd_verify_step(const asd_dims* dims, const asd_verify_args* a, void* workspace,
                           size_t workspace_bytes, void* stream) {
  if (!a) return ASD_ERR_INVALID_ARG;
  if (!a->q || !a->tree_k || !a->tree_v || !a->hidden || !a->w_lm || !a->tokens || !a->parent ||
      !a->cu_nodes || !a->ctx_len || !a->k_cache || !a->v_cache || !a->attn_out || !a->row_max ||
      !a->row_argmax || !a->row_lse || !a->l_draft || !a->ratio || !a->accept || !a->path ||
      !a->path_len || !a->bonus || !a->n_promoted || !a->ctx_len_out)
    return ASD_ERR_INVALID_ARG;
  if (dims && dims->page_size && !a->page_table) return ASD_ERR_INVALID_ARG;
  if (!tau_ok(a->tau)) return ASD_ERR_INVALID_ARG;
  if (!aligned16(a->q) || !aligned16(a->tree_k) || !aligned16(a->tree_v) ||
      !aligned16(a->hidden) || !aligned16(a->w_lm) || !aligned16(a->k_cache) ||
      !aligned16(a->v_cache) || !aligned16(a->attn_out))
    return ASD_ERR_INVALID_ARG;
  Ctx c;
  asd_status st = begin_call(dims, a->total_nodes, workspace, workspace_bytes, stream, &c);
  if (st != ASD_OK) return st;
  record(a->stage_events[0], c.st);
  if (launch_tree_prep(prep_params(c, a->parent, a->tokens, a->cu_nodes, a->ctx_len, a->l_draft),
                       c.st) != cudaSuccess)
    return ASD_ERR_CUDA;
  record(a->stage_events[1], c.st);
  // The LM head goes first and takes one CTA per SM; the attention kernel
  // starts right behind it (it reads no output of the LM head).  Up to 128
  // nodes its CTAs share the SMs with the LM head's while the weights stream
  // in; beyond that the wide LM head fills the SMs' shared memory and the
  // tensor-core attention runs after it.  The lazy schedule also finalises
  // the rows it computes, so the tail only walks.
  const bool lazy = c.d.lm_head_schedule == ASD_LM_LAZY_LEVELS;
  st = lazy ? run_lmhead_lazy(c, a->hidden, a->w_lm, a->parent, a->tokens, a->cu_nodes, a->tau,
                              a->row_max, a->row_argmax, a->row_lse, a->l_draft, a->ratio,
                              a->accept)
            : run_lmhead(c, a->hidden, a->w_lm, a->l_draft);
  if (st != ASD_OK) return st;
  record(a->stage_events[2], c.st);
  st = run_attention(c, a->q, a->k_cache, a->v_cache, a->page_table, a->ctx_len, a->tree_k,
                     a->tree_v, a->parent, a->cu_nodes, a->attn_out);
  if (st != ASD_OK) return st;
  record(a->stage_events[3], c.st);
  TailParams t = tail_params(c, (lazy ? 0 : kTailFinalize) | kTailWalk | kTailCompact);
  t.parent = a->parent;
  t.tokens = a->tokens;
  t.cu_nodes = a->cu_nodes;
  t.seq_flags = ws_at<int>(c.ws, c.L.seq_flags);
  t.ln_tau = ln_tau(a->tau);
  t.row_max = a->row_max;
  t.row_argmax = a->row_argmax;
  t.row_lse = a->row_lse;
  t.l_draft = a->l_draft;
  t.ratio = a->ratio;
  t.accept = a->accept;
  t.path = a->path;
  t.path_len = a->path_len;
  t.bonus = a->bonus;
  t.n_promoted = a->n_promoted;
  t.tree_k = a->tree_k;
  t.tree_v = a->tree_v;
  t.k_cache = a->k_cache;
  t.v_cache = a->v_cache;
  t.ctx_len = a->ctx_len;
  t.page_table = a->page_table;
  t.ctx_len_out = a->ctx_len_out;
  if (launch_tail(t, c.st) != cudaSuccess) return ASD_ERR_CUDA;
  record(a->stage_events[4], c.st);
  return ASD_OK;
}

asd_status asd_get_device_status(const void* workspace, int32_t* status_out, void* stream) {
  if (!workspace || !status_out) return ASD_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  int32_t v = 0;
  if (cudaMemcpyAsync(&v, workspace, sizeof(v), cudaMemcpyDeviceToHost, st) != cudaSuccess)
    return ASD_ERR_CUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return ASD_ERR_CUDA;
  *status_out = v;
  return ASD_OK;
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Allocation-free LM head (asd_lmhead_margin_noalloc).  For callers that may
// not allocate device memory (an engine that owns all free memory, a loop
// that cannot afford cudaMalloc's implicit synchronisation), the scratch of
// the LM-head path lives in this file-scope device array instead of a
// caller-provided workspace.  Host code must not hand `g_noalloc_scratch`
// itself to a kernel: in host code that name is only a host-side stand-in.
// The device address is looked up once per device with cudaGetSymbolAddress.
// ---------------------------------------------------------------------------
static __device__ __align__(256) uint8_t g_noalloc_scratch[ASD_NOALLOC_SCRATCH_BYTES];

namespace {

typedef CUresult (*CtxGetCurrentFn)(CUcontext*);

CtxGetCurrentFn ctx_get_current_fn() {
  static CtxGetCurrentFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &ptr, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<CtxGetCurrentFn>(ptr);
  });
  return fn;
}

std::mutex g_noalloc_mutex;
struct NoallocSlot {
  CUcontext ctx;
  void* ptr;
};
NoallocSlot g_noalloc[128] = {};

// Device address of the scratch array on the current device.  It is looked
// up with the device current on the first call in each context of the device
// (this first call must precede any stream capture); a device reset creates
// a new context, so the next call looks the address up again.
void* noalloc_scratch() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 128) return nullptr;
  CtxGetCurrentFn get = ctx_get_current_fn();
  if (!get) return nullptr;
  CUcontext ctx = nullptr;
  if (get(&ctx) != CUDA_SUCCESS) return nullptr;
  std::lock_guard<std::mutex> lock(g_noalloc_mutex);
  NoallocSlot& slot = g_noalloc[dev];
  if (!ctx || !slot.ptr || slot.ctx != ctx) {
    // the lookup also makes the device's primary context current if no
    // runtime call has done so yet
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return nullptr;
    if (get(&ctx) != CUDA_SUCCESS || !ctx) return nullptr;
    slot.ctx = ctx;
    slot.ptr = p;
  }
  return slot.ptr;
}

}  // namespace

extern "C" asd_status asd_lmhead_margin_noalloc(
    const asd_dims* dims, const void* hidden, const void* w_lm, const int32_t* tokens,
    const int32_t* parent, const int32_t* cu_nodes, int32_t total_nodes, float tau,
    float* row_max, int32_t* row_argmax, float* row_lse, float* l_draft, float* ratio,
    uint8_t* accept, int32_t* device_status, void* stream) {
  if (!hidden || !w_lm || !tokens || !parent || !cu_nodes || !row_max || !row_argmax ||
      !row_lse || !l_draft || !ratio || !accept)
    return ASD_ERR_INVALID_ARG;
  if (!tau_ok(tau)) return ASD_ERR_INVALID_ARG;
  if (!aligned16(hidden) || !aligned16(w_lm)) return ASD_ERR_INVALID_ARG;
  if (!dims_ok(dims)) return dims ? ASD_ERR_SHAPE : ASD_ERR_INVALID_ARG;
  if (!nodes_ok(dims, total_nodes)) return ASD_ERR_SHAPE;
  if (dims->lm_head_schedule != ASD_LM_EVERY_ROW) return ASD_ERR_SHAPE;
  const int nsm = device_sm_count();
  if (nsm <= 0) return ASD_ERR_CUDA;
  Ctx c;
  c.d = *dims;
  c.T = total_nodes;
  // the every-row schedule's workspace regions (status, flags, children lists,
  // LM-head partials), as asd_workspace_bytes counts them
  c.L = layout(*dims, total_nodes, nsm);
  if (c.L.total > ASD_NOALLOC_SCRATCH_BYTES) return ASD_ERR_WORKSPACE;
  c.ws = noalloc_scratch();
  if (!c.ws) return ASD_ERR_CUDA;
  c.st = static_cast<cudaStream_t>(stream);
  // the status word must start at zero; every other region is written before it is read
  if (cudaMemsetAsync(ws_at<int>(c.ws, c.L.status), 0, 16, c.st) != cudaSuccess)
    return ASD_ERR_CUDA;
  if (launch_tree_prep(prep_params(c, parent, tokens, cu_nodes, nullptr, l_draft), c.st) !=
      cudaSuccess)
    return ASD_ERR_CUDA;
  asd_status st = run_lmhead(c, hidden, w_lm, l_draft);
  if (st != ASD_OK) return st;
  TailParams t = tail_params(c, kTailFinalize);
  t.parent = parent;
  t.tokens = tokens;
  t.cu_nodes = cu_nodes;
  t.seq_flags = ws_at<int>(c.ws, c.L.seq_flags);
  t.ln_tau = ln_tau(tau);
  t.row_max = row_max;
  t.row_argmax = row_argmax;
  t.row_lse = row_lse;
  t.l_draft = l_draft;
  t.ratio = ratio;
  t.accept = accept;
  if (launch_tail(t, c.st) != cudaSuccess) return ASD_ERR_CUDA;
  if (device_status &&
      cudaMemcpyAsync(device_status, ws_at<int>(c.ws, c.L.status), sizeof(int32_t),
                      cudaMemcpyDeviceToDevice, c.st) != cudaSuccess)
    return ASD_ERR_CUDA;
  return ASD_OK;
}
