/*
 * asd.h - C ABI of libasd: the per-step tree-verification path of margin-based
 * lossy speculative decoding ("Margins, Not Windows: Training-Free Per-Step
 * Lossy Speculative Decoding", arXiv 2609.02897) on one NVIDIA GB300 (sm_103a).
 *
 * One verify step (Sec. 2 "Verify", Sec. 3.1-3.2) takes a draft tree of N nodes
 * per sequence - node 0 is the root (the last committed token, whose K/V is not
 * yet in the cache), nodes 1..N-1 carry drafted tokens - and
 *   1. runs the target's attention for every node over the committed context
 *      plus the node's tree ancestors (asd_tree_attention);
 *   2. projects the node hidden states through the LM head and, without
 *      writing logits to memory, reduces every row to its max, argmax and
 *      log-sum-exp and evaluates the margin rule of Eq. 1 for every drafted
 *      token (asd_lmhead_margin);
 *   3. picks the committed root-to-node path of accepted nodes (asd_accept_path);
 *   4. appends the K/V of that path to the cache (asd_kv_compact).
 * asd_verify_step chains the four on one stream.
 *
 * Conventions shared by every call
 *  - All tensor arguments are DEVICE pointers owned by the caller; the library
 *    never allocates, frees or keeps pointers after a call returns.  Every
 *    call only enqueues work on `stream` (a cudaStream_t passed as void*; NULL
 *    is the legacy default stream) and returns without synchronising, so a
 *    sequence of calls can be captured in a CUDA graph.
 *  - Sequences are packed: cu_nodes[B+1] (int32, cu_nodes[0] = 0) delimits the
 *    nodes of each sequence in every [T, ...] array, T = cu_nodes[B] =
 *    total_nodes.  parent[T] holds LOCAL parent ids: parent[root] = -1 and
 *    0 <= parent[i] < i for the other nodes (topological numbering).  At most
 *    ASD_MAX_TREE_NODES nodes per sequence.
 *  - Row-major layouts, innermost dimension last.  Element type of q, caches,
 *    tree K/V, hidden, W and the attention output: dims->dtype (fp32 or bf16).
 *    Tensors read through TMA (q, caches, tree K/V, hidden, W) must be
 *    16-byte aligned; the calls check it and return ASD_ERR_INVALID_ARG.
 *  - tau is the paper's margin threshold kappa (Eq. 1 and the rule after it),
 *    0 < tau <= 1.  The rule is evaluated as l_draft - row_max >= ln(tau) with
 *    ln(tau) computed on the host in double precision.
 *  - Errors: arguments that the host can check (null pointers, dims, tau,
 *    workspace size) make a call return a non-OK status before anything is
 *    enqueued.  Errors that only the device can see (malformed parent array,
 *    token id outside [0, vocab), ctx_len beyond the cache, a page id outside
 *    the pool, a path longer than max_path, a bounded wait that gave up) are
 *    recorded as the FIRST error code in the workspace status word and the
 *    affected sequence gets path_len = 0 and no cache write; kernels never
 *    trap.  Every call that takes a workspace clears its status word first;
 *    asd_get_device_status reads it.  Launch failures return ASD_ERR_CUDA.
 */
#ifndef ASD_H_
#define ASD_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define ASD_ABI_VERSION 5
#define ASD_MAX_TREE_NODES 128
#define ASD_NUM_STAGE_EVENTS 5

typedef enum asd_status {
  ASD_OK = 0,
  ASD_ERR_INVALID_ARG = 1, /* null pointer, bad enum, tau outside (0, 1]       */
  ASD_ERR_SHAPE = 2,       /* dims inconsistent or unsupported; path too long   */
  ASD_ERR_TREE = 3,        /* device: malformed parent array or cu_nodes        */
  ASD_ERR_TOKEN_RANGE = 4, /* device: drafted token id outside [0, vocab)       */
  ASD_ERR_CTX_RANGE = 5,   /* device: ctx_len beyond the cache / bad page id    */
  ASD_ERR_WORKSPACE = 6,   /* workspace too small or misaligned                 */
  ASD_ERR_CUDA = 7,        /* a CUDA runtime/driver call or launch failed       */
  ASD_ERR_TIMEOUT = 8,     /* device: a bounded wait inside a kernel gave up    */
  ASD_ERR_UNSUPPORTED = 9  /* device is not sm_103 / feature not built          */
} asd_status;

typedef enum asd_dtype { ASD_F32 = 0, ASD_BF16 = 1 } asd_dtype;

/* Which committed path a verify step picks (step 3).  The paper states the
 * margin rule at the first mismatch position of a verification walk (Sec.
 * 3.2); these are its readings on a tree ("promoted" = accepted by the margin
 * rule but not the parent row's top-1):
 *   LONGEST      the longest root-to-node path of accepted nodes (default);
 *   ONCE         the longest one holding at most one promoted node;
 *   GREEDY       from the root, a strict child if any (lowest index), else the
 *                accepted child of largest ratio (lowest index on ties);
 *   GREEDY_ONCE  the greedy walk with a single promotion.
 * Equally long candidates are ordered by their node-index sequences, the
 * smallest wins. */
typedef enum asd_accept_rule {
  ASD_ACCEPT_LONGEST = 0,
  ASD_ACCEPT_ONCE = 1,
  ASD_ACCEPT_GREEDY = 2,
  ASD_ACCEPT_GREEDY_ONCE = 3
} asd_accept_rule;

/* Layout of the LM-head weight passed as w_lm. */
typedef enum asd_lm_layout {
  ASD_LM_ROWS = 0,   /* [vocab, hidden] row-major (HF lm_head.weight)            */
  ASD_LM_PACKED = 1  /* bf16 only: the buffer written by asd_pack_lm_head        */
} asd_lm_layout;

/* Which LM-head rows a call computes (asd_lmhead_margin, asd_verify_step).
 *   ASD_LM_EVERY_ROW    every node's row (default).
 *   ASD_LM_LAZY_LEVELS  only the rows the accepted-path walk can read: the
 *       roots and the nodes whose every ancestor (root excluded) was
 *       accepted, computed one tree level per pass over W (max_path passes,
 *       the later ones empty when the accepted region ends).  A verdict needs
 *       the parent's row (Eq. 1), so this is what a walk from the root can
 *       reach; the committed path, bonus token, n_promoted and the cache are
 *       those of ASD_LM_EVERY_ROW, and every computed row and verdict is
 *       bit-identical to it.  Nodes not reached keep row_max = row_lse = NaN,
 *       row_argmax = -1, ratio = l_draft = NaN and accept = 0.  Pays when the
 *       levels cost fewer weight passes than the full tree costs in flops
 *       (many sequences, few accepted nodes).  bf16 only; every tree must be
 *       shallower than max_path (a reached node at depth max_path records
 *       ASD_ERR_SHAPE).  The workspace grows by 2 x (T rounded up to 128) x
 *       hidden x 2 bytes for the levels' hidden rows.  Not available in
 *       asd_lmhead_margin_noalloc (ASD_ERR_SHAPE). */
typedef enum asd_lm_schedule {
  ASD_LM_EVERY_ROW = 0,
  ASD_LM_LAZY_LEVELS = 1
} asd_lm_schedule;

/* Shapes of one verify step.  All fields are int32. */
typedef struct asd_dims {
  int32_t batch;        /* B: number of sequences (trees)                      */
  int32_t num_q_heads;  /* Hq                                                  */
  int32_t num_kv_heads; /* Hkv; Hq % Hkv == 0 (grouped-query attention)        */
  int32_t head_dim;     /* D: 64 or 128                                        */
  int32_t hidden;       /* LM-head input width (multiple of 8)                 */
  int32_t vocab;        /* V: LM-head rows                                     */
  int32_t dtype;        /* asd_dtype                                           */
  int32_t page_size;    /* 0: contiguous cache; else tokens per page, a power
                           of two in [8, 256]                                  */
  int32_t ctx_max;      /* cache slots per sequence: contiguous capacity, or
                           (page-table columns) * page_size when paged         */
  int32_t num_pages;    /* P: pages in the pool (paged), else 0                */
  int32_t max_nodes;    /* upper bound on nodes per tree, 1..128               */
  int32_t max_path;     /* columns of the path output, >= longest root-to-leaf
                           path (nodes, root included)                         */
  int32_t lm_head_layout; /* asd_lm_layout of w_lm                             */
  int32_t accept_rule;    /* asd_accept_rule of step 3                          */
  int32_t lm_head_schedule; /* asd_lm_schedule                                  */
} asd_dims;

/* Bytes of device workspace that the calls below need for `total_nodes`
 * nodes with these dims on the current device (depends on its SM count).
 * Returns 0 if the dims are invalid.  The workspace needs no initialisation;
 * its address must be 256-byte aligned. */
size_t asd_workspace_bytes(const asd_dims* dims, int32_t total_nodes);

/*
 * Tree attention (step 1; Sec. 2 "Verify", Sec. 3.1: the target scores all
 * drafted nodes in one forward pass).
 * For node i of sequence b and query head h (KV head g = h / (Hq/Hkv)):
 *   keys   = context positions 0..ctx_len[b]-1, then the tree ancestors of i
 *            from the root down to i itself;
 *   out[i,h] = softmax_j(q[i,h] . k_j / sqrt(D)) . v_j      (fp32 softmax)
 *  q       [T, Hq, D]
 *  k_cache, v_cache: contiguous [B, Hkv, ctx_max, D], or paged pool
 *            [P, Hkv, page_size, D] addressed through
 *  page_table [B, ctx_max / page_size] int32 (NULL when contiguous)
 *  ctx_len [B] int32, 0 <= ctx_len[b] <= ctx_max
 *  tree_k, tree_v [T, Hkv, D]: the K/V of the tree nodes themselves
 *  out     [T, Hq, D] (dtype of the inputs)
 * q and K are taken as given (positions already applied).
 */
asd_status asd_tree_attention(const asd_dims* dims, const void* q, const void* k_cache,
                              const void* v_cache, const int32_t* page_table,
                              const int32_t* ctx_len, const void* tree_k, const void* tree_v,
                              const int32_t* parent, const int32_t* cu_nodes,
                              int32_t total_nodes, void* out, void* workspace,
                              size_t workspace_bytes, void* stream);

/*
 * LM head fused with the margin rule (step 2; Eq. 1 and the kappa rule).
 * logits[i,v] = sum_k hidden[i,k] * w_lm[v,k]  (fp32 accumulation; never stored)
 *  hidden [T, hidden], w_lm [V, hidden] (HF lm_head.weight layout),
 *  tokens [T] int32: drafted token of each node (the root's is ignored).
 * Per row i:  row_max[i], row_argmax[i] (lowest index attaining the max),
 *             row_lse[i] = row_max + ln sum_v exp(logit - row_max).
 * Per non-root node c with parent p:  l_draft[c] = logits[p, tokens[c]],
 *             ratio[c] = exp(l_draft[c] - row_max[p])  (Eq. 1),
 *             accept[c] = tokens[c] == row_argmax[p]  ||  ratio >= tau.
 * Roots: accept = 1, l_draft = ratio = NaN.  Outputs are [T] arrays
 * (float32 / int32 / uint8).  With dims->lm_head_layout = ASD_LM_PACKED,
 * w_lm is a buffer from asd_pack_lm_head (same results, bit for bit).
 */
asd_status asd_lmhead_margin(const asd_dims* dims, const void* hidden, const void* w_lm,
                             const int32_t* tokens, const int32_t* parent,
                             const int32_t* cu_nodes, int32_t total_nodes, float tau,
                             float* row_max, int32_t* row_argmax, float* row_lse,
                             float* l_draft, float* ratio, uint8_t* accept, void* workspace,
                             size_t workspace_bytes, void* stream);

/*
 * Streaming layout of the LM-head weight (no counterpart in the paper: a
 * one-time repacking at model load that lets the LM head read W as one
 * contiguous stream per SM instead of 128-byte pieces of 128 rows at a time,
 * which HBM serves measurably slower).
 * asd_lm_head_packed_bytes: size of the packed buffer for dims (bf16 only;
 *   0 if the dims are invalid or fp32): 256 header bytes + W rounded up to
 *   32 rows and 64 columns.
 * asd_pack_lm_head: reads w [vocab, hidden] bf16 row-major and writes
 *   w_packed (device, 256-byte aligned, packed_bytes >= the size above) on
 *   `stream`.  The order depends on the SM count of the current device: use
 *   the buffer on a device of the same kind, with the same vocab and hidden;
 *   otherwise the LM head records ASD_ERR_SHAPE in the status word (its
 *   outputs are then unspecified).  w and w_packed must not overlap.
 *   Host errors: ASD_ERR_INVALID_ARG (null / misaligned pointers),
 *   ASD_ERR_SHAPE (dims, fp32), ASD_ERR_WORKSPACE (packed_bytes too small).
 */
size_t asd_lm_head_packed_bytes(const asd_dims* dims);
asd_status asd_pack_lm_head(const asd_dims* dims, const void* w, void* w_packed,
                            size_t packed_bytes, void* stream);

/*
 * Accepted path (step 3; Sec. 3.2 and Fig. 1: verification commits the
 * drafted tokens up to the first node that is neither a strict match nor
 * promoted by the margin rule).  Over the tree: the path dims->accept_rule
 * picks among root-to-node paths whose non-root nodes all have accept = 1
 * (by default the longest, equally long paths ordered by their node-index
 * sequences, the smallest winning).
 *  accept [T] uint8, row_argmax [T] int32, tokens [T] int32 (inputs)
 *  ratio [T] float (Eq. 1, as asd_lmhead_margin writes it): read by the
 *  greedy rules only, may be NULL for the others
 *  path [B, max_path] int32: local node ids, root first, -1 padded
 *  path_len [B]: nodes on the path including the root (>= 1)
 *  bonus [B]: row_argmax of the last path node (the next committed token)
 *  n_promoted [B]: path nodes whose token is not the parent row's argmax
 */
asd_status asd_accept_path(const asd_dims* dims, const int32_t* parent, const int32_t* tokens,
                           const uint8_t* accept, const int32_t* row_argmax, const float* ratio,
                           const int32_t* cu_nodes, int32_t total_nodes, int32_t* path,
                           int32_t* path_len, int32_t* bonus, int32_t* n_promoted,
                           void* workspace, size_t workspace_bytes, void* stream);

/*
 * K/V commit of the accepted path (step 4; Sec. 2: the accepted tokens are
 * committed after one target pass).  For k < path_len[b], the K and V rows
 * (all Hkv heads) of tree node path[b,k] go to cache slot ctx_len[b] + k of
 * sequence b - in place in a contiguous cache, or through page_table (whose
 * columns past the context must already name fresh pages) when paged.
 * ctx_len_out[b] = ctx_len[b] + path_len[b].  Tree K/V and cache never alias.
 */
asd_status asd_kv_compact(const asd_dims* dims, const void* tree_k, const void* tree_v,
                          const int32_t* cu_nodes, int32_t total_nodes, const int32_t* path,
                          const int32_t* path_len, const int32_t* ctx_len,
                          const int32_t* page_table, void* k_cache, void* v_cache,
                          int32_t* ctx_len_out, void* workspace, size_t workspace_bytes,
                          void* stream);

/* Arguments of asd_verify_step: the union of the four calls above. */
typedef struct asd_verify_args {
  /* inputs */
  const void* q;
  const void* tree_k;
  const void* tree_v;
  const void* hidden;
  const void* w_lm;
  const int32_t* tokens;
  const int32_t* parent;
  const int32_t* cu_nodes;
  const int32_t* ctx_len;
  const int32_t* page_table; /* NULL when contiguous                          */
  int32_t total_nodes;
  float tau;
  /* read by attention, appended to by the commit (disjoint slots)         */
  void* k_cache;
  void* v_cache;
  /* outputs */
  void* attn_out;
  float* row_max;
  int32_t* row_argmax;
  float* row_lse;
  float* l_draft;
  float* ratio;
  uint8_t* accept;
  int32_t* path;
  int32_t* path_len;
  int32_t* bonus;
  int32_t* n_promoted;
  int32_t* ctx_len_out;
  /* optional cudaEvent_t handles (NULL to skip), recorded on `stream` at:
     [0] start, [1] after tree preparation, [2] after the LM-head GEMM
     kernel, [3] after attention, [4] after path choice and commit.  An event
     between two kernels stops them from overlapping. */
  void* stage_events[ASD_NUM_STAGE_EVENTS];
} asd_verify_args;

/* One whole verify step, steps 1-4 on one stream (same semantics as the
 * individual calls; attention reads only the slots below ctx_len, the commit
 * writes only slots at or above it). */
asd_status asd_verify_step(const asd_dims* dims, const asd_verify_args* args, void* workspace,
                           size_t workspace_bytes, void* stream);

/* Copies the workspace status word (first device-side error of the most
 * recent call, ASD_OK if none) to *status_out.  Synchronises `stream`. */
asd_status asd_get_device_status(const void* workspace, int32_t* status_out, void* stream);

const char* asd_status_string(int32_t status);
int32_t asd_abi_version(void);

/*
 * Which LM-head kernel a call with these dims, node count and weight pointer
 * runs (a diagnostic query; no counterpart in the paper; nothing is
 * launched): 1 the weight-streaming tensor-core kernel (up to 128 nodes),
 * 2 the wide kernel (more nodes, or a level of the lazy schedule), 3 the wide
 * kernel in clusters of two SMs that multicast W between them (two pairs of
 * 128-node tiles, or four and more, and an even range count), 4 the fp32 kernel,
 * 0 for invalid arguments.  The clustered form multicasts from the calling
 * GPU's own memory only: when w_lm is not device memory of the current device
 * the call runs form 2.
 */
int32_t asd_lm_head_variant(const asd_dims* dims, int32_t total_nodes, const void* w_lm);

/*
 * Which tree-attention kernel a call with these dims and node count runs (a
 * diagnostic query; no counterpart in the paper; nothing is launched): 1 the
 * bf16 split-KV kernel beside the LM head (up to 128 nodes), 2 the tensor-core
 * kernel with one 128-row query tile per CTA, 3 the tensor-core kernel with two
 * query tiles per CTA in ping-pong (when its 256-row items fill at least two
 * waves of CTAs), 4 the fp32 kernel, 0 for invalid arguments.
 */
int32_t asd_attention_variant(const asd_dims* dims, int32_t total_nodes);

/*
 * Test hook for the failure path (no counterpart in the paper).  Every wait
 * of a kernel on its own pipeline (a TMA copy, an MMA, another warp) gives up
 * after a bounded number of SM clock cycles, records ASD_ERR_TIMEOUT in the
 * workspace status word, waits for the copies and MMAs it already started,
 * releases its tensor memory and returns; the tail then commits nothing for
 * any sequence of that call (path_len 0, ctx_len_out = ctx_len).  The bound
 * is about 2 s of SM clocks.  This sets it, for the workspace-taking calls
 * enqueued afterwards in this process, to `cycles` (0 restores the default)
 * so that a test can make a wait give up on purpose; the waits for copies and
 * MMAs already in flight keep the full bound.  Set it outside any stream
 * capture.  Returns ASD_ERR_INVALID_ARG for a negative value.
 */
asd_status asd_debug_set_wait_cycles(int64_t cycles);

/*
 * Allocation-free variant of asd_lmhead_margin (the paper has no counterpart;
 * this is a library convenience).  Same arguments and outputs, but instead
 * of a caller-provided workspace it uses scratch memory that the library
 * reserves statically: a device array of ASD_NOALLOC_SCRATCH_BYTES that every
 * GPU which loads libasd holds until the process exits.  It is meant for
 * callers that cannot allocate device memory themselves, for example a plugin
 * inside a serving engine that has reserved all free device memory for its
 * own KV-cache pool, or a latency-critical loop where cudaMalloc (which may
 * synchronise the device) is not acceptable.  The call itself allocates
 * nothing.
 *  - The first call on a device, with that device current, looks up the
 *    array's device address; make that first call before any stream capture.
 *    A device reset (cudaDeviceReset) gives the device a new context; the
 *    first call after it looks the address up again, and should likewise
 *    precede any capture.
 *  - Requests whose scratch needs exceed ASD_NOALLOC_SCRATCH_BYTES return
 *    ASD_ERR_WORKSPACE without enqueuing anything (about 3,400 tree nodes on a
 *    152-SM GB300: the scratch holds 16 bytes per node per SM plus 32 bytes
 *    per node).
 *  - All calls share the one array per device and it keeps the last call's
 *    contents; every call clears what must start at zero.  Calls that overlap
 *    on the GPU (different streams without ordering) race on the scratch and
 *    must not be issued.
 *  - device_status (optional device int32, may be NULL) receives the call's
 *    device-side status word (asd_status) at the end of the enqueued work.
 */
#define ASD_NOALLOC_SCRATCH_BYTES (8u << 20)
asd_status asd_lmhead_margin_noalloc(const asd_dims* dims, const void* hidden, const void* w_lm,
                                     const int32_t* tokens, const int32_t* parent,
                                     const int32_t* cu_nodes, int32_t total_nodes, float tau,
                                     float* row_max, int32_t* row_argmax, float* row_lse,
                                     float* l_draft, float* ratio, uint8_t* accept,
                                     int32_t* device_status, void* stream);

/*
 * Dynamic tree-shape policy (Sec. 3.3, Eq. 2).  Per request, once per
 * decoding step, the Draft Confidence Score
 *     DCS = min(1, p_draft(top1) * RAR / divisor)
 * maps linearly onto a range of draft-tree triplets (n_steps, topk, ndt):
 * n_steps and ndt move from `shallow` (DCS = 0) to `deep` (DCS = 1) with DCS,
 * topk with 1 - DCS; each coordinate is start + round(span * u) with the
 * product in binary64 and halves rounded upward.  RAR is an exponential
 * moving average of the fraction of drafted nodes the target accepted:
 *     RAR <- alpha * (path_len - 1) / (nodes - 1) + (1 - alpha) * RAR,
 * starting at rar_init; the DCS of a step uses the RAR after the previous
 * step's verification.  A request with `breaker` consecutive verify steps that
 * accepted no drafted node returns to its starting state (RAR = rar_init).
 * Steps that verified only the root, or whose sequence was rejected
 * (path_len 0), leave the state unchanged.  All arithmetic is binary64 with
 * every product and sum rounded on its own (no fused multiply-add), so the
 * results do not depend on the compiler.
 * The paper's settings: alpha 0.3, divisor 0.5, shallow (3, 4, 4), deep
 * (7, 1, 8), breaker 5.
 */
typedef struct asd_policy_params {
  double alpha;       /* EMA weight of the newest step, in (0, 1]                */
  double divisor;     /* d > 0                                                    */
  double rar_init;    /* RAR at the start and after a breaker reset, in [0, 1]    */
  int32_t shallow[3]; /* (n_steps, topk, ndt) at DCS = 0; each in [1, 128]        */
  int32_t deep[3];    /* (n_steps, topk, ndt) at DCS = 1; each in [1, 128]        */
  int32_t breaker;    /* consecutive zero-accept steps that reset a request, >= 1 */
  int32_t reserved;   /* must be 0                                                */
} asd_policy_params;

/* Per-request policy state, an array of `batch` of these in device memory
 * (16 bytes each, 8-byte aligned), owned by the caller. */
typedef struct asd_policy_state {
  double rar;          /* running acceptance rate                          */
  int32_t zero_streak; /* consecutive steps without an accepted draft      */
  int32_t breaks;      /* circuit-breaker resets so far                    */
} asd_policy_state;

/* Host only (no CUDA call): every triplet the mapping returns for some DCS in
 * [0, 1], in the order of increasing DCS, so that a caller can capture one
 * CUDA graph per triplet ahead of time (Sec. 3.3).  Writes min(count, cap)
 * triplets to out[3 * i + {0, 1, 2}] (out may be NULL when cap is 0) and
 * returns their count, or -ASD_ERR_INVALID_ARG for invalid params. */
int32_t asd_policy_triplets(const asd_policy_params* params, int32_t* out, int32_t cap);

/* Sets every request's state to its start (RAR = rar_init, counts 0).
 * state: device array [batch].  Enqueued on `stream`; batch 0 enqueues
 * nothing.  Errors: null pointers, invalid params or batch < 0 ->
 * ASD_ERR_INVALID_ARG; launch failure -> ASD_ERR_CUDA. */
asd_status asd_policy_init(const asd_policy_params* params, asd_policy_state* state,
                           int32_t batch, void* stream);

/* Folds one verify step into each request's state: request b verified
 * cu_nodes[b+1] - cu_nodes[b] nodes (root included) and committed path_len[b]
 * of them (root included), as written by asd_accept_path or
 * asd_verify_step.  cu_nodes [batch+1], path_len [batch]: device int32.  A
 * request whose counts are inconsistent (path_len outside [0, nodes]) is left
 * unchanged.  Errors as asd_policy_init. */
asd_status asd_policy_update(const asd_policy_params* params, const int32_t* cu_nodes,
                             const int32_t* path_len, int32_t batch, asd_policy_state* state,
                             void* stream);

/* Picks each request's next triplet.  p_draft(top1) of request b is
 * exp(row_max[r] - row_lse[r]) of the draft model's LM-head row r = rows[b]
 * (rows may be NULL: r = b), i.e. the row statistics asd_lmhead_margin
 * writes when run on the draft's LM head.  row_max, row_lse: device float
 * [num_rows].  Writes triplet[3 * b + {0, 1, 2}] = (n_steps, topk, ndt)
 * (device int32 [batch][3]) and, if dcs is not NULL, dcs[b] (device double).
 * The state is only read.  A row index outside [0, num_rows) gives the
 * triplet (0, 0, 0) and DCS NaN for that request; a probability that is not
 * a number counts as 0.  Errors as asd_policy_init. */
asd_status asd_policy_select(const asd_policy_params* params, const float* row_max,
                             const float* row_lse, const int32_t* rows, int32_t num_rows,
                             int32_t batch, const asd_policy_state* state, int32_t* triplet,
                             double* dcs, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* ASD_H_ */
