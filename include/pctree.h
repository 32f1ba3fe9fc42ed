/*
 * pctree.h -- C ABI of the PCTree drafting-round library for NVIDIA GB300
 * (sm_103a).
 *
 * One call, pctree_draft, runs a whole PCTree drafting round (Algorithm 1) for
 * a batch of independent requests on one GPU: B sequential stages, each a
 * batched parent-conditioned Markov-head evaluation over every frontier
 * parent (Eq. 3), a vocabulary-wide log-softmax (Eq. 2), per-parent top-k
 * children scored by their joint path log-probability (Eq. 4) and a
 * layer-wise frontier prune (Sec. 4.1); then the global top-N selection under
 * the node budget and the tree tensors (Sec. 4.2; Appendix A "Tensor
 * implementation").  pctree_accept runs the greedy tree acceptance against
 * the target model's tokens (Sec. 4.2; Appendix A).
 *
 * Conventions for every entry point:
 *  - Pointers to tensors are DEVICE pointers owned by the caller; the library
 *    never allocates device memory and keeps no pointer after returning.
 *  - Work is enqueued on `stream` (a cudaStream_t; NULL = legacy default
 *    stream) and runs asynchronously: outputs are valid once the stream has
 *    reached this point.  The host returns without synchronising.
 *  - A negative return value is an error found on the host before any work
 *    was enqueued (argument checks) or a failed launch (PCTREE_ERR_CUDA).
 *    Conditions found on the device (non-finite values, a bounded wait that
 *    ran out, a root token out of range) are written to `out->status` on the
 *    device; read it after the stream has synchronised.
 *  - Tensors are dense and row-major ("C order") with the shapes stated.
 *  - Thread-safety: calls on different streams may run concurrently if they
 *    use different workspaces; the profiling switch is process-wide.
 */
#ifndef PCTREE_H_
#define PCTREE_H_

#include <stddef.h>
#include <stdint.h>

/* Symbols of this header are the library's only exported names. */
#if defined(__GNUC__)
#define PCTREE_API __attribute__((visibility("default")))
#else
#define PCTREE_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  PCTREE_OK = 0,
  PCTREE_ERR_INVALID_ARG = -1, /* a size, pointer, alignment or token is bad */
  PCTREE_ERR_WORKSPACE = -2,   /* workspace NULL, misaligned or too small    */
  PCTREE_ERR_CUDA = -3,        /* a CUDA call or launch failed               */
  PCTREE_ERR_TIMEOUT = -4,     /* a bounded device-side wait ran out         */
  PCTREE_ERR_NONFINITE = -5,   /* NaN/+inf input, or a depth with no finite
                                  logit (probabilities undefined)            */
  PCTREE_ERR_UNSUPPORTED = -6  /* shape outside the compiled limits          */
} pctree_status;

typedef enum { PCTREE_F32 = 0, PCTREE_BF16 = 1 } pctree_dtype;

/* Scoring of the tree's children.
 *   PCTREE_MODE_PARENT  PCTree: every frontier parent gets its own Markov bias
 *                       (Eqs. 2-3).
 *   PCTREE_MODE_SHARED  the Shared-Markov control of the mechanism study
 *                       (Sec. 5.3): the greedy DSpark chain of Eq. 1 is built
 *                       alongside the tree and its distribution at depth d
 *                       serves every parent at that depth (one batch-1 Markov
 *                       call per stage and request); frontier, budget,
 *                       selection and packing are unchanged.
 * k = 1 with either mode is DSpark's single chain (Sec. 4.2). */
typedef enum { PCTREE_MODE_PARENT = 0, PCTREE_MODE_SHARED = 1 } pctree_mode;

/* Storage of the Markov-head output projection W_out (bf16 heads).
 *   PCTREE_HEAD_ROWMAJOR  [V][H], row-major, as trained.
 *   PCTREE_HEAD_TILED     the same values in vocabulary tiles: an array
 *                         [ceil(V/128)][ceil(H/64)][128][64] whose block
 *                         (t, c) holds rows 128 t .. 128 t + 127 and columns
 *                         64 c .. 64 c + 63 of W_out, row-major within the
 *                         block, zero where a row >= V or a column >= H.
 *                         Every 16 KB block the round streams is then one
 *                         contiguous piece of memory.  pctree_pack_head makes
 *                         it once from the row-major matrix (the weights are
 *                         fixed, so a serving process packs them at load). */
typedef enum { PCTREE_HEAD_ROWMAJOR = 0, PCTREE_HEAD_TILED = 1 } pctree_head_layout;

/* Compiled limits. */
#define PCTREE_MAX_K 32        /* per-parent top-k and frontier width        */
#define PCTREE_MAX_N 1024      /* node budget, root included                 */
#define PCTREE_MAX_POOL 16384  /* 1 + k + (B-1) k^2 candidate nodes          */
#define PCTREE_MAX_ROWS 4096   /* batch * k Markov rows per stage            */

/*
 * Round configuration.
 *   V            vocabulary size |V|; 1 <= k <= V.
 *   H            Markov-head rank.  BF16 weights need H % 8 == 0 (16-byte
 *                rows for TMA); F32 weights take any H >= 1.
 *   B            block size: number of sequential Markov stages and the
 *                deepest drafted level (Sec. 4.1), 1 <= B.
 *   k            local branching factor: children kept per parent and width
 *                of the frontier (Sec. 4.1), 1 <= k <= PCTREE_MAX_K.
 *   N            verification node budget including the root (Sec. 4.1),
 *                1 <= N <= PCTREE_MAX_N.
 *   batch        independent requests drafted together, 1 <= batch and
 *                batch * k <= PCTREE_MAX_ROWS.
 *   pos_offset   verified prefix length: position id = depth + pos_offset
 *                (Appendix A).
 *   weight_dtype storage type of both head matrices (pctree_dtype).
 *   mode         child scoring (pctree_mode).
 *   head_layout  storage of head_out (pctree_head_layout); TILED needs
 *                BF16 weights.  E_in is always row-major.
 * The candidate pool holds 1 + k + (B-1) k^2 nodes (Sec. 4.1); it must not
 * exceed PCTREE_MAX_POOL.
 */
typedef struct {
  int32_t V, H, B, k, N, batch, pos_offset, weight_dtype, mode, head_layout;
} pctree_config;

/*
 * Output tree tensors, one block per request.  Nodes are listed breadth
 * first: by depth, then by the parent's index, then by token id; the root is
 * node 0 and every node's parent has a smaller index.  Rows beyond
 * n_nodes[r] hold -1 (logp: -inf; mask: 0).
 *   n_nodes      [batch]          min(N, pool size)
 *   tokens       [batch][N]       draft token of each node (root: root token)
 *   parent       [batch][N]       index of the parent node; root -1
 *   depth        [batch][N]       0 for the root, 1..B for drafted nodes
 *   logp         [batch][N]       joint path log-probability s (Eq. 4); root 0
 *   position_ids [batch][N]       depth + pos_offset; siblings share one
 *   mask         [batch][N][N]    1 iff column j is row i or an ancestor of i
 *                                 (the ancestor-only tree attention mask; the
 *                                 verified prefix is always visible and not
 *                                 part of this tensor)
 *   retrieve     [batch][N][B+1]  one row per leaf, in leaf-index order: the
 *                                 node indices from the root to the leaf,
 *                                 -1 padded; rows >= n_leaves[r] are all -1
 *   n_leaves     [batch]
 *   status       [1]              device status word, set to PCTREE_OK at the
 *                                 start of pctree_draft and to the first
 *                                 device-detected error code; required
 *   pool_token   [batch][P]       optional (NULL: not written).  The
 *   pool_parent  [batch][P]       candidate pool in creation order
 *   pool_logp    [batch][P]       (P = pctree_pool_capacity): token, parent's
 *                                 pool id (-1 for the root) and joint score.
 *                                 Node ids: root 0, then layer by layer; in
 *                                 a layer, the parent's frontier slot major
 *                                 and the child's rank minor.
 */
typedef struct {
  int32_t* n_nodes;
  int32_t* tokens;
  int32_t* parent;
  int32_t* depth;
  float* logp;
  int32_t* position_ids;
  uint8_t* mask;
  int32_t* retrieve;
  int32_t* n_leaves;
  int32_t* status;
  int32_t* pool_token;
  int32_t* pool_parent;
  float* pool_logp;
} pctree_tree;

/* Checks a configuration against the rules above; no GPU work. */
PCTREE_API pctree_status pctree_check_config(const pctree_config* cfg);

/* Candidate pool size 1 + k + (B-1) k^2 (Sec. 4.1); 0 for a bad config. */
PCTREE_API int32_t pctree_pool_capacity(const pctree_config* cfg);

/* Device workspace bytes pctree_draft needs for `cfg` (256-byte aligned
 * start required); 0 for a bad config.  The workspace holds the per-stage
 * Markov rows, the softmax/top-k partials of each stage, the candidate pool
 * and the frontier (and, for F32 heads only, the stage logits); its contents
 * are scratch between calls.  bf16 heads never write stage logits to memory:
 * 4.74 MB for V=151936, H=2560, B=16, k=8, N=64, batch 1; 25.6 MB for
 * V=151936, H=5120, B=16, k=16, N=128, batch 32. */
PCTREE_API size_t pctree_workspace_bytes(const pctree_config* cfg);

/*
 * One PCTree drafting round (Algorithm 1; Eqs. 2-4; Sec. 4.2; Appendix A).
 *   base_logits  [batch][B][V] float32: the backbone's shared logits L_d per
 *                request (Sec. 3.2 "Parallel backbone"); -inf allowed.
 *                Device memory, or page-locked host memory that CUDA maps
 *                into the device's address space (cudaHostAlloc,
 *                cudaHostRegister): the kernels then read it over the host
 *                link as each stage needs it, and no copy is made.  Any
 *                other host pointer: PCTREE_ERR_INVALID_ARG.
 *   head_emb     [V][H] E_in  (weight_dtype), 16-byte aligned: Markov-head
 *                input rows, one per parent token.
 *   head_out     W_out (weight_dtype), 16-byte aligned, [V][H] or tiled as
 *                cfg->head_layout says: Markov-head output projection.
 *                The head's bias for parent p is
 *                Markov(p)[v] = sum_h W_out[v][h] * E_in[p][h] (Sec. 3.2,
 *                "low-rank Markov head"), accumulated in float32.
 *   root_token   [batch] int32: the last verified token x_t of each request;
 *                out of range -> status PCTREE_ERR_INVALID_ARG.  Device
 *                memory or mapped page-locked host memory, as base_logits.
 *   out          output tensors (see pctree_tree); all non-optional pointers
 *                required.
 *   workspace    device scratch of at least pctree_workspace_bytes(cfg)
 *                bytes, 256-byte aligned, not used concurrently by another
 *                call.
 * Ranking rules: children of a parent by (log pi desc, token asc); the
 * frontier by (score desc, id asc); the global budget by (score desc, depth
 * asc, id asc).  Scores are ranked as float32; along a path they are
 * accumulated exactly as an unevaluated float pair (hi + lo, each step added
 * with Knuth's TwoSum), so the only rounding is that of each stage's float32
 * log-probability.  No float64 arithmetic runs on the device.
 * Errors: PCTREE_ERR_INVALID_ARG / _WORKSPACE / _UNSUPPORTED before any work;
 * PCTREE_ERR_CUDA if a launch fails.
 */
PCTREE_API pctree_status pctree_draft(const pctree_config* cfg, const float* base_logits,
                           const void* head_emb, const void* head_out,
                           const int32_t* root_token, const pctree_tree* out,
                           void* workspace, size_t workspace_bytes,
                           void* stream);

/*
 * The same drafting round as pctree_draft, without a caller-provided
 * workspace.  The paper has no counterpart: this is a library convenience.
 * It serves callers that cannot allocate device memory when they draft -- a
 * host framework that owns a fixed memory budget and forbids side
 * allocations, a plug-in that only receives the buffers its host hands it, a
 * latency-critical serving loop where cudaMalloc / cudaFree would
 * synchronise the device.  Inputs and outputs are as for pctree_draft.
 * Scratch: a fixed 16 MiB array inside the library, reserved on every GPU
 * that loads it until the process exits; a round whose
 * pctree_workspace_bytes exceeds 16 MiB returns PCTREE_ERR_WORKSPACE before
 * any work (batch-1 Qwen3-shaped rounds fit: V=151936 with H=2560, B=16,
 * k=8, N=64 needs 4.74 MB; with H=5120, B=16, k=16, N=128, 5.54 MB).  The first call on
 * a device, with that device current, looks up the array's address; make
 * that first call before any stream capture begins.  Every call on a device
 * shares the array, which keeps the previous call's contents (the round
 * clears what must start at zero); calls whose GPU work overlaps -- other
 * streams, other host threads -- race on it and must not be issued.  The
 * call allocates nothing: no cudaMalloc, cudaFree or allocating library
 * routine.
 */
PCTREE_API pctree_status pctree_draft_noalloc(const pctree_config* cfg,
                                              const float* base_logits,
                                              const void* head_emb,
                                              const void* head_out,
                                              const int32_t* root_token,
                                              const pctree_tree* out,
                                              void* stream);

/* Bytes of head_out in the PCTREE_HEAD_TILED layout for cfg's V and H:
 * ceil(V/128) * ceil(H/64) * 128 * 64 * 2; 0 for a bad config or F32
 * weights. */
PCTREE_API size_t pctree_packed_head_bytes(const pctree_config* cfg);

/*
 * A storage transform with no counterpart in the paper (the head's values
 * are unchanged).  Repacks a row-major bf16 W_out [V][H] (16-byte aligned)
 * into the
 * PCTREE_HEAD_TILED layout in `packed` (pctree_packed_head_bytes(cfg) bytes,
 * 16-byte aligned, not overlapping head_out); padding is written as zeros.
 * cfg->head_layout is ignored.  Stream-ordered; reads and writes each byte
 * once.  Returns PCTREE_ERR_INVALID_ARG for F32 weights, NULL or misaligned
 * pointers, PCTREE_ERR_CUDA if the launch fails.
 */
PCTREE_API pctree_status pctree_pack_head(const pctree_config* cfg, const void* head_out,
                                          void* packed, void* stream);

/*
 * Greedy tree acceptance (Sec. 4.2 "standard greedy tree rule"; Appendix A).
 * Starting at the root, repeatedly accept the child whose token equals the
 * target model's token at the current node, until no child matches.
 *   tree           the tokens, parent and n_nodes of a drafted tree (other
 *                  fields unused); an n_nodes[r] outside [0, N] is clamped
 *                  to that range, so the walk never leaves the request's rows
 *   target_tokens  [batch][N] int32: the target's greedy token at each node's
 *                  position, i.e. the token it wants as that node's child
 *   accepted_idx   [batch][B+1] out: node indices of the accepted path from
 *                  the root, -1 padded
 *   accepted_len   [batch] out: accepted draft tokens (tau = len + 1 with the
 *                  bonus token, Sec. 5.1)
 *   bonus_token    [batch] out: the target's token at the last accepted node
 */
PCTREE_API pctree_status pctree_accept(const pctree_config* cfg, const pctree_tree* tree,
                            const int32_t* target_tokens,
                            int32_t* accepted_idx, int32_t* accepted_len,
                            int32_t* bonus_token, void* stream);

/*
 * Accepted-row compaction (Appendix A "Tensor implementation": once the
 * longest accepted row is known, the KV tensors and the target's hidden
 * states are gathered along it and placed right after the verified prefix).
 * This is the step after pctree_accept.
 *
 * The verification forward wrote one row per packed tree node i into slot
 * T + i of every cache plane, T = prefix_len[r] the request's verified
 * prefix.  For accepted nodes a = accepted_idx[r][0 .. L], L =
 * accepted_len[r] (a[0] = 0 is the root):
 *   every plane:   slot T + j  <-  slot T + a[j]       (j = 0 .. L, in place)
 *   hidden states: hidden_out[r][j] <- hidden_in[r][a[j]]   (j = 0 .. L)
 * Every other slot and hidden_out row keeps its content.  The caller's next
 * verified prefix is T + L + 1 (root and accepted tokens); the bonus token
 * becomes the next root.
 *
 * A cache plane is a block of byte rows addressed as
 *   cache + layer * layer_stride + plane * plane_stride
 *         + r * request_stride + slot * slot_stride
 * (layer < layers, plane < planes, e.g. planes = 2 for K and V), which
 * covers the usual contiguous layouts ([layers][2][batch][slots][heads*dim],
 * [batch][layers][2][slots][...], ...).  Rows of distinct (layer, plane,
 * request, slot) must not overlap.  Rows are moved as raw bytes: any
 * element type.
 */
typedef struct {
  int32_t batch;          /* requests                                       */
  int32_t B;              /* draft depth: accepted_idx rows hold B+1 ints   */
  int32_t N;              /* packed tree size (nodes written after prefix)  */
  int32_t layers;         /* cache layers (0 with planes = 0: hidden only)  */
  int32_t planes;         /* cache planes per layer                         */
  int32_t max_slots;      /* slots per (layer, plane, request); T + N <= it */
  int64_t row_bytes;      /* bytes of one slot's row, multiple of 16        */
  int64_t slot_stride;    /* byte strides, each a multiple of 16            */
  int64_t request_stride;
  int64_t plane_stride;
  int64_t layer_stride;
  int64_t hidden_bytes;   /* one hidden-state row, multiple of 16; 0 = none */
} pctree_compact_layout;

/*
 *   accepted_idx  [batch][B+1] int32, as written by pctree_accept
 *   accepted_len  [batch] int32
 *   prefix_len    [batch] int32, verified prefix length T of each request
 *   cache         base of the cache planes (16-byte aligned; NULL allowed
 *                 only when layers * planes == 0)
 *   hidden_in     [batch][N][hidden_bytes] (16-byte aligned; NULL allowed
 *                 only when hidden_bytes == 0)
 *   hidden_out    [batch][B+1][hidden_bytes], must not overlap hidden_in
 *   status        one device int32, or NULL.  A request whose accepted path
 *                 is not one pctree_accept can return (a[0] != 0, indices
 *                 not strictly increasing or >= N, L outside [0, B]) or
 *                 whose T < 0 or T + N > max_slots is left untouched and
 *                 PCTREE_ERR_INVALID_ARG is stored to *status; otherwise
 *                 *status is not written (clear it before the call).
 * Returns PCTREE_ERR_INVALID_ARG for a bad layout, pointer or alignment
 * (nothing enqueued) and PCTREE_ERR_CUDA if the launch fails.  Memory
 * bound: reads and writes each moved row once.
 */
PCTREE_API pctree_status pctree_compact(const pctree_compact_layout* layout,
                                        const int32_t* accepted_idx,
                                        const int32_t* accepted_len,
                                        const int32_t* prefix_len, void* cache,
                                        const void* hidden_in, void* hidden_out,
                                        int32_t* status, void* stream);

/*
 * Tree-verification attention (Sec. 4.2: the packed tree is verified in one
 * target forward; Appendix A "Tensor implementation": a node attends to the
 * verified prefix, itself and its root-to-node ancestors).  One
 * grouped-query attention layer of that forward, for a batch of requests:
 *
 *   for node i < n_nodes[r] and query head h (KV head h / G, G = Hq / Hkv):
 *     keys  = slots 0 .. T-1 (T = prefix_len[r]) and the slots T + m of the
 *             nodes m on the path from i to the root (i included)
 *     out[r][i][h] = softmax_j(scale * <q[r][i][h], k[r][j][h/G]>) . v[r][j][h/G]
 *   rows i >= n_nodes[r] are 0.
 *
 * The ancestor sets come from the packed parent indices (parent[i] < i,
 * -1 at the root), the same tree pctree_draft writes (its `parent`
 * output); they equal the rows of its ancestor mask.  Rotary embeddings
 * (positions depth + T) are applied to q and k by the caller.
 *
 * Layouts, all bf16 and dense:
 *   q, out       [batch][N][Hq][D]
 *   k_cache,
 *   v_cache      [batch][max_slots][Hkv][D], node i of the tree at slot T + i
 * Limits: D = 128, Hq a multiple of Hkv, Hq / Hkv <= 128,
 * N <= PCTREE_ATTN_MAX_N.  Cache slots past T + n_nodes are never used
 * (their values may be anything).
 */
#define PCTREE_ATTN_MAX_N 256

typedef struct {
  int32_t batch, N, Hq, Hkv, D;
  int32_t max_slots;     /* slots per request in the caches, >= N         */
  float scale;           /* softmax scale, e.g. 1/sqrt(D)                  */
} pctree_attn_config;

/* Workspace bytes pctree_tree_attention needs (0 when a request's keys are
 * never split over several work items); 256-byte aligned, any prior content. */
PCTREE_API size_t pctree_tree_attention_workspace_bytes(const pctree_attn_config* cfg);

/*
 *   prefix_len, n_nodes  [batch] int32 (device)
 *   parent               [batch][N] int32 (device)
 *   status               one device int32 or NULL: set to
 *                        PCTREE_ERR_INVALID_ARG for a request with T < 0,
 *                        n_nodes outside [0, N] or T + n_nodes > max_slots
 *                        (its rows are 0), PCTREE_ERR_TIMEOUT if a bounded
 *                        wait ran out; otherwise not written.
 * Pointers 16-byte aligned.  Returns PCTREE_ERR_INVALID_ARG /
 * PCTREE_ERR_UNSUPPORTED / PCTREE_ERR_WORKSPACE for bad arguments (nothing
 * enqueued) and PCTREE_ERR_CUDA if the launch fails.
 */
PCTREE_API pctree_status pctree_tree_attention(
    const pctree_attn_config* cfg, const void* q, const void* k_cache,
    const void* v_cache, const int32_t* prefix_len, const int32_t* n_nodes,
    const int32_t* parent, void* out, void* workspace, size_t workspace_bytes,
    int32_t* status, void* stream);

/* Human-readable name of a status code. */
PCTREE_API const char* pctree_status_string(int32_t status);

/*
 * Kernel timing for roofline reports.  While enabled, pctree_draft records a
 * CUDA event before and after every Markov-projection launch on the call's
 * stream (at most 8192 launches are recorded).  pctree_profile_collect
 * waits for the recorded events, returns the number of launches and their
 * summed duration in milliseconds, and clears the record.  Not thread-safe.
 */
PCTREE_API pctree_status pctree_profile_enable(int32_t on);
PCTREE_API pctree_status pctree_profile_collect(int64_t* launches, double* total_ms);

/*
 * Kernel path.  PCTREE_PATH_AUTO (default) runs rounds with bf16 heads and
 * batch * k <= 16, k <= 16 as one persistent cooperative launch (all B stages
 * fused: projection, log-softmax, top-k, merge and frontier); other rounds
 * run three kernels per stage.  PCTREE_PATH_STAGEWISE forces the per-stage
 * kernels for every round (same results; used to compare the two).
 * Process-wide; not thread-safe.  Returns PCTREE_ERR_INVALID_ARG for an
 * unknown value.
 */
#define PCTREE_PATH_AUTO 0
#define PCTREE_PATH_STAGEWISE 1
PCTREE_API pctree_status pctree_set_path(int32_t path);

/*
 * Failure-detection test hook (the paper has no counterpart).  While
 * `stage` >= 1, the fused round kernel withholds the cross-CTA release of
 * that stage's parent rows, so every CTA's wait for it runs out after
 * `wait_limit_ns`; the kernel then records PCTREE_ERR_TIMEOUT in
 * out->status, drains its copies and MMAs, frees its tensor memory and
 * returns, leaving the context usable.  `wait_limit_ns` bounds every wait
 * of that kernel (1000 ns .. 10 s).  pctree_debug_stall_stage(-1,
 * 1000000000) restores normal operation (no stall, 1 s bound).
 * Process-wide, not thread-safe; returns PCTREE_ERR_INVALID_ARG for values
 * out of range.
 */
PCTREE_API pctree_status pctree_debug_stall_stage(int32_t stage, int64_t wait_limit_ns);

/* ABI version (major * 100 + minor). */
PCTREE_API int32_t pctree_version(void);

#ifdef __cplusplus
}
#endif

#endif /* PCTREE_H_ */
