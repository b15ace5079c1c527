/*
 * pf_verify.h -- C ABI of the GB300 verify step for retrieval-based
 * multi-token proposals (PastForward, "Experience-Guided Adaptive Decoding").
 *
 * Section 3.2 ("Single-pass token verification"): given the current token
 * y_i and a proposal retrieved from decoding-experience memory, one forward
 * pass predicts a token at every proposed position plus one more; the
 * longest proposal prefix equal to those greedy predictions is accepted and
 * the model's prediction at the first mismatch is appended, so the output
 * advances by l_acc + 1 tokens.  Section 3.4 / Section 4 ("Runtime state
 * management"): K/V states are carried forward in a cache and reused.
 *
 * This library runs the data-parallel part of that pass on one GPU:
 *   pf_verify_attention  tree-masked GQA attention of the proposal nodes over
 *                        the cached prefix (one call = one layer)
 *   pf_lmhead_accept     LM-head logits, greedy argmax per node and the greedy
 *                        descent of the proposal tree (accepted length, tokens)
 *   pf_kv_commit         copy of the accepted path's K/V rows into the cache,
 *                        all layers in one launch
 * A proposal is a tree: node 0 is the current token (its K/V is not cached
 * yet), nodes 1..N-1 are drafts, parent[j] < j.  A chain is the special case
 * parent[j] = j - 1.  Queries and tree keys arrive rotary-embedded at
 * position P + depth(node); hidden states arrive after the final norm.
 *
 * Conventions shared by every call
 *   - All tensor pointers are caller-owned DEVICE memory unless stated; the
 *     library keeps no pointer after a call returns and allocates no device
 *     memory.  Tensors are dense row-major in the layouts documented below.
 *   - Calls are asynchronous and stream-ordered on the given cudaStream_t
 *     (passed as void*; NULL = legacy default stream).
 *   - Argument errors are detected on the host before any launch and return a
 *     non-zero pf_status; pf_last_error() then describes the problem.  No
 *     call aborts the process and no kernel traps.
 *   - error_flag (optional, may be NULL): a device int32 the kernels OR a
 *     PF_DEVERR_* bit into when a device-side check fails (a bounded wait ran
 *     out, or a row fell outside the cache); the caller clears and reads it.
 */
#ifndef PF_VERIFY_H
#define PF_VERIFY_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#if defined(__GNUC__)
#define PF_API __attribute__((visibility("default")))
#else
#define PF_API
#endif

#define PF_MAX_NODES 128       /* nodes per proposal tree, root included   */
#define PF_MASK_WORDS 2        /* uint64 words of ancestor mask per node   */
#define PF_PAGE_SIZE 16        /* tokens per page of a paged KV cache      */
#define PF_MAX_LM_ROWS 256     /* total proposal nodes of one LM-head call */

typedef enum pf_status {
  PF_OK = 0,
  PF_ERR_NULL = 1,        /* a required pointer is NULL                    */
  PF_ERR_SHAPE = 2,       /* a size is out of range or inconsistent        */
  PF_ERR_DTYPE = 3,       /* unsupported dtype or dtype/shape combination  */
  PF_ERR_TREE = 4,        /* parent[] is not a topologically ordered tree  */
  PF_ERR_CAPACITY = 5,    /* the cache cannot hold prefix + committed rows */
  PF_ERR_ALIGN = 6,       /* a pointer or stride breaks 16-byte alignment  */
  PF_ERR_CUDA = 7,        /* the CUDA runtime reported an error            */
  PF_ERR_WORKSPACE = 8    /* workspace missing or smaller than required    */
} pf_status;

typedef enum pf_dtype { PF_F32 = 0, PF_BF16 = 1 } pf_dtype;
typedef enum pf_kv_layout { PF_KV_CONTIGUOUS = 0, PF_KV_PAGED = 1 } pf_kv_layout;

/* Device error bits written into *error_flag. */
#define PF_DEVERR_TIMEOUT 1    /* a bounded wait on a barrier ran out      */
#define PF_DEVERR_CAPACITY 2   /* a commit row fell outside the cache      */
#define PF_DEVERR_BOUNDS 4     /* device-side sizes (cu_nodes, prefix_len,
                                  page_table) contradict the host bounds;
                                  the affected work was skipped            */
#define PF_DEVERR_TREE 8       /* a device-side parent array is not a
                                  topologically ordered tree
                                  (pf_tree_prepare_device)                 */

/* Message for the last non-OK status returned on this host thread. */
PF_API const char* pf_last_error(void);
/* Library ABI version (major * 100 + minor). */
PF_API int32_t pf_version(void);

/*
 * pf_tree_prepare -- host-side validation of one proposal tree and its
 * ancestor bitmap (the proposal-tree structure of Section 3.2 generalised
 * from a chain to the union of retrieved chains).
 *   parent    HOST [n_nodes]; parent[0] = -1, 0 <= parent[j] < j
 *   n_nodes   1 .. PF_MAX_NODES
 *   depth_out HOST [n_nodes] or NULL; edges between node and root
 *   mask_out  HOST [n_nodes][PF_MASK_WORDS]; bit i of node j's mask is set
 *             iff node i lies on the path root -> j (j included)
 * Returns PF_ERR_TREE for a malformed tree, PF_ERR_SHAPE for a bad n_nodes.
 */
PF_API pf_status pf_tree_prepare(const int32_t* parent, int32_t n_nodes,
                          int32_t* depth_out, uint64_t* mask_out);

/*
 * pf_tree_prepare_device -- the same for a batch of proposal trees already
 * in device memory, stream-ordered (no host synchronisation), for decode
 * loops whose proposal changes every step (Section 3.2: a new proposal is
 * retrieved and verified at every decoding iteration).
 *   parent     device [total_nodes]: sequence b's tree at cu_nodes[b] ..
 *              cu_nodes[b+1]-1, parent indices local to the sequence
 *              (-1 at its root)
 *   cu_nodes   device [batch+1], cu_nodes[0] = 0, cu_nodes[batch] =
 *              total_nodes
 *   depth_out  device [total_nodes] or NULL
 *   mask_out   device [total_nodes][PF_MASK_WORDS], the layout
 *              pf_verify_attention reads
 *   error_flag optional device int32
 * Host checks: batch >= 1, 1 <= max_nodes <= PF_MAX_NODES, total_nodes >= 1,
 * mask_out 16-byte aligned.  Device checks: a sequence whose node count is
 * outside 1..max_nodes or whose nodes fall outside 0..total_nodes-1 ORs
 * PF_DEVERR_BOUNDS and is skipped; a sequence whose parent array is not a
 * topologically ordered tree (parent[0] != -1, or parent[j] outside
 * [0, j)) ORs PF_DEVERR_TREE and gets masks with only each node's own bit
 * and depth -1, so no later kernel reads outside the tree.  One launch.
 */
PF_API pf_status pf_tree_prepare_device(const int32_t* parent, const int32_t* cu_nodes,
                                        int32_t batch, int32_t total_nodes, int32_t max_nodes,
                                        int32_t* depth_out, uint64_t* mask_out,
                                        int32_t* error_flag, void* stream);

/* One layer's prefix KV cache. */
typedef struct pf_kv_view {
  int32_t layout;              /* pf_kv_layout                               */
  void* k;                     /* contiguous: [B][Hkv][max_seq][D];          */
  void* v;                     /* paged: [num_pages][Hkv][PF_PAGE_SIZE][D]   */
  int32_t max_seq;             /* contiguous: rows per (sequence, KV head)   */
  int32_t num_pages;           /* paged: pages in the pool                   */
  const int32_t* page_table;   /* paged: device [B][pages_per_seq]           */
  int32_t pages_per_seq;       /* paged: row length of page_table            */
} pf_kv_view;

/*
 * pf_verify_attention -- tree-masked grouped-query attention of the
 * proposal nodes of one layer over the reused prefix KV (Section 3.2
 * single-pass verification, over the cache carried forward per Section
 * 3.4).  For node n (global index t = cu_nodes[b] + n) and query head h,
 * KV head g = h / (Hq / Hkv):
 *   out[t,h] = sum_j softmax_j(scale * q[t,h] . k_j) v_j
 * over j in { prefix rows 0 .. prefix_len[b]-1 of sequence b, head g }
 *   U { tree rows i of sequence b : bit i of mask[t] is set }.
 * Layouts: q, out [T][Hq][D]; tree_k, tree_v [T][Hkv][D]; mask [T][2]
 * (from pf_tree_prepare, local node indices); cu_nodes [B+1] with
 * cu_nodes[0] = 0, cu_nodes[B] = T; prefix_len [B].
 * dtype PF_BF16 (D = 64 or 128, tensor cores, fp32 softmax, bf16 P.V) or
 * PF_F32 (D <= 128, CUDA cores).  Every node must have
 * 1 <= cu_nodes[b+1]-cu_nodes[b] <= max_nodes <= PF_MAX_NODES and
 * prefix_len[b] <= max_prefix_len (and <= max_seq or the page table's
 * reach).  Pointers must be 16-byte aligned.  Cache rows at positions
 * >= prefix_len[b] are never used, whatever they hold.
 */
typedef struct pf_attn_desc {
  int32_t dtype;               /* pf_dtype of q, tree_k/v, cache and out     */
  int32_t batch;               /* B >= 1                                     */
  int32_t n_q_heads;           /* Hq, a multiple of n_kv_heads               */
  int32_t n_kv_heads;          /* Hkv                                        */
  int32_t head_dim;            /* D                                          */
  float scale;                 /* <= 0 selects 1/sqrt(D)                     */
  int32_t total_nodes;         /* T = cu_nodes[B]                            */
  int32_t max_nodes;           /* bound on the nodes of any one sequence     */
  int32_t max_prefix_len;      /* bound on every prefix_len[b]               */
  const int32_t* cu_nodes;     /* device [B+1]                               */
  const int32_t* prefix_len;   /* device [B]                                 */
  const void* q;               /* device [T][Hq][D]                          */
  const void* tree_k;          /* device [T][Hkv][D]                         */
  const void* tree_v;          /* device [T][Hkv][D]                         */
  const uint64_t* mask;        /* device [T][PF_MASK_WORDS]                  */
  pf_kv_view cache;            /* this layer's prefix cache                  */
  void* out;                   /* device [T][Hq][D]                          */
  int32_t* error_flag;         /* optional device int32                      */
  int32_t flags;               /* PF_ATTN_* bits, 0 = none                   */
  void* workspace;             /* optional device scratch (see below)        */
  size_t workspace_bytes;      /* its size                                   */
  /* Launch choices (0 = the library's automatic choice for the shape).
   * They change which kernel runs and how the work is split, never the
   * result beyond floating-point rounding order. */
  int32_t kernel;              /* pf_attn_kernel                             */
  int32_t splits;              /* K/V splits per row block (cluster width):
                                  1..16; 0 for PAIR, STREAM and BATCH        */
  int32_t rows_per_cta;        /* PF_ATTN_KERNEL_TC64: 128 or 256            */
  int32_t stages;              /* PF_ATTN_KERNEL_TC128 ring depth: 2 or 3    */
  /* Optional host copies of cu_nodes[B+1] and prefix_len[B] (NULL: not
   * given).  With both given and splits = 0, PF_ATTN_KERNEL_TWO_BLOCK deals
   * the CTAs of its clusters out to the (sequence, KV head) groups in
   * proportion to their tiles (a team of CTAs per group inside one cluster)
   * where that shortens the longest piece.  The kernels read only the
   * device arrays: host copies that differ from them cost balance, never
   * correctness.  Read during the call only. */
  const int32_t* host_cu_nodes;
  const int32_t* host_prefix_len;
} pf_attn_desc;

/* Attention kernels (bf16; the fp32 path has one kernel and takes 0).
 *   MMA    warp-level mma.sync tiles (D = 64 or 128)
 *   TC64   tcgen05 tensor cores, 64-token K/V tiles, 128 or 256 query rows
 *          per CTA; the only kernel for head sizes other than 128 on them
 *   TC128  tcgen05, 128-token tiles with P kept in tensor memory, 128 rows
 *          per CTA (no balanced batch mode: a workspace is ignored)
 *   PAIR   tcgen05 on pairs of SMs (one 2-SM MMA of 256 query rows per
 *          128-token tile, each SM loading half of every K/V tile); all
 *          sequences' tiles are laid end to end and cut into one equal range
 *          per SM pair, pieces of a sequence merged by a second kernel; needs
 *          the workspace
 *   STREAM TC128's pipeline, one CTA per SM, with the same continuous split
 *          (one equal range of all sequences' tiles per SM); needs the
 *          workspace
 *   BATCH  TC128's pipeline, one CTA per SM, no cluster: each (sequence, KV
 *          head, row block) gets as many CTAs as its share of all tiles
 *          calls for (every KV head and row block of a sequence the same
 *          pieces, so they read the same pages together), and the last
 *          piece of each to finish merges the pieces in the same kernel
 *          (one launch per call); needs the workspace
 *   TWO_BLOCK  TC128's tiles with two 128-row blocks of one (sequence, KV
 *          head) per CTA, so that each K/V tile enters the SM once for up
 *          to 256 query rows (KV heads with more than 128 rows: G x nodes);
 *          clusters split the tiles as for TC128
 * TC64, TC128, PAIR, STREAM, BATCH and TWO_BLOCK need bf16 and D = 128.
 * The automatic choice takes no workspace: TWO_BLOCK with teams for a batch
 * (B > 1) whose KV heads have more than 128 query rows, when host_cu_nodes
 * and host_prefix_len are given and the team plan leaves each CTA at least
 * four tiles; otherwise TC128 (128-row CTAs in clusters that split each row
 * block's tiles) where a CTA holds several 128-token tiles, TC64 otherwise,
 * MMA for other head sizes. */
typedef enum pf_attn_kernel {
  PF_ATTN_KERNEL_AUTO = 0,
  PF_ATTN_KERNEL_MMA = 1,
  PF_ATTN_KERNEL_TC64 = 2,
  PF_ATTN_KERNEL_TC128 = 3,
  PF_ATTN_KERNEL_PAIR = 4,
  PF_ATTN_KERNEL_STREAM = 5,
  PF_ATTN_KERNEL_BATCH = 6,
  PF_ATTN_KERNEL_TWO_BLOCK = 7
} pf_attn_kernel;

/* PF_ATTN_EARLY_PREFETCH: the prefix cache, page_table, cu_nodes, prefix_len
 * and mask were all written before the kernel that precedes this call in the
 * stream started (for example: layers after the first of one verify step,
 * whose cache only the previous step's pf_kv_commit wrote).  The kernel then
 * requests its cache tiles before waiting for that preceding kernel to
 * finish (programmatic dependent launch); q, tree_k and tree_v are still
 * read only after it finishes.  Leave it clear when the preceding kernel may
 * write any of those inputs. */
#define PF_ATTN_EARLY_PREFETCH 1
/* PF_ATTN_NO_PDL: launch without programmatic dependent launch (the kernel
 * then starts only after the preceding kernel in the stream has finished). */
#define PF_ATTN_NO_PDL 2

/* Workspace (bf16, head_dim 128; needed by PF_ATTN_KERNEL_PAIR, _STREAM and
 * _BATCH, optional for PF_ATTN_KERNEL_TC64): with workspace != NULL and at
 * least pf_verify_attention_workspace_size(d) bytes (16-byte aligned), the
 * KV tiles are dealt out in proportion to each sequence's length (prefix
 * plus proposal tiles) -- on BATCH (any B) and TC64 (B > 1) to one CTA per
 * SM, on STREAM and PAIR in one equal range of all sequences' tiles per SM
 * (pair) for any B -- so long and short prefixes finish together.
 * Sequences spread over several CTAs are merged by the last of their CTAs
 * to finish (BATCH) or by a second kernel in the same stream (TC64, STREAM,
 * PAIR: the call then launches two kernels; see
 * pf_verify_attention_launches).  Without it every (sequence, KV head) gets
 * the same number of CTAs.  The size query returns 0 where the chosen kernel
 * takes none.  The contents need no initialisation and are scratch between
 * calls; one workspace serves calls in stream order but not concurrent
 * calls.  A workspace that is too small is an error (PF_ERR_WORKSPACE);
 * for shapes that do not use it, it is ignored. */
PF_API size_t pf_verify_attention_workspace_size(const pf_attn_desc* d);

/* Kernels one pf_verify_attention(d) call launches (1 or 2) for this
 * descriptor as it stands (workspace given or not); 0 if the call would be
 * rejected.  Host-only: no device work, the last error is left alone. */
PF_API int32_t pf_verify_attention_launches(const pf_attn_desc* d);

/* pf_verify_attention_team_plan -- the team plan that PF_ATTN_KERNEL_TWO_BLOCK
 * makes from host copies of the lengths (see host_cu_nodes above), for
 * inspection and host-side tests.  Host-only: no device work, the last error
 * is left alone.
 *   cu_nodes[batch + 1], prefix_len[batch]   host arrays, read only
 *   n_kv_heads, group (query heads per KV head, 1..128), max_nodes,
 *   max_prefix_len     as in pf_attn_desc (bf16, head_dim 128)
 *   num_sms            SMs the launch may use (>= 1)
 *   max_clusters       [17] or NULL: max_clusters[s] = how many clusters of s
 *                      CTAs of the kernel fit on the GPU at once (NULL: the
 *                      current device's figures, which needs a GPU)
 *   uniform_splits     CTAs per group of the one-group clusters to beat
 *   entries            [PF_TEAM_MAX_CTAS] out, one word per CTA: group |
 *                      piece << 12 | pieces << 17 | rank of the team's first
 *                      CTA in its cluster << 22 (pieces = 0: no work), group =
 *                      (sequence * n_kv_heads + KV head) * pairs + pair of
 *                      row blocks, pairs = ceil(max_nodes / (2 * floor(128 /
 *                      group)))
 *   cluster_size, ctas, tiles_per_cta   out: CTAs per cluster, CTAs of the
 *                      launch (a multiple of it), the longest piece in tiles
 * Returns 1 with the plan written, 0 where no team plan beats the one-group
 * clusters or the lengths contradict the bounds, -1 for a NULL pointer or a
 * size out of range. */
#define PF_TEAM_MAX_CTAS 160
PF_API int32_t pf_verify_attention_team_plan(const int32_t* cu_nodes,
                                             const int32_t* prefix_len, int32_t batch,
                                             int32_t n_kv_heads, int32_t group,
                                             int32_t max_nodes, int32_t max_prefix_len,
                                             int32_t num_sms, const int32_t* max_clusters,
                                             int32_t uniform_splits, uint32_t* entries,
                                             int32_t* cluster_size, int32_t* ctas,
                                             int32_t* tiles_per_cta);

PF_API pf_status pf_verify_attention(const pf_attn_desc* d, void* stream);

/*
 * pf_lmhead_accept -- LM head, greedy prediction and acceptance
 * (Section 3.2: predictions at every proposed position and one more; accept
 * the longest matching proposal prefix; append the model's prediction).
 *   logits[t, v] = sum_c hidden[t, c] * W[v, c]   (fp32 accumulation)
 *   argmax[t]    = argmax_v logits[t, v], ties -> lowest v
 * then, per sequence b, descend from the root: at node u the prediction is
 * argmax[u]; move to the lowest-index child of u whose token equals it, or
 * stop.  Outputs for sequence b (path length a+1, a = accept_len[b]):
 *   path[b][0..a]        local node indices, path[b][0] = 0
 *   out_tokens[b][0..a]  tokens of path[1..a], then the bonus argmax[path[a]]
 *   last_node[b]         path[b][a] (its state is the next retrieval query)
 * Rows of path/out_tokens have stride max_nodes.
 * Layouts: hidden [T][H], weight [V][H] (row-major, H % 8 == 0), tokens and
 * parent [T] (parent local to its sequence, -1 at each root).
 * T <= PF_MAX_LM_ROWS.  dtype PF_BF16 (tensor cores) or PF_F32.
 * Workspace: device memory of pf_lmhead_accept_workspace_size() bytes,
 * zero-filled before its first use; every call leaves it zero-filled again,
 * so one workspace serves calls in stream order but not concurrent calls.
 */
typedef struct pf_lm_desc {
  int32_t dtype;               /* pf_dtype of hidden and weight              */
  int32_t batch;               /* B >= 1                                     */
  int32_t hidden;              /* H                                          */
  int32_t vocab;               /* V                                          */
  int32_t total_nodes;         /* T = cu_nodes[B]                            */
  int32_t max_nodes;           /* bound on nodes per sequence; row stride    */
  const int32_t* cu_nodes;     /* device [B+1]                               */
  const void* hidden_states;   /* device [T][H]                              */
  const void* weight;          /* device [V][H]                              */
  const int32_t* tokens;       /* device [T]                                 */
  const int32_t* parent;       /* device [T]                                 */
  int32_t* argmax;             /* out device [T]                             */
  float* max_logit;            /* out device [T], optional                   */
  int32_t* accept_len;         /* out device [B]                             */
  int32_t* path;               /* out device [B][max_nodes]                  */
  int32_t* out_tokens;         /* out device [B][max_nodes]                  */
  int32_t* last_node;          /* out device [B], optional                   */
  int32_t* error_flag;         /* optional device int32                      */
  int32_t flags;               /* PF_LM_* bits, 0 = none                     */
  int32_t stages;              /* bf16 weight-tile pipeline depth: 0 = the
                                  library's choice, else 2..16 (at most 12
                                  are used, fewer if shared memory is short) */
} pf_lm_desc;

/* PF_LM_EARLY_WEIGHT: the weight was written before the kernel that precedes
 * this call in the stream started (model weights normally are).  The kernel
 * then starts streaming its first weight tiles before waiting for that
 * preceding kernel to finish (programmatic dependent launch); the hidden
 * states, tokens and tree are read only after it finishes. */
#define PF_LM_EARLY_WEIGHT 1
/* PF_LM_NO_PDL: launch without programmatic dependent launch. */
#define PF_LM_NO_PDL 2

PF_API size_t pf_lmhead_accept_workspace_size(const pf_lm_desc* d);
PF_API pf_status pf_lmhead_accept(const pf_lm_desc* d, void* workspace, size_t workspace_bytes,
                           void* stream);

/*
 * pf_lmhead_accept_noalloc -- pf_lmhead_accept without a workspace argument.
 * The paper has no counterpart: this exists for callers that cannot
 * allocate device memory where they verify -- plug-ins whose host framework
 * owns every device allocation, and decode loops that must never reach an
 * allocator (allocating can synchronise the device or fail under memory
 * pressure).  The scratch lives in a file-scope device array of 2112 bytes
 * (room for PF_MAX_LM_ROWS = 256 proposal rows) that every GPU loading this
 * library holds until exit; total_nodes above 256 is rejected with
 * PF_ERR_SHAPE.  The first call on each device looks up that array's device
 * address (cudaGetSymbolAddress) and keeps it for the life of the process,
 * so make the first call on a device before any stream capture, and make no
 * call after cudaDeviceReset (the reset discards the array the kept address
 * points to).  Every call checks its arguments, then clears the array
 * (cudaMemsetAsync on the given stream) and runs exactly pf_lmhead_accept;
 * a rejected call queues nothing, and nothing is allocated or freed.  All
 * calls share the one array, so calls that overlap on the GPU (other
 * streams, other host threads) race: serialise them.  Same outputs and
 * errors as pf_lmhead_accept otherwise.
 */
PF_API pf_status pf_lmhead_accept_noalloc(const pf_lm_desc* d, void* stream);

/*
 * pf_kv_commit -- carry the accepted rows forward (Section 1 and Section
 * 3.4: accepted positions keep their K/V; Section 4: one contiguous cache).
 * For every layer l, K and V, sequence b and k = 0..accept_len[b]:
 *   cache_l[b, g, prefix_len[b] + k, :] = tree_l[cu_nodes[b] + path[b][k], g, :]
 * and new_len[b] = prefix_len[b] + accept_len[b] + 1.  Rejected proposal rows
 * are not copied.  accept_len and path are read from device memory (the
 * outputs of pf_lmhead_accept), so no host synchronisation is needed.
 * Layer l of the tree K/V starts at tree_k + l * tree_layer_stride elements
 * ([T][Hkv][D] per layer); layer l of the cache at cache.k + l *
 * cache_layer_stride elements (the pf_kv_view layout per layer).  The host
 * checks max_prefix_len + max_nodes fits the cache; the kernel re-checks
 * every row and sets PF_DEVERR_CAPACITY instead of writing outside it.
 * new_len must not alias prefix_len.  The copy is bit-exact.
 */
typedef struct pf_commit_desc {
  int32_t dtype;               /* pf_dtype (element size only)               */
  int32_t batch;               /* B                                          */
  int32_t n_layers;            /* L                                          */
  int32_t n_kv_heads;          /* Hkv                                        */
  int32_t head_dim;            /* D; D * element size must be a multiple of 16 */
  int32_t total_nodes;         /* T                                          */
  int32_t max_nodes;           /* bound on nodes per sequence; path row stride */
  int32_t max_prefix_len;      /* bound on every prefix_len[b]               */
  const int32_t* cu_nodes;     /* device [B+1]                               */
  const int32_t* prefix_len;   /* device [B]                                 */
  const int32_t* accept_len;   /* device [B]                                 */
  const int32_t* path;         /* device [B][max_nodes]                      */
  const void* tree_k;          /* device [L][T][Hkv][D] (see stride)         */
  const void* tree_v;
  int64_t tree_layer_stride;   /* elements between layers of tree_k/v        */
  pf_kv_view cache;            /* layer 0's view; k and v advance per layer  */
  int64_t cache_layer_stride;  /* elements between layers of cache.k/v       */
  int32_t* new_len;            /* out device [B]                             */
  int32_t* error_flag;         /* optional device int32                      */
} pf_commit_desc;

PF_API pf_status pf_kv_commit(const pf_commit_desc* d, void* stream);

/*
 * pf_kv_shift -- rolling-image KV carryover (Section 3.4): when the window
 * of retained screenshots advances, a retained visual-token block moves to
 * a new span of the prompt.  For every layer and KV head of sequence `seq`:
 *   K[dst + j] = R(dst + j) R(src + j)^-1 K[src + j]   (rotary re-rotation)
 *   V[dst + j] = V[src + j]                             j = 0 .. count-1
 * R is the rotary embedding in the rotate-half layout: the pair
 * (x_i, x_{i+D/2}) turns by position * rope_base^(-2i/D); for multi-axis
 * rotary embeddings every axis moves by the same shift, so the same
 * rotation applies.  The move is in place: source and destination spans may
 * overlap (rows are staged in the right order), and rows of the source span
 * outside the destination keep their contents.  The rotation angles are
 * formed on the host in double precision.  Layout as pf_kv_view (layer l at
 * cache.k/v + l * cache_layer_stride elements); D even, D * element size a
 * multiple of 16.  The host checks both spans fit the cache; the kernel
 * flags PF_DEVERR_CAPACITY for a page-table entry outside the pool.
 */
typedef struct pf_shift_desc {
  int32_t dtype;               /* pf_dtype                                   */
  int32_t n_layers;            /* L                                          */
  int32_t n_kv_heads;          /* Hkv                                        */
  int32_t head_dim;            /* D                                          */
  int32_t seq;                 /* sequence of the cache to move within       */
  int32_t batch;               /* sequences (page-table rows when paged)     */
  int32_t src;                 /* first source position                      */
  int32_t dst;                 /* first destination position                 */
  int32_t count;               /* rows to move (>= 0)                        */
  float rope_base;             /* rotary base, e.g. 10000 or 1e6             */
  pf_kv_view cache;            /* layer 0's view                             */
  int64_t cache_layer_stride;  /* elements between layers                    */
  int32_t* error_flag;         /* optional device int32                      */
} pf_shift_desc;

PF_API pf_status pf_kv_shift(const pf_shift_desc* d, void* stream);

/*
 * pf_retrieval_key -- the int8 retrieval key of a final-layer state
 * (Section 4 "Memory and retrieval": normalised final-layer states mapped
 * to 256-dimensional int8 keys by a fixed random projection).
 *   z = P h / |h|,  key = round_half_even(127 * z / max_i |z_i|)
 * (the per-vector scale keeps every key at full int8 range; cosine
 * similarity is scale invariant).  hidden_state [H] and projection [256][H]
 * in dtype; key_out [256] int8.  Workspace: pf_retrieval_workspace_size()
 * bytes, zero-filled before first use and left zero-filled.
 */
typedef struct pf_key_desc {
  int32_t dtype;               /* pf_dtype of hidden_state and projection    */
  int32_t hidden;              /* H                                          */
  const void* hidden_state;    /* device [H]                                 */
  const void* projection;      /* device [256][H]                            */
  int8_t* key_out;             /* out device [256]                           */
  int32_t* error_flag;         /* optional device int32                      */
} pf_key_desc;

#define PF_KEY_DIM 256

/*
 * pf_retrieve -- context-compatible retrieval (Section 3.2): among the
 * stored entries j in [lo, hi) whose token equals `token` and whose
 * position is before its output boundary (entry_pos[j] < entry_bound[j]),
 * the entry whose int8 key has the highest cosine similarity with
 * query_key.  The comparison is exact (integer dot products and squared
 * norms compared in 128-bit arithmetic); ties go to the lowest index;
 * all-zero keys are never selected.  keys, query_key and the three entry
 * arrays must be 16-byte aligned.  Outputs: best[0] = index or -1,
 * similarity[0] = its cosine (fp32, relative error below 3e-7).  keys [n_entries][256] int8;
 * entry_token, entry_pos, entry_bound [n_entries] int32.  Workspace:
 * pf_retrieval_workspace_size() bytes, zero-filled before first use and
 * left zero-filled; calls sharing a workspace must not overlap.
 */
typedef struct pf_retrieval_desc {
  int32_t n_entries;           /* M                                          */
  int32_t lo;                  /* first entry scanned                        */
  int32_t hi;                  /* one past the last entry scanned            */
  int32_t token;               /* the query's current token                  */
  const int8_t* query_key;     /* device [256]                               */
  const int8_t* keys;          /* device [M][256]                            */
  const int32_t* entry_token;  /* device [M]                                 */
  const int32_t* entry_pos;    /* device [M]                                 */
  const int32_t* entry_bound;  /* device [M]                                 */
  int32_t* best;               /* out device [1]                             */
  float* similarity;           /* out device [1]                             */
  int32_t* error_flag;         /* optional device int32                      */
} pf_retrieval_desc;

PF_API size_t pf_retrieval_workspace_size(void);
PF_API pf_status pf_retrieval_key(const pf_key_desc* d, void* workspace, size_t workspace_bytes,
                                  void* stream);
PF_API pf_status pf_retrieve(const pf_retrieval_desc* d, void* workspace, size_t workspace_bytes,
                             void* stream);

/*
 * pf_prefix_match -- prompt-prefix KV carryover (Section 3.4 "Prompt-prefix
 * KV-state carryover"): p = the length of the longest identical prefix of
 * the prompt whose K/V is cached (prev) and the new prompt (next).  Cached
 * rows 0 .. p-1 stay valid; computation resumes at position p.  Prompts are
 * int32 token keys: text tokens are their ids, image tokens an identifier of
 * the image content at that position, so that "identical" covers content.
 * Outputs (device): lcp[0] = p and, if cache_len is not NULL, cache_len[0]
 * = p (the cache's new length; rows >= p are stale).  n_prev and n_next are
 * in [0, 2^30]; prev / next may be NULL only when their length is 0.
 * 16-byte aligned arrays are read with vector loads.  One launch, no
 * workspace, no host synchronisation.
 */
typedef struct pf_prefix_desc {
  const int32_t* prev;         /* device [n_prev] keys of the cached prompt  */
  int32_t n_prev;
  const int32_t* next;         /* device [n_next] keys of the new prompt     */
  int32_t n_next;
  int32_t* lcp;                /* out device [1]                             */
  int32_t* cache_len;          /* optional out device [1]                    */
} pf_prefix_desc;

PF_API pf_status pf_prefix_match(const pf_prefix_desc* d, void* stream);

/*
 * pf_selftest_wait -- exercises the failure path shared by every kernel's
 * waits (no counterpart in the paper).  One GPU thread waits on an
 * mbarrier with the library's bounded wait, limited to limit_ns (1e3 ..
 * 5e9).  signal = 0: nothing arrives, so the wait runs out, ORs
 * PF_DEVERR_TIMEOUT into *error_flag and the kernel returns normally (the
 * context stays usable); signal = 1: the barrier completes at once.
 * waited_ok (device int32) receives 1 if the wait completed, else 0.
 */
PF_API pf_status pf_selftest_wait(int32_t* error_flag, int64_t limit_ns, int32_t signal,
                                  int32_t* waited_ok, void* stream);

/*
 * Proposal-length controller (Section 3.2 "Runtime-adaptive
 * proposal-length controller", eq. 1).  Host code: no GPU, no allocation.
 *
 *   L* = argmin_{0 <= l <= l_max}  T(l) / (A(l, s) + 1),
 *   A(l, s) = sum_{k=1..l} p1 * pc^(k-1)
 *
 * p1 (first proposal token accepted) and pc (token k accepted given token
 * k-1 was) come from two online logistic regressions on x = (1, l/l_max,
 * s); one observation (l, s, a accepted tokens) is one first-token trial
 * (success iff a >= 1) and, if a >= 1, the continuation trials k = 2 ..
 * min(a+1, l) (success iff k <= a), each a gradient step
 * w += lr (y - sigmoid(w.x)) x.  T(l) = exp(c0 + c1 u + c2 u^2), u =
 * l / l_max, is fitted to observed iteration latencies by recursive least
 * squares from a zero prior of variance 1e8.  Ties go to the shorter length.  Exploration: with
 * the caller's uniform draw u < epsilon the choice moves to an adjacent
 * length (up unless at l_max, or down when u_dir >= 0.5 and above 0).
 */
typedef struct pf_length_controller {
  int32_t l_max;
  int32_t n_latency;   /* latency observations so far                      */
  double lr;           /* logistic-regression step size                    */
  double epsilon;      /* exploration rate                                 */
  double w_first[3];
  double w_cont[3];
  double c[3];         /* log-latency coefficients                         */
  double P[9];         /* recursive-least-squares covariance, row-major    */
} pf_length_controller;

#define PF_CTL_MAX_LEN 4096

/* l_max in [1, PF_CTL_MAX_LEN], lr > 0, epsilon in [0, 1]. */
PF_API pf_status pf_controller_init(pf_length_controller* c, int32_t l_max, double lr,
                                    double epsilon);
/* One decoding iteration's outcome: ell in [0, l_max], similarity s,
 * accepted in [0, ell] (or < 0: no acceptance observation), latency_us > 0
 * (or <= 0: no latency observation). */
PF_API pf_status pf_controller_observe(pf_length_controller* c, int32_t ell, double similarity,
                                       int32_t accepted, double latency_us);
/* The next length for similarity s; u, u_dir are the caller's uniform
 * draws in [0, 1) for exploration.  objective_out may be NULL. */
PF_API pf_status pf_controller_choose(const pf_length_controller* c, double similarity, double u,
                                      double u_dir, int32_t* ell_out, double* objective_out);
/* Eq. 1 over explicit estimates t_hat[l], p_first[l], p_cont[l], l = 0..l_max. */
PF_API pf_status pf_length_select(const double* t_hat, const double* p_first,
                                  const double* p_cont, int32_t l_max, int32_t* ell_out,
                                  double* objective_out);

#ifdef __cplusplus
}
#endif

#endif /* PF_VERIFY_H */
