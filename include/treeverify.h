/*
 * treeverify.h -- C ABI of the GB300 tree-verification library.
 *
 * One decode step of Medusa/Hydra multi-token-prediction decoding verifies a
 * draft tree of N <= 64 candidate tokens in one target-model pass: tree-masked
 * attention over the KV cache, the LM head with the greedy token, top-1
 * probability and entropy per node, greedy acceptance of the longest root path
 * whose drafts the target agrees with, and the KV-cache update that keeps the
 * accepted path (EntMTP, Sec. 3.2: proposal -> tree decoding -> verification ->
 * KV-cache update).  Trees live in a TopologyBank of precompiled topologies so
 * that switching trees between steps is an O(1) pointer swap (Sec. 1 and
 * Sec. 4, "Cost").
 *
 * Conventions that hold for every entry point:
 *  - Device pointers are owned by the caller.  The library allocates device
 *    memory only in tb_create (the bank); no other call allocates.
 *  - Calls that take a stream only enqueue work on it and return without
 *    synchronising.  Host-side argument errors are returned before anything is
 *    enqueued.  Errors that only the GPU can detect are reported in the
 *    workspace status word (tb_workspace_status) and, for verify_step and
 *    greedy_accept, in tb_result.status.
 *  - bf16 tensors are IEEE bfloat16 bit patterns.  All device buffers must be
 *    16-byte aligned.
 *  - Errors are negative tb_status codes; tb_last_error() returns a message
 *    for the last failing call on the calling thread.  No C++ exception
 *    crosses this interface.
 */
#ifndef TREEVERIFY_H
#define TREEVERIFY_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#if defined(__GNUC__)
#define TB_API __attribute__((visibility("default")))
#else
#define TB_API
#endif

#define TB_MAX_NODES 64 /* nodes per draft tree, root included */
#define TB_MAX_BATCH 16 /* sequences per verify_step_batched call */

typedef enum {
    TB_OK = 0,
    TB_EINVAL = -1,      /* bad argument (pointer, size, stride, alignment, tree) */
    TB_ENOMEM = -2,      /* device allocation failed (tb_create only) */
    TB_ECUDA = -3,       /* a CUDA runtime or driver call failed */
    TB_ENOTFOUND = -4,   /* bank_id does not name a topology */
    TB_ECAPACITY = -5,   /* bank full, workspace too small, or L + N > L_cap */
    TB_ETIMEOUT = -6,    /* a bounded device-side wait expired (kernel gave up) */
    TB_EUNSUPPORTED = -7 /* shape outside what the kernels implement */
} tb_status;

/* Same type as cudaStream_t; NULL is the legacy default stream. */
typedef struct CUstream_st *tb_stream;

/* Opaque TopologyBank: the precompiled draft trees of one device. */
typedef struct tb_bank tb_bank;

/* ------------------------------------------------------------------------
 * Topologies (Sec. 2.3: draft trees with precomputed attention masks,
 * position offsets and gather indices; Sec. 4 "Cost": per-tree buffers, so a
 * switch is a pointer swap with no GPU work).
 * ---------------------------------------------------------------------- */

/* Pure host.  Validates parent[0..n) as a tree rooted at node 0 (parent[0] ==
 * -1, every other parent in [0, n), no cycle) and returns it in canonical
 * breadth-first order: children of a node in increasing original index.
 *   order[c]      original index of canonical node c          (may be NULL)
 *   bfs_parent[c] canonical parent (-1 for the root)          (may be NULL)
 *   depth[c]      edges from the root = position offset        (may be NULL)
 *   anc[c]        bit j set iff canonical node j is c or an ancestor of c
 *                 (the tree attention mask row of c)          (may be NULL)
 * In canonical order parent < child and depth is non-decreasing.
 * Returns TB_EINVAL for 1 > n > 64 or a parent array that is not such a tree. */
TB_API tb_status tb_canonicalize(const int32_t *parent, int n, int32_t *order, int32_t *bfs_parent,
                          int32_t *depth, uint64_t *anc);

/* Creates an empty bank of max_topologies (1..4096) trees on CUDA device
 * `device` and allocates its device table.  Synchronous. */
TB_API tb_status tb_create(tb_bank **out, int max_topologies, int device);

/* Canonicalises parent[0..n) (host array, see tb_canonicalize), uploads the
 * ancestor bitsets, depths and parents once (synchronous copy), and returns
 * its id (0, 1, ... in insertion order).  `order` (n entries, may be NULL)
 * receives the canonical -> caller index map: draft tokens, queries and tree
 * K/V slots are passed in canonical order.  TB_ECAPACITY when the bank is full. */
TB_API tb_status tb_add_topology(tb_bank *bank, const int32_t *parent, int n, int *out_id, int32_t *order);

/* Host copy of a stored topology (canonical order).  Any output may be NULL;
 * parent/depth/anc need room for *n entries (at most 64). */
TB_API tb_status tb_get_topology(const tb_bank *bank, int id, int *n, int32_t *parent, int32_t *depth,
                          uint64_t *anc);

/* Frees the bank's device table.  Work already enqueued that uses the bank
 * must have completed.  NULL is accepted. */
TB_API tb_status tb_destroy(tb_bank *bank);

/* ------------------------------------------------------------------------
 * KV cache and results
 * ---------------------------------------------------------------------- */

/* The caller's bf16 KV cache.  Element (layer, kv head g, slot s, c) of K is at
 * k + layer * layer_stride + g * head_stride + s * head_dim + c, likewise V.
 * Slots [0, L) hold the prefix; the N tree nodes of the step occupy slots
 * [L, L + N) in canonical node order (the keys/values of the draft tokens,
 * produced by the model's K/V projection before the call).  Strides are in
 * elements and must be multiples of 8; head_dim is 64 or 128.
 *
 * rope_theta = 0: the queries and every key are already rotary-embedded.
 * rope_theta > 0: the calls apply the base model's rotary
 * embedding (Llama convention: frequencies rope_theta^(-2i/d), element i
 * paired with element i + d/2) at the tree's position offsets, node i at
 * position L + depth(i): the queries are passed pre-rotary, and the tree
 * slots [L, L + N) of K hold pre-rotary keys when the call starts; the call
 * rotates them in place (the cache then holds rotated keys, as for the
 * prefix, and the accepted ones keep their positions after compaction: path
 * index i has depth i).  A second call on the same tree slots would rotate
 * them again. */
typedef struct tb_kv {
    void *k;
    void *v;
    int64_t layer_stride;
    int64_t head_stride;
    int32_t n_layers;
    int32_t n_kv_heads;
    int32_t head_dim;
    int32_t L;          /* prefix length of this step */
    int32_t L_cap;      /* slots per head: L + N <= L_cap */
    float rope_theta;   /* 0, or the rotary base (e.g. 10000) applied by the call */
} tb_kv;

/* Device-resident result of one verification, written by the GPU. */
typedef struct tb_result {
    int32_t accept_len;  /* accepted tokens incl. the bonus token: depth(j*) + 1 */
    int32_t bonus_token; /* target greedy token after the last accepted node */
    int32_t new_L;       /* L + accept_len: the prefix length for the next step */
    int32_t status;      /* TB_OK or a device-detected tb_status */
    int32_t path[TB_MAX_NODES]; /* path[0 .. accept_len) = root .. j*, canonical ids */
} tb_result;

/* ------------------------------------------------------------------------
 * Workspace: scratch for split-L attention partials, LM-head partials and
 * arrival counters.  Caller-allocated device memory; must be zero-filled
 * before its first use (tb_workspace_init) and again after any call that
 * reported TB_ETIMEOUT.  Kernels leave their counters at zero on success.
 * One workspace must not be used by two calls that can run concurrently.
 * ---------------------------------------------------------------------- */

/* Bytes of workspace for calls with up to max_rows LM-head rows and up to
 * n_layers x n_kv_heads attention heads of head_dim, vocab entries, on device
 * `device` (the grid size depends on its SM count). */
TB_API size_t tb_workspace_size(int max_rows, int n_layers, int n_kv_heads, int n_q_heads, int head_dim,
                         int vocab, int device);

/* Zero-fills the workspace on `stream` (asynchronous). */
TB_API tb_status tb_workspace_init(void *workspace, size_t workspace_bytes, tb_stream stream);

/* Synchronously reads the workspace status word: TB_OK or the first
 * device-detected error (TB_ETIMEOUT, TB_EINVAL). */
TB_API tb_status tb_workspace_status(const void *workspace, int32_t *status);

/* Test support for the debug build of the library (compiled with
 * TB_DEBUG_BOUNDS; the paper has no counterpart).  In that build every kernel
 * checks its global-memory indices against the extents it was given; a failed
 * check skips the access, raises an error bit in the workspace status word
 * (reported as TB_EINVAL by tb_workspace_status and in tb_result.status) and
 * is counted.  tb_debug_bounds_violations synchronises the device, stores the
 * number of failed checks since its previous call in *count and resets it
 * (always 0 in a normal build).  tb_debug_bounds_build returns 1 in the debug
 * build, 0 otherwise. */
TB_API tb_status tb_debug_bounds_violations(uint32_t *count);
TB_API int tb_debug_bounds_build(void);

/* Instrumentation (the paper has no counterpart): stores in *count the number
 * of kernels the library has enqueued in this process so far, counted on the
 * host as each launch is accepted.  Kernels that a CUDA graph replays are not
 * counted again: a graph holds the kernels counted while it was captured.
 * TB_EINVAL if count is NULL; never touches the device. */
TB_API tb_status tb_launch_count(uint64_t *count);

/* ------------------------------------------------------------------------
 * The verification pass and its stages
 * ---------------------------------------------------------------------- */

/* Tree-masked attention (tree decoding, Sec. 3.2; mask = ancestor bitsets,
 * Sec. 2.3) for layers [layer_begin, layer_begin + n_layers) of kv:
 *   O[i, h] = sum_s softmax_s(q[i, h] . k[s, g] / sqrt(head_dim)) v[s, g]
 * over s in [0, L) and the tree slots L + j of the ancestors-or-self j of node
 * i; g = h / (n_q_heads / n_kv_heads).
 *   q   bf16 [n_layers][N][n_q_heads][head_dim] (post-rotary), read only
 *   out bf16 [n_layers][N][n_q_heads][head_dim]
 * N is the topology's node count.  n_q_heads must be a multiple of
 * n_kv_heads, N * (n_q_heads / n_kv_heads) <= 256. */
TB_API tb_status tree_attention(const tb_bank *bank, int bank_id, const tb_kv *kv, int layer_begin,
                         int n_layers, const void *q, int n_q_heads, void *out, void *workspace,
                         size_t workspace_bytes, tb_stream stream);

/* Fused LM head: z_r = W h_r for every row, never written to memory; per row
 * the greedy token argmax_v z (lowest index on ties), the top-1 probability
 * max softmax(z) (the base-LM p0 of Sec. 4) and the entropy -sum p ln p in
 * nats (the entropy feature of the scheduler, Sec. 4 / App. A).
 *   hidden bf16 [n_rows][d_model]; lm_head bf16 [vocab][d_model] (nn.Linear)
 *   argmax int32 [n_rows]; top1, entropy float [n_rows]
 * 1 <= n_rows <= 256, d_model a multiple of 8, vocab >= 1.
 * Two kernels: the LM head proper, which writes per-row statistics of every
 * vocab tile into the workspace, then their merge in a fixed order; the
 * outputs are bitwise reproducible for the same inputs, whatever the launch
 * placement. */
TB_API tb_status lm_head_stats(const void *hidden, int n_rows, const void *lm_head, int d_model, int vocab,
                        int32_t *argmax, float *top1, float *entropy, void *workspace,
                        size_t workspace_bytes, tb_stream stream);

/* Greedy acceptance (verification, Sec. 3.2, greedy form): node i is accepted
 * when every non-root node j on its root path has draft_tokens[j] ==
 * argmax[parent(j)]; j* is the deepest accepted node (smallest canonical id
 * among equally deep ones).  Writes accept_len, path, bonus_token =
 * argmax[j*], new_L = L + accept_len and status into *result.  A draft token
 * outside [0, vocab) never matches and sets status TB_EINVAL.
 * draft_tokens, argmax: device int32 [N]; draft_tokens[0] is ignored. */
TB_API tb_status greedy_accept(const tb_bank *bank, int bank_id, const int32_t *draft_tokens,
                        const int32_t *argmax, int vocab, int L, tb_result *result,
                        tb_stream stream);

/* KV-cache update after acceptance (Sec. 3.2): for every layer and kv head of
 * kv, slot L + j receives the K and V of slot L + path[j], j < accept_len.
 * path: device int32 [accept_len], canonical node ids from the root, each at
 * least its position (path[j] >= j, as every root path of a canonical tree
 * is); accept_len: device int32, clamped to 1..TB_MAX_NODES; both are read on
 * the device, so they may come from a kernel earlier on `stream` -- for the
 * result of greedy_accept: path = result->path, accept_len =
 * &result->accept_len.  In place; all other slots are untouched, and so is
 * slot L + j when path[j] <= j or L + path[j] >= L_cap.  TB_EINVAL for a NULL
 * pointer or a bad kv. */
TB_API tb_status kv_compact(const tb_kv *kv, const int32_t *path, const int32_t *accept_len, tb_stream stream);

#define TB_NO_COMPACT 1 /* verify_step flag: skip the KV-cache update */
/* verify_step test hook for failure detection: the LM-head kernel waits on a
 * barrier that nothing arrives on, so its bounded wait (about one second)
 * expires; the kernel then stops cleanly (in-flight copies land, issued MMAs
 * retire, TMEM is freed), the step reports TB_ETIMEOUT in tb_result.status
 * and in the workspace status word, and argmax/top1/entropy are not written.
 * The workspace must be re-initialised (tb_workspace_init) afterwards. */
#define TB_DEBUG_EXPIRE_WAIT (1 << 30)

/* One full verification step of topology bank_id: tree_attention over all
 * kv->n_layers layers, lm_head_stats over the N node rows, greedy_accept, and
 * (unless TB_NO_COMPACT) kv_compact, enqueued on `stream` in that order.
 *   hidden bf16 [N][d_model] (final hidden state of each node)
 *   attn_out bf16 [n_layers][N][n_q_heads][head_dim]
 *   argmax int32 / top1, entropy float [N]; result: device tb_result. */
TB_API tb_status verify_step(const tb_bank *bank, int bank_id, const tb_kv *kv, const void *q,
                      int n_q_heads, const void *hidden, const void *lm_head, int d_model,
                      int vocab, const int32_t *draft_tokens, void *attn_out, int32_t *argmax,
                      float *top1, float *entropy, tb_result *result, void *workspace,
                      size_t workspace_bytes, int flags, tb_stream stream);

/* ------------------------------------------------------------------------
 * Per-step tree selection (Sec. 4, "Policy"): which bank entry the next step
 * verifies.  Pure host functions, O(1); switching is then the bank_id passed
 * to the next verify_step (no GPU work).
 * ---------------------------------------------------------------------- */

/* Hysteretic step ladder over trees 0..n_trees-1 ordered from smallest to
 * largest, driven by a feature that is LOW when the continuation is
 * predictable (the entropy of the verifier's distribution, nats): move one
 * tree up when feature < up_below, one tree down when feature > down_above,
 * otherwise stay (up_below <= down_above gives a dead band against flapping).
 * Returns the next index, clamped to [0, n_trees). */
TB_API int tb_schedule_hysteretic_ladder(int current, int n_trees, double feature, double up_below,
                                         double down_above);

/* The paper's binary hysteretic rule on the path-value score s (HIGH when
 * deep drafts are likely): switch to the aggressive tree when s > tau_on,
 * back to the conservative tree when s <= tau_off, tau_off <= tau_on.
 * `aggressive` is 1 when the current tree is the aggressive one; returns the
 * new value. */
TB_API int tb_schedule_binary(int aggressive, double s, double tau_on, double tau_off);

/* threshold_ladder: the index of the interval of s among n_trees - 1
 * ascending edges (s < edges[0] -> 0, ..., s >= edges[n_trees-2] -> n_trees-1). */
TB_API int tb_schedule_threshold_ladder(double s, const double *edges, int n_trees);

/* One sequence of a batched verification step. */
typedef struct tb_seq {
    int32_t bank_id;              /* its draft-tree topology */
    int32_t reserved;             /* 0 */
    tb_kv kv;                     /* its KV cache and prefix length (all sequences of a batch share
                                     n_layers, n_kv_heads and head_dim) */
    const void *q;                /* bf16 [kv.n_layers][N_b][n_q_heads][head_dim] */
    const int32_t *draft_tokens;  /* device int32 [N_b] */
    void *attn_out;               /* bf16 [kv.n_layers][N_b][n_q_heads][head_dim] */
    tb_result *result;            /* device */
} tb_seq;

/* verify_step for a batch of 1..TB_MAX_BATCH independent sequences, each with
 * its own topology, prefix length and KV cache (ragged batch).  The LM head
 * reads W once for the whole batch: hidden holds the rows of every sequence,
 * sequence 0 first (sum of N_b rows, at most 1024); argmax / top1 / entropy
 * follow the same row order.  Tree attention of every sequence runs in one
 * launch whose work is balanced over the GPU whatever the prefix lengths;
 * acceptance and compaction run in one launch.  `seqs` is a
 * host array; everything else is as for verify_step. */
TB_API tb_status verify_step_batched(const tb_bank *bank, int batch, const tb_seq *seqs, int n_q_heads,
                                     const void *hidden, const void *lm_head, int d_model, int vocab, int32_t *argmax,
                                     float *top1, float *entropy, void *workspace, size_t workspace_bytes, int flags,
                                     tb_stream stream);

/* lm_head_stats for callers that cannot allocate device memory.  Code that
 * runs inside a host framework which owns every device allocation, in a
 * sandbox that forbids cudaMalloc, or next to a memory pool that is already
 * fully carved up has no way to provide the workspace that lm_head_stats
 * needs.  This variant computes the same argmax / top1 / entropy with the
 * same kernel, but keeps its scratch in a 16 MiB array compiled into the
 * library (every GPU that loads the library holds it until the process
 * exits); it calls no cudaMalloc, cudaFree or allocating library routine.
 *  - Outside stream capture every call looks up that array's device address
 *    (cudaGetSymbolAddress) on the current device; while `stream` is being
 *    captured the address found by the last call on this device is used, so
 *    make one call outside capture first (and again after a cudaDeviceReset).
 *  - Every call clears the array's arrival counters and status word on
 *    `stream` and reuses the array, which keeps the previous call's partial
 *    results: calls that can overlap on the GPU (different streams without
 *    ordering) race.
 *  - The scratch is one partial per 128 vocabulary entries for every row
 *    (rows padded to 16, 24 bytes each): about vocab / 128 x 24 x padded
 *    rows bytes, 10 MiB at 256 rows and vocab 200000; a call that needs more
 *    than 16 MiB is rejected with TB_ECAPACITY before anything is enqueued.
 *  - A bounded device wait that runs out (TB_ETIMEOUT) leaves argmax / top1 /
 *    entropy unwritten and is visible only through
 *    lm_head_stats_noalloc_status.
 * flags: 0, or TB_DEBUG_EXPIRE_WAIT (test hook, as for verify_step).
 * Arguments, layouts, argument checks and tolerances are those of
 * lm_head_stats.  The paper has no counterpart: this is an integration
 * convenience of this library. */
TB_API tb_status lm_head_stats_noalloc(const void *hidden, int n_rows, const void *lm_head, int d_model, int vocab,
                                       int32_t *argmax, float *top1, float *entropy, int flags, tb_stream stream);

/* Device-detected status of the last lm_head_stats_noalloc call enqueued on
 * `stream`: waits for `stream`, then reads the built-in array's status word
 * into *status (TB_OK, or TB_ETIMEOUT when a bounded wait of that call ran
 * out).  Synchronous; allocates nothing.  The next lm_head_stats_noalloc call
 * clears the word. */
TB_API tb_status lm_head_stats_noalloc_status(int32_t *status, tb_stream stream);

/* ------------------------------------------------------------------------
 * Typical acceptance: the Medusa/Hydra verification rule that the paper keeps
 * unchanged and runs with T = 0.7, eps = 0.09, alpha = 0.3 (Sec. 5.1, 5.2).
 * ---------------------------------------------------------------------- */

/* Parameters of the rule (host struct, read at call time). */
typedef struct tb_typical {
    float temperature; /* T > 0: the target distribution is softmax(z / T) */
    float eps;         /* posterior threshold epsilon >= 0 */
    float alpha;       /* mixing coefficient alpha >= 0 */
    int32_t reserved;  /* 0 */
} tb_typical;

/* lm_head_stats over the N node rows of topology bank_id (canonical order)
 * plus, from the same pass over W, what typical acceptance consumes:
 *   logz_t[r]      = ln sum_v e^(z_r[v] / T)              (log-partition at T)
 *   entropy_t[r]   = -sum_v p ln p with p = softmax(z_r / T) (nats)
 *   draft_logit[j] = z_{parent(j)}[draft_tokens[j]] for every non-root node j
 *                    whose draft token lies in [0, vocab); other entries are
 *                    left unwritten.
 *   hidden bf16 [N][d_model]; draft_tokens device int32 [N];
 *   argmax int32, top1 / entropy / logz_t / entropy_t / draft_logit float,
 *   all device [N].  top1 and entropy stay at temperature 1. */
TB_API tb_status lm_head_stats_typical(const tb_bank *bank, int bank_id, const void *hidden, const void *lm_head,
                                       int d_model, int vocab, float temperature, const int32_t *draft_tokens,
                                       int32_t *argmax, float *top1, float *entropy, float *logz_t, float *entropy_t,
                                       float *draft_logit, void *workspace, size_t workspace_bytes, tb_stream stream);

/* Typical acceptance over topology bank_id: the edge into non-root node j
 * passes when
 *   p_j = e^(draft_logit[j] / T - logz_t[parent(j)]) > min(eps, alpha e^(-entropy_t[parent(j)])),
 * node i is accepted when every edge of its root path passes, and j* is the
 * deepest accepted node with the largest path log-likelihood sum ln p_j over
 * its edges (smallest canonical id on exact ties).  Writes *result as
 * greedy_accept does, bonus_token = argmax[j*]; a draft token outside
 * [0, vocab) never passes and sets status TB_EINVAL.  All arrays are device
 * [N] in canonical node order (the outputs of lm_head_stats_typical). */
TB_API tb_status typical_accept(const tb_bank *bank, int bank_id, const int32_t *draft_tokens,
                                const int32_t *argmax, const float *logz_t, const float *entropy_t,
                                const float *draft_logit, int vocab, int L, const tb_typical *params,
                                tb_result *result, tb_stream stream);

/* verify_step with typical acceptance: the LM-head pass also produces the
 * tempered statistics and draft logits (kept in the workspace) and the
 * acceptance follows typical_accept.  Arguments as for verify_step. */
TB_API tb_status verify_step_typical(const tb_bank *bank, int bank_id, const tb_kv *kv, const void *q,
                                     int n_q_heads, const void *hidden, const void *lm_head, int d_model, int vocab,
                                     const int32_t *draft_tokens, void *attn_out, int32_t *argmax, float *top1,
                                     float *entropy, const tb_typical *params, tb_result *result, void *workspace,
                                     size_t workspace_bytes, int flags, tb_stream stream);

/* verify_step_batched with typical acceptance (same parameters for every
 * sequence).  Arguments as for verify_step_batched. */
TB_API tb_status verify_step_batched_typical(const tb_bank *bank, int batch, const tb_seq *seqs, int n_q_heads,
                                             const void *hidden, const void *lm_head, int d_model, int vocab,
                                             int32_t *argmax, float *top1, float *entropy, const tb_typical *params,
                                             void *workspace, size_t workspace_bytes, int flags, tb_stream stream);

/* ------------------------------------------------------------------------
 * Speculative sampling: the stochastic verification rule of Sec. 2.1 (accept
 * a drafted token t with probability min(1, p(t) / q(t)); at the first
 * rejection draw the replacement from norm(max(0, p - q))), applied on the
 * tree: at every node the children are tried in increasing canonical id
 * order, the residual norm(max(0, r - q_u)) replacing the target r after each
 * rejected sibling; the walk stops at the node none of whose children is
 * accepted and the token after it is drawn from r by inverse CDF (the
 * smallest v with sum_{w <= v} r(w) > uniforms[N + u] * sum_w r(w)).  The
 * target at node u is p_u = softmax(z_u / T).  Lossless when the children of
 * each node u are independent draws from q_u.
 * ---------------------------------------------------------------------- */

/* The walk alone, from the target logits:
 *   draft_tokens int32 [N]; logits float [N][vocab]; logz_t float [N] =
 *   ln sum_v e^(z_v / T) (lm_head_stats_typical); draft_probs float [N][vocab]:
 *   row u = the distribution the children of u were drawn from (rows of
 *   leaves unused); uniforms float [2N] in [0, 1): uniforms[c] decides child
 *   c, uniforms[N + u] draws the token at the final node u; scratch float
 *   [vocab].  All device memory.  *result: accept_len, path, bonus_token = the
 *   drawn token, new_L = L + accept_len, status (a draft token outside
 *   [0, vocab) is never accepted and sets TB_EINVAL).  One cluster of 8 CTAs
 *   for vocab <= 131072 (scratch unused), else one CTA (scratch holds the
 *   residual). */
TB_API tb_status spec_sample_accept(const tb_bank *bank, int bank_id, const int32_t *draft_tokens, const float *logits,
                                    const float *logz_t, const float *draft_probs, const float *uniforms, int vocab,
                                    int L, float temperature, float *scratch, tb_result *result, tb_stream stream);

/* One verification step with speculative sampling: tree_attention, the LM
 * head (greedy statistics, tempered log-partition, and the logits of every
 * node written to logits[0 .. N) -- the sampling needs whole rows), the walk
 * (scratch: logits row N), then (unless TB_NO_COMPACT) kv_compact.
 *   logits float [N + 1][vocab] (device scratch written by the call);
 *   draft_probs, uniforms as for spec_sample_accept; the rest as verify_step. */
TB_API tb_status verify_step_sampled(const tb_bank *bank, int bank_id, const tb_kv *kv, const void *q,
                                     int n_q_heads, const void *hidden, const void *lm_head, int d_model, int vocab,
                                     const int32_t *draft_tokens, const float *draft_probs, const float *uniforms,
                                     float temperature, void *attn_out, int32_t *argmax, float *top1, float *entropy,
                                     float *logits, tb_result *result, void *workspace, size_t workspace_bytes,
                                     int flags, tb_stream stream);

/* ------------------------------------------------------------------------
 * Device-driven decode loop: the per-step tree selection of Sec. 4 ("Policy",
 * "Cost") taken on the GPU.  The prefix length and the tree of the next step
 * live in device memory (tb_state); the acceptance kernel's last CTA updates
 * them after each step, so consecutive verify_step_scheduled calls need no
 * host read in between and a sequence of them can be captured into one CUDA
 * graph.
 * ---------------------------------------------------------------------- */

/* Device-resident state (caller-allocated device memory, 4-byte aligned). */
typedef struct tb_state {
    int32_t rung;        /* index into tb_policy.bank_ids of the tree the next step verifies */
    int32_t L;           /* prefix length of the next step */
    int32_t step;        /* steps completed */
    float feature;       /* feature value of the last policy decision */
    int32_t accept_len;  /* accepted length of the last step */
    int32_t reserved[3];
} tb_state;

#define TB_POLICY_HYSTERETIC_LADDER 0 /* one rung up when feature < a, one down when feature > b */
#define TB_POLICY_BINARY 1            /* rung 1 when feature > a (tau_on), rung 0 when feature <= b (tau_off) */
#define TB_POLICY_THRESHOLD_LADDER 2  /* rung = number of edges[0..n_rungs-2] that are <= feature */

#define TB_FEATURE_TRACE 0      /* feature = trace[min(step, n_trace - 1)] (a per-step feature series) */
#define TB_FEATURE_PATH_VALUE 1 /* s = max(p0, g_1 .. g_D), g_d = p0 * prod_{i <= d} p_i: p0 = top1 of the last accepted
                                   node, p_i = trace[min(step, n_trace - 1) * n_heads + i - 1] (Sec. 4 "Path-value score") */
#define TB_FEATURE_ENTROPY 2    /* feature = entropy of the last accepted node (nats, temperature 1) */

/* Policy of the device-driven loop (host struct, read at call time). */
typedef struct tb_policy {
    int32_t kind;          /* TB_POLICY_* */
    int32_t feature;       /* TB_FEATURE_* */
    int32_t n_rungs;       /* 1..8 (TB_POLICY_BINARY: 2) */
    int32_t bank_ids[8];   /* the tree of each rung, smallest first */
    float a, b;            /* ladder: up_below, down_above; binary: tau_on, tau_off (b <= a) */
    float edges[7];        /* threshold ladder: n_rungs - 1 ascending edges */
    const float *trace;    /* device array for TB_FEATURE_TRACE / TB_FEATURE_PATH_VALUE, else NULL */
    int32_t n_trace;       /* entries (rows of n_heads for TB_FEATURE_PATH_VALUE), >= 1 when trace is used */
    int32_t n_heads;       /* head probabilities per row (TB_FEATURE_PATH_VALUE), 0..8 */
    int32_t node_stride;   /* nodes per layer / per draft row of the per-node arrays; 0: the largest tree of the
                              policy; otherwise at least that */
} tb_policy;

/* One verification step whose tree and prefix length come from *state:
 * tree = policy->bank_ids[state->rung], L = state->L (kv->L is ignored).
 * N_max is policy->node_stride (0: the largest node count among the policy's
 * trees); per-node arrays are laid out for N_max nodes and the step uses the
 * first N of them:
 *   q, attn_out   bf16 [kv->n_layers][N_max][n_q_heads][128]
 *   hidden        bf16 [N_max][d_model]
 *   draft_tokens  int32 [n_rungs][N_max]: row r holds the drafts of rung r's tree
 *   argmax/top1/entropy [N_max] (rows >= N are scratch)
 * After tree_attention, the LM head and greedy acceptance (+ compaction unless
 * TB_NO_COMPACT), the last CTA of the acceptance kernel evaluates the feature
 * and the policy and writes the next rung, L + accept_len, step + 1, the
 * feature and accept_len into *state; *result is written as by verify_step.
 * A state whose L + N exceeds kv->L_cap, or whose rung is out of range, makes
 * the step report TB_ECAPACITY / TB_EINVAL in result->status and leaves
 * *state unchanged. */
TB_API tb_status verify_step_scheduled(const tb_bank *bank, const tb_policy *policy, tb_state *state,
                                       const tb_kv *kv, const void *q, int n_q_heads, const void *hidden,
                                       const void *lm_head, int d_model, int vocab, const int32_t *draft_tokens,
                                       void *attn_out, int32_t *argmax, float *top1, float *entropy,
                                       tb_result *result, void *workspace, size_t workspace_bytes, int flags,
                                       tb_stream stream);

/* Message for the last failing call on this thread ("" if none). */
TB_API const char *tb_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* TREEVERIFY_H */
