// kernels.cuh -- host-side interface between the C-ABI layer and the kernels.
#pragma once

#include "common.cuh"

namespace tv {

// Counts one kernel enqueued by the library (tb_launch_count).
void count_launch();

// Launches `kernel` on `stream` in clusters of `cluster_x` CTAs (1: none);
// with pdl, with the programmatic-serialization attribute, so that it may be
// launched while the previous kernel of the stream still runs (the kernel
// waits for it with pdl_wait before touching memory it writes).
template <typename... KArgs, typename... Args>
cudaError_t launch_kernel_cluster(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                                  bool pdl, int cluster_x, Args &&...args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    int n = 0;
    if (pdl) {
        attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[n].val.programmaticStreamSerializationAllowed = 1;
        ++n;
    }
    if (cluster_x > 1) {
        attr[n].id = cudaLaunchAttributeClusterDimension;
        attr[n].val.clusterDim.x = (unsigned)cluster_x;
        attr[n].val.clusterDim.y = 1;
        attr[n].val.clusterDim.z = 1;
        ++n;
    }
    cfg.attrs = n ? attr : nullptr;
    cfg.numAttrs = n;
    const cudaError_t e = cudaLaunchKernelEx(&cfg, kernel, static_cast<Args &&>(args)...);
    if (e == cudaSuccess)
        count_launch();
    return e;
}

template <typename... KArgs, typename... Args>
cudaError_t launch_kernel(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream, bool pdl,
                          Args &&...args)
{
    return launch_kernel_cluster(kernel, grid, block, smem, stream, pdl, 1, static_cast<Args &&>(args)...);
}

// LM head (lm_head.cu)
struct LmPlan {
    int R_pad, n_tiles, n_kblocks, stages, acc_cols;
    int ctas_per_sm;  // 2 when two rings fit side by side, else 1
    bool pair;        // CTA pairs share each MMA (M = 256); tiles are then 256 vocab entries
    int units;        // the tile split's units: CTAs, or CTA pairs
    int P;            // persistent CTAs: ctas_per_sm per SM, at most one per vocab tile (two per pair tile)
    int n_slots;      // per-tile partials: one per tile and CTA (two per pair tile)
    int n_counters;   // workspace counters used (the tile counter)
    size_t smem_bytes;
    size_t ws_bytes;  // per-tile partials, 256-byte aligned
};
// n_sm: the SMs the launch may use; max_pairs: the clusters of two that can
// be resident at once (-1: n_sm / 2), which bounds the pairs of a pair plan.
LmPlan lm_plan(int R, int D, int V, int n_sm, int max_pairs = -1);
// typical-acceptance inputs produced by the same pass: per-row statistics at
// temperature T and the draft-token logit of every tree edge j, written to
// seq[b].out[j] for edges whose parent row row_base + parent[j] is in [0, R)
struct LmGatherSeq {
    const TreeDesc *tree;
    const int32_t *draft;
    float *out;
    int row_base, n;
};
struct LmGather {
    LmGatherSeq seq[TB_MAX_BATCH];
    int n_seq;
};
struct LmTypical {
    float temperature;
    float *logz_t;
    float *ent_t;
    LmGather gather;
    float *logits_out;  // null, or [R][V] fp32: the logits themselves (speculative sampling needs whole rows)
};
// pdl: launched as a programmatic dependent of the stream's previous kernel (a
// verification step's attention); the LM head does not wait for it, but
// completes only after it
cudaError_t lm_head_launch(const void *hidden, int R, const void *W, int D, int V, int32_t *argmax, float *top1,
                           float *entropy, void *parts, int *counters, int *status, int n_sm, cudaStream_t stream,
                           const char **err, int expire_wait = 0, const LmTypical *typ = nullptr, bool pdl = false);

// rotary embedding at the tree's position offsets (rope.cu)
constexpr int kRopeMaxHalf = 64;                                // pairs per head (head_dim <= 128)
constexpr int kRopeTableEntries = kMaxNodes * kRopeMaxHalf;    // cos / sin per (depth, pair)
struct RopeSeq {
    __nv_bfloat16 *k;
    long long layer_stride, head_stride;  // elements
    const TreeDesc *tree;
    int L;
};
struct RopeParams {
    RopeSeq seq[TB_MAX_BATCH];
    int layer_begin, Hkv, d;
    double inv_freq[kRopeMaxHalf];
    float2 *table;  // [n_seq][kRopeTableEntries]: (cos, sin) at position L + depth
    // scheduled mode: tree = rung_tree[sched[0]], L = sched[1]
    const int32_t *sched;
    const TreeDesc *rung_tree[8];
    int n_rungs, L_cap;
};
void rope_inv_freq(double theta, int d, double *inv_freq);
// the table, then the in-place rotation of every sequence's tree keys in
// layers [layer_begin, layer_begin + n_layers)
cudaError_t rope_launch(const RopeParams &p, int n_seq, int max_nodes, int n_layers, cudaStream_t stream);

// tree attention on tcgen05 (attention_tc.cu): head_dim 64 or 128, one or
// several sequences (each with its own cache, prefix length and tree; one
// head_dim and kv-head count) per launch
constexpr int kMaxSeqPerLaunch = TB_MAX_BATCH;
// The work split of one sequence: (layer, kv head, row block) units of T
// 128-key tiles each, over P persistent CTAs.
struct AttnPlan {
    int group, rows, row_blocks, T, n_units, P;
    long long total;
};
struct AttnSeq {
    const tb_kv *kv;
    const TreeDesc *tree;
    int N;
    const void *q;
    void *out;
};
int attn_tc_units(const AttnSeq *seqs, int n_seq, int Hq, int Hkv, int n_layers);
// The split-unit merge of an attention launch, kept to be enqueued later in a
// verification step by attn_merge_launch, as a programmatic dependent of the
// stream's previous kernel: after the LM head, or (after_step) after the
// acceptance kernel, beside which it runs.
struct AttnMerge {
    bool pdl_launch;  // set by the caller: launch the attention itself as a programmatic dependent
    bool pending;
    bool batched;
    alignas(64) unsigned char params[8192];
};
cudaError_t attn_merge_launch(const AttnMerge &m, cudaStream_t stream, bool after_step);
// rope_tab: null, or the (cos, sin) tables of rope.cu: the queries are then
// pre-rotary and are rotated at L + depth while they are staged
// merge_later: the split-unit merge is not enqueued but kept there
cudaError_t attn_tc_launch_batch(const AttnSeq *seqs, int n_seq, int layer_begin, int n_layers, int Hq, float *part,
                                 int *status, int n_sm, cudaStream_t stream, const char **err,
                                 const float2 *rope_tab = nullptr, AttnMerge *merge_later = nullptr);
bool attn_tc_supported(int d);
AttnPlan attn_tc_plan(int L, int N, int Hq, int Hkv, int n_layers, int n_sm);
size_t attn_tc_slot_floats(int d);  // floats per partial slot (two slots per CTA)
// scheduled mode: the tree (rung_tree[sched[0]]) and L (sched[1]) are read on
// the device; q / out hold N_max nodes per layer; all kv->n_layers layers
struct AttnSched {
    const tb_kv *kv;
    const TreeDesc *rung_tree[8];
    int n_rungs, N_max;
    const int32_t *sched;
    const void *q;
    void *out;
    const float2 *rope_tab;  // null, or the rotary tables (pre-rotary queries)
};
cudaError_t attn_tc_launch_sched(const AttnSched &sc, int Hq, float *part, int *status, int n_sm,
                                 cudaStream_t stream, const char **err, AttnMerge *merge_later = nullptr);
cudaError_t attn_tc_launch(const tb_kv *kv, const TreeDesc *d_tree, int N, int layer_begin, int n_layers,
                           const void *q, int Hq, void *out, float *part, int *status, int n_sm,
                           cudaStream_t stream, const char **err, const float2 *rope_tab = nullptr,
                           AttnMerge *merge_later = nullptr);

// acceptance + compaction (accept.cu)
struct AcceptParams {
    const TreeDesc *tree;
    const int32_t *draft;
    const int32_t *argmax;
    int vocab, L;
    // typical acceptance (typical != 0): per-row tempered log-partition and
    // entropy (indexed by node) and per-edge draft-token logits
    int typical;
    float inv_t, eps, alpha;
    const float *logz_t, *ent_t, *draft_logit;
    tb_result *result;
    const int *ws_status;  // may be null
    // compaction (n_layers == 0: acceptance only)
    uint8_t *k;
    uint8_t *v;
    long long layer_stride_b, head_stride_b;
    int n_layers, n_kv_heads, row_bytes;
    int L_cap;        // slots per head: copies touching slots >= L_cap are skipped
    // compaction of an existing path (kv_compact, a sampled step): no acceptance;
    // from_len: device accept_len, from_path: device path[accept_len]
    const int32_t *from_path, *from_len;
    // scheduled mode (sched != null, one sequence): tree = rung_tree[sched[0]],
    // drafts = draft + sched[0] * n_max, L = sched[1]; the last CTA to finish
    // (arrival ticket) evaluates the feature and the policy and writes the
    // next state: rung, L + accept_len, step + 1, feature bits, accept_len
    int32_t *sched;
    const TreeDesc *rung_tree[8];
    int n_rungs, n_max;
    int *ticket;
    int pol_kind, pol_feature, n_trace, n_heads;
    float pol_a, pol_b, pol_edges[7];
    const float *trace;
    const float *top1, *entropy;
};
// pdl: launched as a programmatic dependent of the stream's previous kernel
// (the step's LM head), whose outputs the kernel reads after pdl_wait
cudaError_t accept_launch(const AcceptParams &p, int n_sm, cudaStream_t stream, bool pdl = false);
cudaError_t accept_launch_batch(const AcceptParams *ps, int n, int n_sm, cudaStream_t stream, bool pdl = false);

// speculative sampling on the tree (sample.cu): one CTA walks the tree
struct SampleParams {
    const TreeDesc *tree;
    const int32_t *draft;
    const float *logits;  // [N][V]
    const float *logz_t;  // [N]: ln sum_v e^(z_v / T)
    const float *q;       // [N][V]: the draft distribution of each node's children
    const float *unif;    // [2N]
    float *resid;         // [V] scratch
    int V, L;
    float inv_t;
    tb_result *result;
    const int *ws_status;  // may be null
};
cudaError_t sample_launch(const SampleParams &p, cudaStream_t stream);

// Debug-bounds violation counters of the kernel translation units (0 in a
// normal build); each call resets the count it returns.
unsigned int bounds_violations_attention_tc();
unsigned int bounds_violations_lm_head();
unsigned int bounds_violations_accept();
unsigned int bounds_violations_rope();
unsigned int bounds_violations_sample();

// Raises a kernel's dynamic shared-memory limit to the device maximum, once
// per (kernel, device) (treeverify.cu).
cudaError_t allow_max_smem(const void *kernel);

// sets the message returned by tb_last_error() on this thread (treeverify.cu)
tb_status record_error(tb_status st, const char *fmt, ...);

// Argument checks of every LM-head entry point (pointers, alignment, 1..256
// rows, d_model a multiple of 8, vocab, counter capacity); fills *plan for the
// current device (treeverify.cu).
tb_status lm_validate(const void *hidden, int R, const void *W, int D, int V, const void *am, const void *t1,
                      const void *en, const char *fn, LmPlan *plan);

// tensor maps (treeverify.cu)
bool make_tmap_2d(CUtensorMap *map, const void *base, uint64_t inner, uint64_t outer, uint64_t row_bytes,
                  uint32_t box_inner, uint32_t box_outer, const char **err);
bool make_tmap_kv(CUtensorMap *map, const void *base, int d, int n_keys, int n_heads, int n_layers,
                  int64_t head_stride, int64_t layer_stride, int box_keys, const char **err);

}  // namespace tv
