// treeverify.cu -- host side of the C ABI (include/treeverify.h): the
// TopologyBank, argument validation, workspace layout, TMA tensor maps and
// the launches of the three kernels of the verification pass.
#include <cudaTypedefs.h>

#include <atomic>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <new>
#include <vector>

#include "kernels.cuh"

namespace tv {

// ------------------------------------------------------------------ errors

static thread_local char g_err[512];

static tb_status fail(tb_status st, const char *fmt, ...)
{
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof g_err, fmt, ap);
    va_end(ap);
    return st;
}

cudaError_t allow_max_smem(const void *kernel)
{
    static std::mutex mu;
    static std::vector<std::pair<const void *, int>> done;
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess)
        return e;
    std::lock_guard<std::mutex> lk(mu);
    for (auto &kd : done)
        if (kd.first == kernel && kd.second == dev)
            return cudaSuccess;
    int max_optin = 0;
    if ((e = cudaDeviceGetAttribute(&max_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev)) != cudaSuccess)
        return e;
    cudaFuncAttributes attr;
    if ((e = cudaFuncGetAttributes(&attr, kernel)) != cudaSuccess)
        return e;
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             max_optin - (int)attr.sharedSizeBytes);
    if (e == cudaSuccess)
        done.emplace_back(kernel, dev);
    return e;
}

tb_status record_error(tb_status st, const char *fmt, ...)
{
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof g_err, fmt, ap);
    va_end(ap);
    return st;
}

static tb_status ok()
{
    g_err[0] = 0;
    return TB_OK;
}

static tb_status cuda_fail(cudaError_t e, const char *what)
{
    return fail(TB_ECUDA, "%s: %s", what, cudaGetErrorString(e));
}

// ------------------------------------------------------------------ tensor maps

static PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
static std::once_flag g_encode_once;

// cuTensorMapEncodeTiled is a driver entry point: it needs a context current
// on the calling thread, which the runtime binds (the device's primary
// context, unless the caller made another one current) only at the thread's
// first runtime call that needs one.  A host thread whose first library call
// encodes a tensor map before any launch (a verification step run as one
// chain) would otherwise find none.  cudaFree(nullptr) is such a call and
// does nothing else.
static void ensure_context()
{
    static thread_local bool done = false;
    if (done)
        return;
    if (cudaFree(nullptr) == cudaSuccess)
        done = true;
}

static bool get_encode(const char **err)
{
    ensure_context();
    std::call_once(g_encode_once, [] {
        void *fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    });
    if (!g_encode) {
        *err = "cuTensorMapEncodeTiled unavailable from the driver";
        return false;
    }
    return true;
}

bool make_tmap_2d(CUtensorMap *map, const void *base, uint64_t inner, uint64_t outer, uint64_t row_bytes,
                  uint32_t box_inner, uint32_t box_outer, const char **err)
{
    if (!get_encode(err))
        return false;
    cuuint64_t dims[2] = {inner, outer};
    cuuint64_t strides[1] = {row_bytes};
    cuuint32_t box[2] = {box_inner, box_outer};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box,
                          estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
        *err = "cuTensorMapEncodeTiled (2-D) rejected the tensor";
        return false;
    }
    return true;
}

bool make_tmap_kv(CUtensorMap *map, const void *base, int d, int n_keys, int n_heads, int n_layers,
                  int64_t head_stride, int64_t layer_stride, int box_keys, const char **err)
{
    if (!get_encode(err))
        return false;
    cuuint64_t dims[4] = {(cuuint64_t)d, (cuuint64_t)n_keys, (cuuint64_t)n_heads, (cuuint64_t)n_layers};
    cuuint64_t strides[3] = {(cuuint64_t)d * 2, (cuuint64_t)head_stride * 2, (cuuint64_t)layer_stride * 2};
    cuuint32_t box[4] = {64, (cuuint32_t)box_keys, 1, 1};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(base), dims, strides, box,
                          estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
        *err = "cuTensorMapEncodeTiled (KV cache) rejected the tensor";
        return false;
    }
    return true;
}

// ------------------------------------------------------------------ workspace layout
//
//   [0, 256)                    status word
//   [256, 256 + 4 KiB)          LM-head counters (1024 int32; the tile counter)
//   [.., + 12 KiB)              typical acceptance: logZ_T, H_T, draft logits (3 x 1024 float)
//   [.., + 512 KiB)             rotary tables: (cos, sin) per (depth, pair), one per sequence
//   [kPartBase, ..)             attention partials, then LM-head partials
// Counters sit at fixed offsets so that calls of different shapes sharing one
// workspace always find them zero; partials are written before they are read.

constexpr size_t kTicketOff = 128;  // scheduled acceptance: arrival ticket, inside the status page
// (layer, kv head, row block) units of one attention launch: keeps the
// kernels' 32-bit unit indices in range
constexpr int kMaxAttnUnits = 1 << 24;
constexpr size_t kLmCounterOff = 256;
constexpr int kMaxLmCounters = 1024;
constexpr int kMaxTypRows = 1024;
constexpr size_t kTypOff = kLmCounterOff + (size_t)kMaxLmCounters * 4;
constexpr size_t kRopeOff = kTypOff + (size_t)3 * kMaxTypRows * 4;
constexpr size_t kPartBase = kRopeOff + (size_t)TB_MAX_BATCH * kRopeTableEntries * sizeof(float2);

static size_t align256(size_t x)
{
    return (x + 255) / 256 * 256;
}

// Partial slots of the split-L merge: two per CTA of the attention kernel.
static size_t attn_part_bytes(int n_sm, int d)
{
    return align256((size_t)n_sm * 2 * attn_tc_slot_floats(d) * 4);
}

static int sm_count(int device)
{
    static std::mutex mu;
    static std::vector<int> cache;
    std::lock_guard<std::mutex> lk(mu);
    if (device < 0)
        return 0;
    if ((int)cache.size() <= device)
        cache.resize(device + 1, 0);
    if (cache[device] == 0) {
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, device) != cudaSuccess)
            return 0;
        cache[device] = n;
    }
    return cache[device];
}

static int current_device()
{
    int d = -1;
    if (cudaGetDevice(&d) != cudaSuccess)
        return -1;
    return d;
}

static bool aligned16(const void *p)
{
    return (reinterpret_cast<uintptr_t>(p) & 15u) == 0;
}

}  // namespace tv

using namespace tv;

// ------------------------------------------------------------------ bank

struct tb_bank {
    int device;
    int capacity;
    int count;
    TreeDesc *d_desc;
    std::vector<TreeDesc> h_desc;
    std::vector<int32_t> h_parent;  // canonical parents, capacity x 64
    // A step whose attention is the longer pass forks the LM head onto `aux`
    // so that it runs in the tail of the attention kernel (whose CTAs each hold
    // a whole SM), then joins back before acceptance.  The mutex keeps one
    // step's fork/join enqueue sequence contiguous when several host threads
    // share the bank.
    cudaStream_t aux;
    cudaEvent_t ev_fork, ev_join;
    std::mutex fork_mu;
};

// The order in which one verification step's kernels are enqueued.  Two
// structures:
//  - The attention grid is capped beside a longer LM head (a single layer
//    against a large vocabulary; attn_ctas_beside_lm): one chain on the
//    caller's stream, each kernel a programmatic dependent of the one before:
//    [rotary embedding,] attention, LM head, acceptance + compaction, then the
//    attention's (small) split-unit merge, beside the acceptance kernel
//    (nothing in the step reads the attention output).  The LM head does not
//    depend on the attention: it is launched as soon as every attention CTA has
//    started and fills the SMs the attention is kept off; it completes only
//    after the attention has, so the acceptance kernel, which waits for it,
//    compacts the cache after the attention read it, and its launch overlaps
//    the LM head's tail.  The capped attention grid is itself a programmatic
//    dependent of the previous step.
//  - Otherwise: the LM head is forked onto the bank's helper stream just before
//    the attention launch (after the rotary embedding's, so that the attention
//    CTAs are placed first) and runs on the SMs that attention CTAs release,
//    the split-unit merge follows the attention on the caller's stream beside
//    the LM head, and the streams join before acceptance.  The bank's fork and
//    join events are shared, so the bank's mutex is held from construction to
//    the end of the step's enqueueing.
// Measured on GB300 against the second structure: the chain saves 1-1.5 us
// per step at the 7B single-layer shape; with an uncapped grid it cost 4-8 us
// (ragged batch, device-driven bank loop), the split-unit merge then lying on
// the critical path behind the acceptance kernel.
class StepStreams {
  public:
    StepStreams(const tb_bank *bank, cudaStream_t s, bool chain)
        : bank_(const_cast<tb_bank *>(bank)), s_(s), chain_(chain), merge_{}
    {
        if (!chain_)
            lk_ = std::unique_lock<std::mutex>(bank_->fork_mu);
    }
    bool chain() const { return chain_; }
    // the split-unit merge is kept for finish() in the chain, enqueued right
    // after the attention otherwise
    AttnMerge *merge_later() { return chain_ ? &merge_ : nullptr; }
    // an attention grid capped beside a longer LM head is itself a programmatic dependent
    void attention_pdl(bool pdl) { merge_.pdl_launch = chain_ && pdl; }
    // called between the rotary launch and the attention launch
    tb_status before_attention(const char *fn)
    {
        if (chain_)
            return TB_OK;
        cudaError_t e = cudaEventRecord(bank_->ev_fork, s_);
        if (e == cudaSuccess)
            e = cudaStreamWaitEvent(bank_->aux, bank_->ev_fork, 0);
        return e == cudaSuccess ? TB_OK : fail(TB_ECUDA, "%s: fork: %s", fn, cudaGetErrorString(e));
    }
    cudaStream_t lm_stream() const { return chain_ ? s_ : bank_->aux; }
    bool lm_pdl() const { return chain_; }
    // called after the LM head, before the kernels that read its outputs
    tb_status before_accept(const char *fn)
    {
        if (chain_)
            return TB_OK;
        cudaError_t e = cudaEventRecord(bank_->ev_join, bank_->aux);
        if (e == cudaSuccess)
            e = cudaStreamWaitEvent(s_, bank_->ev_join, 0);
        return e == cudaSuccess ? TB_OK : fail(TB_ECUDA, "%s: join: %s", fn, cudaGetErrorString(e));
    }
    bool accept_pdl() const { return chain_; }
    // the kept split-unit merge; after_step: behind the acceptance kernel (see k1_merge_split)
    tb_status merge(const char *fn, bool after_step)
    {
        cudaError_t e = chain_ ? attn_merge_launch(merge_, s_, after_step) : cudaSuccess;
        return e == cudaSuccess ? TB_OK : fail(TB_ECUDA, "%s: split-unit merge: %s", fn, cudaGetErrorString(e));
    }

  private:
    tb_bank *bank_;
    cudaStream_t s_;
    bool chain_;
    AttnMerge merge_;
    std::unique_lock<std::mutex> lk_;
};

extern "C" tb_status tb_canonicalize(const int32_t *parent, int n, int32_t *order, int32_t *bfs_parent,
                                     int32_t *depth, uint64_t *anc)
{
    if (!parent)
        return fail(TB_EINVAL, "tb_canonicalize: parent is NULL");
    if (n < 1 || n > TB_MAX_NODES)
        return fail(TB_EINVAL, "tb_canonicalize: n=%d outside 1..%d", n, TB_MAX_NODES);
    if (parent[0] != -1)
        return fail(TB_EINVAL, "tb_canonicalize: parent[0] must be -1 (node 0 is the root)");
    int children_count[TB_MAX_NODES] = {0};
    for (int i = 1; i < n; ++i) {
        if (parent[i] < 0 || parent[i] >= n || parent[i] == i)
            return fail(TB_EINVAL, "tb_canonicalize: parent[%d]=%d out of range", i, parent[i]);
        ++children_count[parent[i]];
    }
    // breadth-first from the root, children in increasing original index
    int queue[TB_MAX_NODES];
    int newid[TB_MAX_NODES];
    for (int i = 0; i < n; ++i)
        newid[i] = -1;
    int head = 0, tail = 0;
    queue[tail++] = 0;
    newid[0] = 0;
    while (head < tail) {
        const int x = queue[head++];
        for (int c = 1; c < n; ++c)
            if (parent[c] == x && newid[c] < 0) {
                newid[c] = tail;
                queue[tail++] = c;
            }
    }
    if (tail != n)
        return fail(TB_EINVAL, "tb_canonicalize: %d of %d nodes are not reachable from the root (cycle)", n - tail,
                    n);
    int32_t cpar[TB_MAX_NODES], cdep[TB_MAX_NODES];
    uint64_t canc[TB_MAX_NODES];
    for (int c = 0; c < n; ++c) {
        const int orig = queue[c];
        cpar[c] = (c == 0) ? -1 : newid[parent[orig]];
        cdep[c] = (c == 0) ? 0 : cdep[cpar[c]] + 1;
        canc[c] = (1ull << c) | (c == 0 ? 0ull : canc[cpar[c]]);
    }
    for (int c = 0; c < n; ++c) {
        if (order)
            order[c] = queue[c];
        if (bfs_parent)
            bfs_parent[c] = cpar[c];
        if (depth)
            depth[c] = cdep[c];
        if (anc)
            anc[c] = canc[c];
    }
    return ok();
}

extern "C" tb_status tb_create(tb_bank **out, int max_topologies, int device)
{
    if (!out)
        return fail(TB_EINVAL, "tb_create: out is NULL");
    *out = nullptr;
    if (max_topologies < 1 || max_topologies > 4096)
        return fail(TB_EINVAL, "tb_create: max_topologies=%d outside 1..4096", max_topologies);
    int ndev = 0;
    cudaError_t e = cudaGetDeviceCount(&ndev);
    if (e != cudaSuccess)
        return cuda_fail(e, "tb_create: cudaGetDeviceCount");
    if (device < 0 || device >= ndev)
        return fail(TB_EINVAL, "tb_create: device %d outside 0..%d", device, ndev - 1);
    int prev = current_device();
    if ((e = cudaSetDevice(device)) != cudaSuccess)
        return cuda_fail(e, "tb_create: cudaSetDevice");
    tb_bank *b = new (std::nothrow) tb_bank();
    if (!b)
        return fail(TB_ENOMEM, "tb_create: host allocation failed");
    b->device = device;
    b->capacity = max_topologies;
    b->count = 0;
    b->d_desc = nullptr;
    e = cudaMalloc(&b->d_desc, sizeof(TreeDesc) * (size_t)max_topologies);
    if (prev >= 0)
        cudaSetDevice(prev);
    if (e != cudaSuccess) {
        delete b;
        return fail(TB_ENOMEM, "tb_create: cudaMalloc of %zu bytes: %s", sizeof(TreeDesc) * (size_t)max_topologies,
                    cudaGetErrorString(e));
    }
    b->h_desc.resize(max_topologies);
    b->h_parent.assign((size_t)max_topologies * TB_MAX_NODES, -1);
    b->aux = nullptr;
    b->ev_fork = b->ev_join = nullptr;
    if ((e = cudaSetDevice(device)) == cudaSuccess &&
        (e = cudaStreamCreateWithFlags(&b->aux, cudaStreamNonBlocking)) == cudaSuccess &&
        (e = cudaEventCreateWithFlags(&b->ev_fork, cudaEventDisableTiming)) == cudaSuccess)
        e = cudaEventCreateWithFlags(&b->ev_join, cudaEventDisableTiming);
    if (prev >= 0)
        cudaSetDevice(prev);
    if (e != cudaSuccess) {
        tb_destroy(b);
        return cuda_fail(e, "tb_create: helper stream / events");
    }
    *out = b;
    return ok();
}

extern "C" tb_status tb_add_topology(tb_bank *bank, const int32_t *parent, int n, int *out_id, int32_t *order)
{
    if (!bank || !out_id)
        return fail(TB_EINVAL, "tb_add_topology: NULL bank or out_id");
    if (bank->count >= bank->capacity)
        return fail(TB_ECAPACITY, "tb_add_topology: bank full (%d topologies)", bank->capacity);
    int32_t ord[TB_MAX_NODES], bp[TB_MAX_NODES], dep[TB_MAX_NODES];
    uint64_t anc[TB_MAX_NODES];
    tb_status st = tb_canonicalize(parent, n, ord, bp, dep, anc);
    if (st != TB_OK)
        return st;
    TreeDesc t;
    memset(&t, 0, sizeof t);
    t.n = n;
    int md = 0;
    for (int c = 0; c < n; ++c) {
        t.anc[c] = anc[c];
        t.parent[c] = (int8_t)bp[c];
        t.depth[c] = (int8_t)dep[c];
        if (dep[c] > md)
            md = dep[c];
    }
    t.max_depth = md;
    const int id = bank->count;
    int prev = current_device();
    cudaError_t e = cudaSetDevice(bank->device);
    if (e == cudaSuccess)
        e = cudaMemcpy(bank->d_desc + id, &t, sizeof t, cudaMemcpyHostToDevice);
    if (prev >= 0)
        cudaSetDevice(prev);
    if (e != cudaSuccess)
        return cuda_fail(e, "tb_add_topology: upload");
    bank->h_desc[id] = t;
    for (int c = 0; c < n; ++c)
        bank->h_parent[(size_t)id * TB_MAX_NODES + c] = bp[c];
    bank->count = id + 1;
    if (order)
        memcpy(order, ord, sizeof(int32_t) * n);
    *out_id = id;
    return ok();
}

extern "C" tb_status tb_get_topology(const tb_bank *bank, int id, int *n, int32_t *parent, int32_t *depth,
                                     uint64_t *anc)
{
    if (!bank)
        return fail(TB_EINVAL, "tb_get_topology: bank is NULL");
    if (id < 0 || id >= bank->count)
        return fail(TB_ENOTFOUND, "tb_get_topology: no topology %d (bank holds %d)", id, bank->count);
    const TreeDesc &t = bank->h_desc[id];
    if (n)
        *n = t.n;
    for (int c = 0; c < t.n; ++c) {
        if (parent)
            parent[c] = bank->h_parent[(size_t)id * TB_MAX_NODES + c];
        if (depth)
            depth[c] = t.depth[c];
        if (anc)
            anc[c] = t.anc[c];
    }
    return ok();
}

extern "C" tb_status tb_destroy(tb_bank *bank)
{
    if (!bank)
        return ok();
    int prev = current_device();
    cudaError_t e = cudaSetDevice(bank->device);
    if (e == cudaSuccess && bank->d_desc)
        e = cudaFree(bank->d_desc);
    if (bank->ev_fork)
        cudaEventDestroy(bank->ev_fork);
    if (bank->ev_join)
        cudaEventDestroy(bank->ev_join);
    if (bank->aux)
        cudaStreamDestroy(bank->aux);
    if (prev >= 0)
        cudaSetDevice(prev);
    delete bank;
    if (e != cudaSuccess)
        return cuda_fail(e, "tb_destroy");
    return ok();
}

extern "C" const char *tb_last_error(void)
{
    return g_err;
}

// ------------------------------------------------------------------ workspace

extern "C" size_t tb_workspace_size(int max_rows, int n_layers, int n_kv_heads, int n_q_heads, int head_dim,
                                    int vocab, int device)
{
    (void)n_layers;
    (void)n_kv_heads;
    (void)n_q_heads;
    if (device < 0)
        device = current_device();
    const int nsm = sm_count(device);
    if (nsm <= 0)
        return 0;
    size_t bytes = kPartBase;
    if (head_dim > 0)
        bytes += attn_part_bytes(nsm, head_dim);
    if (max_rows > 0 && vocab > 0)  // batched calls run the LM head in chunks of 256 rows
        bytes += align256(lm_plan(max_rows < 256 ? max_rows : 256, 64, vocab, nsm).ws_bytes);
    return bytes;
}

extern "C" tb_status tb_workspace_init(void *workspace, size_t workspace_bytes, tb_stream stream)
{
    if (!workspace)
        return fail(TB_EINVAL, "tb_workspace_init: workspace is NULL");
    cudaError_t e = cudaMemsetAsync(workspace, 0, workspace_bytes, (cudaStream_t)stream);
    if (e != cudaSuccess)
        return cuda_fail(e, "tb_workspace_init");
    return ok();
}

extern "C" tb_status tb_workspace_status(const void *workspace, int32_t *status)
{
    if (!workspace || !status)
        return fail(TB_EINVAL, "tb_workspace_status: NULL argument");
    int32_t w = 0;
    cudaError_t e = cudaMemcpy(&w, workspace, sizeof w, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess)
        return cuda_fail(e, "tb_workspace_status");
    *status = (w & kStatusTimeout) ? TB_ETIMEOUT : (w & (kStatusBadToken | kStatusBounds)) ? TB_EINVAL : TB_OK;
    return ok();
}

static std::atomic<unsigned long long> g_launches{0};

void tv::count_launch()
{
    g_launches.fetch_add(1, std::memory_order_relaxed);
}

extern "C" tb_status tb_launch_count(uint64_t *count)
{
    if (!count)
        return fail(TB_EINVAL, "tb_launch_count: count is NULL");
    *count = g_launches.load(std::memory_order_relaxed);
    return ok();
}

extern "C" tb_status tb_debug_bounds_violations(uint32_t *count)
{
    if (!count)
        return fail(TB_EINVAL, "tb_debug_bounds_violations: count is NULL");
    cudaError_t e = cudaDeviceSynchronize();
    if (e != cudaSuccess)
        return cuda_fail(e, "tb_debug_bounds_violations");
    unsigned int n = 0;
    for (unsigned int (*f)() : {bounds_violations_attention_tc, bounds_violations_lm_head, bounds_violations_accept,
                                bounds_violations_rope, bounds_violations_sample}) {
        const unsigned int x = f();
        if (x == 0xffffffffu)
            return fail(TB_ECUDA, "tb_debug_bounds_violations: reading a device counter failed");
        n += x;
    }
    *count = n;
    return ok();
}

extern "C" int tb_debug_bounds_build(void)
{
#ifdef TB_DEBUG_BOUNDS
    return 1;
#else
    return 0;
#endif
}

// ------------------------------------------------------------------ validation helpers

static tb_status check_bank(const tb_bank *bank, int id, const char *fn)
{
    if (!bank)
        return fail(TB_EINVAL, "%s: bank is NULL", fn);
    if (id < 0 || id >= bank->count)
        return fail(TB_ENOTFOUND, "%s: bank_id %d not in bank (holds %d)", fn, id, bank->count);
    if (current_device() != bank->device)
        return fail(TB_EINVAL, "%s: current device %d is not the bank's device %d", fn, current_device(),
                    bank->device);
    return TB_OK;
}

static tb_status check_kv(const tb_kv *kv, int N, const char *fn)
{
    if (!kv || !kv->k || !kv->v)
        return fail(TB_EINVAL, "%s: kv, kv->k or kv->v is NULL", fn);
    if (!aligned16(kv->k) || !aligned16(kv->v))
        return fail(TB_EINVAL, "%s: kv->k / kv->v must be 16-byte aligned", fn);
    if (kv->head_dim != 64 && kv->head_dim != 128)
        return fail(TB_EUNSUPPORTED, "%s: head_dim %d (64 or 128 supported)", fn, kv->head_dim);
    if (kv->n_layers < 1 || kv->n_kv_heads < 1)
        return fail(TB_EINVAL, "%s: n_layers=%d n_kv_heads=%d", fn, kv->n_layers, kv->n_kv_heads);
    if (kv->L < 0 || kv->L_cap < 1)
        return fail(TB_EINVAL, "%s: L=%d L_cap=%d", fn, kv->L, kv->L_cap);
    if ((long long)kv->L + N > kv->L_cap)
        return fail(TB_ECAPACITY, "%s: L + N = %lld exceeds L_cap %d", fn, (long long)kv->L + N, kv->L_cap);
    if (kv->head_stride % 8 || kv->layer_stride % 8)
        return fail(TB_EINVAL, "%s: strides must be multiples of 8 elements", fn);
    if (kv->head_stride < (int64_t)kv->L_cap * kv->head_dim)
        return fail(TB_EINVAL, "%s: head_stride %lld < L_cap * head_dim", fn, (long long)kv->head_stride);
    if (kv->n_layers > 1 && kv->layer_stride < (int64_t)kv->n_kv_heads * kv->head_stride)
        return fail(TB_EINVAL, "%s: layer_stride %lld overlaps heads", fn, (long long)kv->layer_stride);
    return TB_OK;
}

static tb_status check_ws(void *ws, size_t bytes, size_t need, const char *fn)
{
    if (!ws)
        return fail(TB_EINVAL, "%s: workspace is NULL", fn);
    if (!aligned16(ws))
        return fail(TB_EINVAL, "%s: workspace must be 16-byte aligned", fn);
    if (bytes < need)
        return fail(TB_ECAPACITY, "%s: workspace of %zu bytes, %zu needed", fn, bytes, need);
    return TB_OK;
}

// ------------------------------------------------------------------ stages

struct AttnArgs {
    const tb_bank *bank;
    int bank_id;
    const tb_kv *kv;
    int layer_begin, n_layers;
    const void *q;
    int Hq;
    void *out;
    int max_ctas;  // > 0: the tcgen05 attention grid takes at most this many SMs
};

static tb_status check_rope(const tb_kv *kv, const char *fn);

static tb_status attn_validate(const AttnArgs &a, const char *fn, AttnPlan *plan)
{
    tb_status st = check_bank(a.bank, a.bank_id, fn);
    if (st != TB_OK)
        return st;
    const int N = a.bank->h_desc[a.bank_id].n;
    if ((st = check_kv(a.kv, N, fn)) != TB_OK)
        return st;
    if (!a.q || !a.out || !aligned16(a.q) || !aligned16(a.out))
        return fail(TB_EINVAL, "%s: q / out NULL or not 16-byte aligned", fn);
    if ((st = check_rope(a.kv, fn)) != TB_OK)
        return st;
    if (a.layer_begin < 0 || a.n_layers < 1 || a.layer_begin + a.n_layers > a.kv->n_layers)
        return fail(TB_EINVAL, "%s: layers [%d, %d) outside the cache's %d", fn, a.layer_begin,
                    a.layer_begin + a.n_layers, a.kv->n_layers);
    if (a.Hq < a.kv->n_kv_heads || a.Hq % a.kv->n_kv_heads)
        return fail(TB_EINVAL, "%s: n_q_heads %d not a multiple of n_kv_heads %d", fn, a.Hq, a.kv->n_kv_heads);
    if (N * (a.Hq / a.kv->n_kv_heads) > 256)
        return fail(TB_EUNSUPPORTED, "%s: N * group = %d > 256 query rows per kv head", fn,
                    N * (a.Hq / a.kv->n_kv_heads));
    const long long units = (long long)a.n_layers * a.kv->n_kv_heads * ((N * (a.Hq / a.kv->n_kv_heads) + 127) / 128);
    if (units > kMaxAttnUnits)
        return fail(TB_EUNSUPPORTED, "%s: %lld attention units > %d", fn, units, kMaxAttnUnits);
    const int nsm = sm_count(a.bank->device);
    *plan = attn_tc_plan(a.kv->L, N, a.Hq, a.kv->n_kv_heads, a.n_layers, nsm);
    return TB_OK;
}

static tb_status check_rope(const tb_kv *kv, const char *fn)
{
    if (kv->rope_theta == 0.f)
        return TB_OK;
    if (!(kv->rope_theta > 0.f) || !std::isfinite(kv->rope_theta))
        return fail(TB_EINVAL, "%s: rope_theta %g (0, or a positive base)", fn, (double)kv->rope_theta);
    return TB_OK;
}

static float2 *rope_table(uint8_t *ws)
{
    return reinterpret_cast<float2 *>(ws + kRopeOff);
}

// Rotary tables and in-place rotation of the tree keys of n_seq sequences
// (layers [layer_begin, layer_begin + n_layers)), before their attention.
static tb_status rope_enqueue(RopeParams &rp, const tb_kv *kv0, int n_seq, int layer_begin, int n_layers,
                              int max_nodes, uint8_t *ws, cudaStream_t s, const char *fn)
{
    rp.layer_begin = layer_begin;
    rp.Hkv = kv0->n_kv_heads;
    rp.d = kv0->head_dim;
    rope_inv_freq((double)kv0->rope_theta, kv0->head_dim, rp.inv_freq);
    rp.table = rope_table(ws);
    cudaError_t e = rope_launch(rp, n_seq, max_nodes, n_layers, s);
    if (e != cudaSuccess)
        return cuda_fail(e, fn);
    return TB_OK;
}

static RopeSeq rope_seq(const tb_kv *kv, const TreeDesc *tree)
{
    return RopeSeq{static_cast<__nv_bfloat16 *>(kv->k), (long long)kv->layer_stride, (long long)kv->head_stride,
                   tree, kv->L};
}

// The rotary embedding (if any), then the attention; ss: the verification
// step's structure (the fork comes after the rotary launch; the split-unit
// merge may be kept for later).
static tb_status attn_enqueue(const AttnArgs &a, uint8_t *ws, size_t part_off, cudaStream_t stream, const char *fn,
                              StepStreams *ss = nullptr)
{
    const char *err = "";
    const int N = a.bank->h_desc[a.bank_id].n;
    const bool rope = a.kv->rope_theta != 0.f;
    if (rope) {
        RopeParams rp{};
        rp.seq[0] = rope_seq(a.kv, a.bank->d_desc + a.bank_id);
        tb_status st = rope_enqueue(rp, a.kv, 1, a.layer_begin, a.n_layers, N, ws, stream, fn);
        if (st != TB_OK)
            return st;
    }
    if (ss) {
        tb_status st = ss->before_attention(fn);
        if (st != TB_OK)
            return st;
    }
    AttnMerge *merge_later = ss ? ss->merge_later() : nullptr;
    const int nsm = sm_count(a.bank->device);
    const cudaError_t e =
        attn_tc_launch(a.kv, a.bank->d_desc + a.bank_id, N, a.layer_begin, a.n_layers, a.q, a.Hq, a.out,
                       reinterpret_cast<float *>(ws + part_off), reinterpret_cast<int *>(ws),
                       a.max_ctas > 0 && a.max_ctas < nsm ? a.max_ctas : nsm, stream, &err,
                       rope ? rope_table(ws) : nullptr, merge_later);
    if (e == cudaErrorInvalidValue && err[0])
        return fail(TB_EINVAL, "%s: %s", fn, err);
    if (e != cudaSuccess)
        return cuda_fail(e, fn);
    return TB_OK;
}

tb_status tv::lm_validate(const void *hidden, int R, const void *W, int D, int V, const void *am, const void *t1,
                          const void *en, const char *fn, LmPlan *plan)
{
    if (!hidden || !W || !am || !t1 || !en)
        return fail(TB_EINVAL, "%s: NULL LM-head argument", fn);
    if (!aligned16(hidden) || !aligned16(W))
        return fail(TB_EINVAL, "%s: hidden / lm_head must be 16-byte aligned", fn);
    if (R < 1 || R > 256)
        return fail(TB_EUNSUPPORTED, "%s: %d rows (1..256 supported)", fn, R);
    if (D < 8 || D % 8)
        return fail(TB_EINVAL, "%s: d_model %d must be a positive multiple of 8", fn, D);
    if (V < 1)
        return fail(TB_EINVAL, "%s: vocab %d", fn, V);
    *plan = lm_plan(R, D, V, sm_count(current_device()));
    if (plan->n_counters > kMaxLmCounters)
        return fail(TB_EUNSUPPORTED, "%s: vocab %d too large", fn, V);
    return TB_OK;
}

static tb_status lm_enqueue(const void *hidden, int R, const void *W, int D, int V, int32_t *am, float *t1, float *en,
                            uint8_t *ws, size_t part_off, cudaStream_t stream, const char *fn, int expire_wait = 0,
                            const LmTypical *typ = nullptr, bool pdl = false)
{
    const char *err = "";
    cudaError_t e = lm_head_launch(hidden, R, W, D, V, am, t1, en, ws + part_off,
                                   reinterpret_cast<int *>(ws + kLmCounterOff), reinterpret_cast<int *>(ws),
                                   sm_count(current_device()), stream, &err, expire_wait, typ, pdl);
    if (e == cudaErrorInvalidValue && err[0])
        return fail(TB_EINVAL, "%s: %s", fn, err);
    if (e != cudaSuccess)
        return cuda_fail(e, fn);
    return TB_OK;
}

static AcceptParams accept_params(const tb_bank *bank, int id, const int32_t *draft, const int32_t *argmax, int vocab,
                                  int L, tb_result *result, const int *ws_status)
{
    AcceptParams p{};
    p.tree = bank->d_desc + id;
    p.draft = draft;
    p.argmax = argmax;
    p.vocab = vocab;
    p.L = L;
    p.result = result;
    p.ws_status = ws_status;
    return p;
}

static tb_status check_typical(const tb_typical *t, const char *fn)
{
    if (!t)
        return fail(TB_EINVAL, "%s: typical-acceptance parameters are NULL", fn);
    if (!(t->temperature > 0.f) || !std::isfinite(t->temperature) || !(t->eps >= 0.f) || !(t->alpha >= 0.f) ||
        !std::isfinite(t->eps) || !std::isfinite(t->alpha))
        return fail(TB_EINVAL, "%s: need T > 0 and finite eps, alpha >= 0 (T=%g eps=%g alpha=%g)", fn,
                    (double)t->temperature, (double)t->eps, (double)t->alpha);
    return TB_OK;
}

static void add_typical(AcceptParams &p, const tb_typical *t, const float *logz_t, const float *ent_t,
                        const float *draft_logit)
{
    p.typical = 1;
    p.inv_t = 1.0f / t->temperature;
    p.eps = t->eps;
    p.alpha = t->alpha;
    p.logz_t = logz_t;
    p.ent_t = ent_t;
    p.draft_logit = draft_logit;
}

// Workspace arrays of typical mode, indexed by the batch-wide row.
struct TypRows {
    float *logz_t, *ent_t, *draft_logit;
};
static TypRows typ_rows(uint8_t *ws)
{
    float *f = reinterpret_cast<float *>(ws + kTypOff);
    return TypRows{f, f + kMaxTypRows, f + 2 * kMaxTypRows};
}

static void add_compaction(AcceptParams &p, const tb_kv *kv)
{
    p.k = static_cast<uint8_t *>(kv->k);
    p.v = static_cast<uint8_t *>(kv->v);
    p.layer_stride_b = (long long)kv->layer_stride * 2;
    p.head_stride_b = (long long)kv->head_stride * 2;
    p.n_layers = kv->n_layers;
    p.n_kv_heads = kv->n_kv_heads;
    p.row_bytes = kv->head_dim * 2;
    p.L = kv->L;
    p.L_cap = kv->L_cap;
}

// ------------------------------------------------------------------ entry points

extern "C" tb_status tree_attention(const tb_bank *bank, int bank_id, const tb_kv *kv, int layer_begin, int n_layers,
                                    const void *q, int n_q_heads, void *out, void *workspace, size_t workspace_bytes,
                                    tb_stream stream)
{
    const char *fn = "tree_attention";
    AttnArgs a{bank, bank_id, kv, layer_begin, n_layers, q, n_q_heads, out};
    AttnPlan plan;
    tb_status st = attn_validate(a, fn, &plan);
    if (st != TB_OK)
        return st;
    const size_t need = kPartBase + attn_part_bytes(sm_count(bank->device), kv->head_dim);
    if ((st = check_ws(workspace, workspace_bytes, need, fn)) != TB_OK)
        return st;
    if ((st = attn_enqueue(a, static_cast<uint8_t *>(workspace), kPartBase, (cudaStream_t)stream, fn)) != TB_OK)
        return st;
    return ok();
}

extern "C" tb_status lm_head_stats(const void *hidden, int n_rows, const void *lm_head, int d_model, int vocab,
                                   int32_t *argmax, float *top1, float *entropy, void *workspace,
                                   size_t workspace_bytes, tb_stream stream)
{
    const char *fn = "lm_head_stats";
    LmPlan plan;
    tb_status st = lm_validate(hidden, n_rows, lm_head, d_model, vocab, argmax, top1, entropy, fn, &plan);
    if (st != TB_OK)
        return st;
    if ((st = check_ws(workspace, workspace_bytes, kPartBase + plan.ws_bytes, fn)) != TB_OK)
        return st;
    if ((st = lm_enqueue(hidden, n_rows, lm_head, d_model, vocab, argmax, top1, entropy,
                         static_cast<uint8_t *>(workspace), kPartBase, (cudaStream_t)stream, fn)) != TB_OK)
        return st;
    return ok();
}

extern "C" tb_status greedy_accept(const tb_bank *bank, int bank_id, const int32_t *draft_tokens,
                                   const int32_t *argmax, int vocab, int L, tb_result *result, tb_stream stream)
{
    const char *fn = "greedy_accept";
    tb_status st = check_bank(bank, bank_id, fn);
    if (st != TB_OK)
        return st;
    if (!draft_tokens || !argmax || !result)
        return fail(TB_EINVAL, "%s: NULL argument", fn);
    if (vocab < 1 || L < 0)
        return fail(TB_EINVAL, "%s: vocab=%d L=%d", fn, vocab, L);
    AcceptParams p = accept_params(bank, bank_id, draft_tokens, argmax, vocab, L, result, nullptr);
    cudaError_t e = accept_launch(p, sm_count(bank->device), (cudaStream_t)stream);
    if (e != cudaSuccess)
        return cuda_fail(e, fn);
    return ok();
}

extern "C" tb_status lm_head_stats_typical(const tb_bank *bank, int bank_id, const void *hidden, const void *lm_head,
                                           int d_model, int vocab, float temperature, const int32_t *draft_tokens,
                                           int32_t *argmax, float *top1, float *entropy, float *logz_t,
                                           float *entropy_t, float *draft_logit, void *workspace,
                                           size_t workspace_bytes, tb_stream stream)
{
    const char *fn = "lm_head_stats_typical";
    tb_status st = check_bank(bank, bank_id, fn);
    if (st != TB_OK)
        return st;
    const int N = bank->h_desc[bank_id].n;
    LmPlan plan;
    if ((st = lm_validate(hidden, N, lm_head, d_model, vocab, argmax, top1, entropy, fn, &plan)) != TB_OK)
        return st;
    if (!draft_tokens || !logz_t || !entropy_t || !draft_logit)
        return fail(TB_EINVAL, "%s: NULL draft_tokens / logz_t / entropy_t / draft_logit", fn);
    const tb_typical t{temperature, 0.f, 0.f, 0};
    if ((st = check_typical(&t, fn)) != TB_OK)
        return st;
    if ((st = check_ws(workspace, workspace_bytes, kPartBase + plan.ws_bytes, fn)) != TB_OK)
        return st;
    LmTypical lt{};
    lt.temperature = temperature;
    lt.logz_t = logz_t;
    lt.ent_t = entropy_t;
    lt.gather.n_seq = 1;
    lt.gather.seq[0] = LmGatherSeq{bank->d_desc + bank_id, draft_tokens, draft_logit, 0, N};
    if ((st = lm_enqueue(hidden, N, lm_head, d_model, vocab, argmax, top1, entropy, static_cast<uint8_t *>(workspace),
                         kPartBase, (cudaStream_t)stream, fn, 0, &lt)) != TB_OK)
        return st;
    return ok();
}

extern "C" tb_status typical_accept(const tb_bank *bank, int bank_id, const int32_t *draft_tokens,
                                    const int32_t *argmax, const float *logz_t, const float *entropy_t,
                                    const float *draft_logit, int vocab, int L, const tb_typical *params,
                                    tb_result *result, tb_stream stream)
{
    const char *fn = "typical_accept";
    tb_status st = check_bank(bank, bank_id, fn);
    if (st != TB_OK)
        return st;
    if (!draft_tokens || !argmax || !logz_t || !entropy_t || !draft_logit || !result)
        return fail(TB_EINVAL, "%s: NULL argument", fn);
    if ((st = check_typical(params, fn)) != TB_OK)
        return st;
    if (vocab < 1 || L < 0)
        return fail(TB_EINVAL, "%s: vocab=%d L=%d", fn, vocab, L);
    AcceptParams p = accept_params(bank, bank_id, draft_tokens, argmax, vocab, L, result, nullptr);
    add_typical(p, params, logz_t, entropy_t, draft_logit);
    cudaError_t e = accept_launch(p, sm_count(bank->device), (cudaStream_t)stream);
    if (e != cudaSuccess)
        return cuda_fail(e, fn);
    return ok();
}

// The attention grid beside the LM head of the same step.  The attention's
// persistent grid normally takes one CTA per SM, each holding the whole
// register file, so the LM head (launched once every attention CTA has
// started) runs on the SMs that attention CTAs release.  When the LM head is the longer of the two (a
// single layer against a large vocabulary), the attention instead gets only
// the SMs the LM head's CTAs leave free, and both run from the start.  That
// pays when the attention on those SMs still ends well before the LM head:
// about 3 us per 128-key tile a CTA walks plus 6 us, against the weight
// bytes at 5 TB/s plus 8 us (measured on GB300 at 7B shapes).  An attention
// grid that already fits beside the LM head (a small problem) keeps its own
// size and the step runs as the same chain: both start at once, and the
// programmatic launches hide the launch latencies (the tiny step: 60-65 k
// verify-steps/s against 47-57 k with the LM head forked).  0: no cap.
static int attn_ctas_beside_lm(const AttnPlan &ap, const LmPlan &lp, int d_model, int vocab, int n_sm)
{
    const int lm_sms = (lp.P + lp.ctas_per_sm - 1) / lp.ctas_per_sm;
    const int free_sms = n_sm - lm_sms;
    if (free_sms < 1 || ap.total < 1)
        return 0;
    if (ap.P <= free_sms)
        return ap.P;  // the same split as the uncapped plan (whole units stay whole)
    const double t_attn = 3.0 * (double)((ap.total + free_sms - 1) / free_sms) + 6.0;
    const double t_lm = 2.0 * (double)vocab * (double)d_model / 5.0e6 + 8.0;
    return t_attn < 0.75 * t_lm ? free_sms : 0;
}

static tb_status sample_enqueue(const tb_bank *bank, int bank_id, const int32_t *draft, const float *logits,
                                const float *logz_t, const float *q, const float *unif, int vocab, int L,
                                float temperature, float *scratch, tb_result *result, const int *ws_status,
                                cudaStream_t s, const char *fn)
{
    SampleParams sp{};
    sp.tree = bank->d_desc + bank_id;
    sp.draft = draft;
    sp.logits = logits;
    sp.logz_t = logz_t;
    sp.q = q;
    sp.unif = unif;
    sp.resid = scratch;
    sp.V = vocab;
    sp.L = L;
    sp.inv_t = 1.0f / temperature;
    sp.result = result;
    sp.ws_status = ws_status;
    cudaError_t e = sample_launch(sp, s);
    if (e != cudaSuccess)
        return cuda_fail(e, fn);
    return TB_OK;
}

extern "C" tb_status spec_sample_accept(const tb_bank *bank, int bank_id, const int32_t *draft_tokens,
                                        const float *logits, const float *logz_t, const float *draft_probs,
                                        const float *uniforms, int vocab, int L, float temperature, float *scratch,
                                        tb_result *result, tb_stream stream)
{
    const char *fn = "spec_sample_accept";
    tb_status st = check_bank(bank, bank_id, fn);
    if (st != TB_OK)
        return st;
    if (!draft_tokens || !logits || !logz_t || !draft_probs || !uniforms || !scratch || !result)
        return fail(TB_EINVAL, "%s: NULL argument", fn);
    if (vocab < 1 || L < 0)
        return fail(TB_EINVAL, "%s: vocab=%d L=%d", fn, vocab, L);
    const tb_typical t{temperature, 0.f, 0.f, 0};
    if ((st = check_typical(&t, fn)) != TB_OK)
        return st;
    if ((st = sample_enqueue(bank, bank_id, draft_tokens, logits, logz_t, draft_probs, uniforms, vocab, L,
                             temperature, scratch, result, nullptr, (cudaStream_t)stream, fn)) != TB_OK)
        return st;
    return ok();
}

extern "C" tb_status verify_step_sampled(const tb_bank *bank, int bank_id, const tb_kv *kv, const void *q,
                                         int n_q_heads, const void *hidden, const void *lm_head, int d_model,
                                         int vocab, const int32_t *draft_tokens, const float *draft_probs,
                                         const float *uniforms, float temperature, void *attn_out, int32_t *argmax,
                                         float *top1, float *entropy, float *logits, tb_result *result,
                                         void *workspace, size_t workspace_bytes, int flags, tb_stream stream)
{
    const char *fn = "verify_step_sampled";
    AttnArgs a{bank, bank_id, kv, 0, kv ? kv->n_layers : 0, q, n_q_heads, attn_out};
    AttnPlan aplan;
    tb_status st = attn_validate(a, fn, &aplan);
    if (st != TB_OK)
        return st;
    const int N = bank->h_desc[bank_id].n;
    LmPlan lplan;
    if ((st = lm_validate(hidden, N, lm_head, d_model, vocab, argmax, top1, entropy, fn, &lplan)) != TB_OK)
        return st;
    if (!draft_tokens || !draft_probs || !uniforms || !logits || !result)
        return fail(TB_EINVAL, "%s: NULL draft_tokens / draft_probs / uniforms / logits / result", fn);
    const tb_typical tt{temperature, 0.f, 0.f, 0};
    if ((st = check_typical(&tt, fn)) != TB_OK)
        return st;
    const size_t attn_bytes = attn_part_bytes(sm_count(bank->device), kv->head_dim);
    if ((st = check_ws(workspace, workspace_bytes, kPartBase + attn_bytes + lplan.ws_bytes, fn)) != TB_OK)
        return st;
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    cudaStream_t s = (cudaStream_t)stream;
    const TypRows tr = typ_rows(ws);
    LmTypical lt{};
    lt.temperature = temperature;
    lt.logz_t = tr.logz_t;
    lt.ent_t = tr.ent_t;
    lt.logits_out = logits;
    a.max_ctas = attn_ctas_beside_lm(aplan, lplan, d_model, vocab, sm_count(bank->device));
    // the structure of verify_step, with the walk between the LM head and the compaction
    StepStreams ss(bank, s, a.max_ctas > 0);
    ss.attention_pdl(kv->rope_theta == 0.f);
    if ((st = attn_enqueue(a, ws, kPartBase, s, fn, &ss)) != TB_OK)
        return st;
    if ((st = lm_enqueue(hidden, N, lm_head, d_model, vocab, argmax, top1, entropy, ws, kPartBase + attn_bytes,
                         ss.lm_stream(), fn, 0, &lt, ss.lm_pdl())) != TB_OK)
        return st;
    if ((st = ss.before_accept(fn)) != TB_OK)
        return st;
    if ((st = sample_enqueue(bank, bank_id, draft_tokens, logits, tr.logz_t, draft_probs, uniforms, vocab, kv->L,
                             temperature, logits + (size_t)N * vocab, result, reinterpret_cast<const int *>(ws), s,
                             fn)) != TB_OK)
        return st;
    if (!(flags & TB_NO_COMPACT)) {
        AcceptParams p{};
        p.from_path = result->path;
        p.from_len = &result->accept_len;
        add_compaction(p, kv);
        cudaError_t e = accept_launch(p, sm_count(bank->device), s, ss.accept_pdl());
        if (e != cudaSuccess)
            return cuda_fail(e, fn);
    }
    if ((st = ss.merge(fn, true)) != TB_OK)
        return st;
    return ok();
}

extern "C" tb_status kv_compact(const tb_kv *kv, const int32_t *path, const int32_t *accept_len, tb_stream stream)
{
    const char *fn = "kv_compact";
    tb_status st = check_kv(kv, 0, fn);
    if (st != TB_OK)
        return st;
    if (!path || !accept_len)
        return fail(TB_EINVAL, "%s: path / accept_len is NULL", fn);
    AcceptParams p{};
    p.from_path = path;
    p.from_len = accept_len;
    add_compaction(p, kv);
    cudaError_t e = accept_launch(p, sm_count(current_device()), (cudaStream_t)stream);
    if (e != cudaSuccess)
        return cuda_fail(e, fn);
    return ok();
}

static tb_status verify_step_impl(const tb_bank *bank, int bank_id, const tb_kv *kv, const void *q, int n_q_heads,
                                  const void *hidden, const void *lm_head, int d_model, int vocab,
                                  const int32_t *draft_tokens, void *attn_out, int32_t *argmax, float *top1,
                                  float *entropy, const tb_typical *typ, tb_result *result, void *workspace,
                                  size_t workspace_bytes, int flags, tb_stream stream, const char *fn)
{
    AttnArgs a{bank, bank_id, kv, 0, kv ? kv->n_layers : 0, q, n_q_heads, attn_out};
    AttnPlan aplan;
    tb_status st = attn_validate(a, fn, &aplan);
    if (st != TB_OK)
        return st;
    const int N = bank->h_desc[bank_id].n;
    LmPlan lplan;
    if ((st = lm_validate(hidden, N, lm_head, d_model, vocab, argmax, top1, entropy, fn, &lplan)) != TB_OK)
        return st;
    if (!draft_tokens || !result)
        return fail(TB_EINVAL, "%s: draft_tokens / result is NULL", fn);
    if (typ && (st = check_typical(typ, fn)) != TB_OK)
        return st;
    const size_t attn_bytes = attn_part_bytes(sm_count(bank->device), kv->head_dim);
    const size_t need = kPartBase + attn_bytes + lplan.ws_bytes;
    if ((st = check_ws(workspace, workspace_bytes, need, fn)) != TB_OK)
        return st;
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    cudaStream_t s = (cudaStream_t)stream;
    const TypRows tr = typ_rows(ws);
    LmTypical lt{};
    if (typ) {
        lt.temperature = typ->temperature;
        lt.logz_t = tr.logz_t;
        lt.ent_t = tr.ent_t;
        lt.gather.n_seq = 1;
        lt.gather.seq[0] = LmGatherSeq{bank->d_desc + bank_id, draft_tokens, tr.draft_logit, 0, N};
    }
    // the step's structure: see StepStreams
    a.max_ctas = attn_ctas_beside_lm(aplan, lplan, d_model, vocab, sm_count(bank->device));
    StepStreams ss(bank, s, a.max_ctas > 0);
    ss.attention_pdl(kv->rope_theta == 0.f);
    if ((st = attn_enqueue(a, ws, kPartBase, s, fn, &ss)) != TB_OK)
        return st;
    if ((st = lm_enqueue(hidden, N, lm_head, d_model, vocab, argmax, top1, entropy, ws, kPartBase + attn_bytes,
                         ss.lm_stream(), fn, (flags & TB_DEBUG_EXPIRE_WAIT) ? 1 : 0, typ ? &lt : nullptr,
                         ss.lm_pdl())) != TB_OK)
        return st;
    if ((st = ss.before_accept(fn)) != TB_OK)
        return st;
    AcceptParams p =
        accept_params(bank, bank_id, draft_tokens, argmax, vocab, kv->L, result, reinterpret_cast<const int *>(ws));
    if (typ)
        add_typical(p, typ, tr.logz_t, tr.ent_t, tr.draft_logit);
    if (!(flags & TB_NO_COMPACT))
        add_compaction(p, kv);
    cudaError_t e = accept_launch(p, sm_count(bank->device), s, ss.accept_pdl());
    if (e != cudaSuccess)
        return cuda_fail(e, fn);
    if ((st = ss.merge(fn, true)) != TB_OK)
        return st;
    return ok();
}

extern "C" tb_status verify_step(const tb_bank *bank, int bank_id, const tb_kv *kv, const void *q, int n_q_heads,
                                 const void *hidden, const void *lm_head, int d_model, int vocab,
                                 const int32_t *draft_tokens, void *attn_out, int32_t *argmax, float *top1,
                                 float *entropy, tb_result *result, void *workspace, size_t workspace_bytes, int flags,
                                 tb_stream stream)
{
    return verify_step_impl(bank, bank_id, kv, q, n_q_heads, hidden, lm_head, d_model, vocab, draft_tokens, attn_out,
                            argmax, top1, entropy, nullptr, result, workspace, workspace_bytes, flags, stream,
                            "verify_step");
}

extern "C" tb_status verify_step_typical(const tb_bank *bank, int bank_id, const tb_kv *kv, const void *q,
                                         int n_q_heads, const void *hidden, const void *lm_head, int d_model,
                                         int vocab, const int32_t *draft_tokens, void *attn_out, int32_t *argmax,
                                         float *top1, float *entropy, const tb_typical *params, tb_result *result,
                                         void *workspace, size_t workspace_bytes, int flags, tb_stream stream)
{
    const char *fn = "verify_step_typical";
    if (!params)
        return fail(TB_EINVAL, "%s: typical-acceptance parameters are NULL", fn);
    return verify_step_impl(bank, bank_id, kv, q, n_q_heads, hidden, lm_head, d_model, vocab, draft_tokens, attn_out,
                            argmax, top1, entropy, params, result, workspace, workspace_bytes, flags, stream, fn);
}

static tb_status verify_step_batched_impl(const tb_bank *bank, int batch, const tb_seq *seqs, int n_q_heads,
                                          const void *hidden, const void *lm_head, int d_model, int vocab,
                                          int32_t *argmax, float *top1, float *entropy, const tb_typical *typ,
                                          void *workspace, size_t workspace_bytes, int flags, tb_stream stream,
                                          const char *fn)
{
    if (!bank)
        return fail(TB_EINVAL, "%s: bank is NULL", fn);
    if (batch < 1 || batch > TB_MAX_BATCH || !seqs)
        return fail(TB_EINVAL, "%s: batch %d outside 1..%d (or seqs NULL)", fn, batch, TB_MAX_BATCH);
    tb_status st;
    int rows_total = 0;
    int Ns[TB_MAX_BATCH];
    for (int b = 0; b < batch; ++b) {
        const tb_seq &sq = seqs[b];
        if ((st = check_bank(bank, sq.bank_id, fn)) != TB_OK)
            return st;
        Ns[b] = bank->h_desc[sq.bank_id].n;
        if ((st = check_kv(&sq.kv, Ns[b], fn)) != TB_OK)
            return st;
        if ((st = check_rope(&sq.kv, fn)) != TB_OK)
            return st;
        if (sq.kv.n_layers != seqs[0].kv.n_layers || sq.kv.n_kv_heads != seqs[0].kv.n_kv_heads ||
            sq.kv.head_dim != seqs[0].kv.head_dim || sq.kv.rope_theta != seqs[0].kv.rope_theta)
            return fail(TB_EINVAL, "%s: sequence %d has another layer / head / head_dim count than sequence 0", fn,
                        b);
        if (!sq.q || !sq.attn_out || !sq.draft_tokens || !sq.result || !aligned16(sq.q) || !aligned16(sq.attn_out))
            return fail(TB_EINVAL, "%s: sequence %d: NULL or unaligned q / attn_out / draft_tokens / result", fn, b);
        rows_total += Ns[b];
    }
    const tb_kv &kv0 = seqs[0].kv;
    if (n_q_heads < kv0.n_kv_heads || n_q_heads % kv0.n_kv_heads)
        return fail(TB_EINVAL, "%s: n_q_heads %d not a multiple of n_kv_heads %d", fn, n_q_heads, kv0.n_kv_heads);
    const int group = n_q_heads / kv0.n_kv_heads;
    for (int b = 0; b < batch; ++b)
        if (Ns[b] * group > 256)
            return fail(TB_EUNSUPPORTED, "%s: sequence %d: N * group = %d > 256", fn, b, Ns[b] * group);
    if (rows_total > kMaxTypRows)
        return fail(TB_EUNSUPPORTED, "%s: %d LM-head rows > %d", fn, rows_total, kMaxTypRows);
    if (typ && (st = check_typical(typ, fn)) != TB_OK)
        return st;
    LmPlan lplan;
    const int chunk = rows_total < 256 ? rows_total : 256;
    if ((st = lm_validate(hidden, chunk, lm_head, d_model, vocab, argmax, top1, entropy, fn, &lplan)) != TB_OK)
        return st;
    const int nsm = sm_count(bank->device);
    AttnSeq as[TB_MAX_BATCH];
    long long units = 0;  // counted wide first: the plan's counts are 32-bit
    for (int b = 0; b < batch; ++b) {
        as[b] = AttnSeq{&seqs[b].kv, bank->d_desc + seqs[b].bank_id, Ns[b], seqs[b].q, seqs[b].attn_out};
        units += (long long)kv0.n_layers * kv0.n_kv_heads * ((Ns[b] * group + 127) / 128);
    }
    if (units > kMaxAttnUnits || attn_tc_units(as, batch, n_q_heads, kv0.n_kv_heads, kv0.n_layers) != units)
        return fail(TB_EUNSUPPORTED, "%s: %lld attention units > %d", fn, units, kMaxAttnUnits);
    const size_t attn_bytes = attn_part_bytes(nsm, kv0.head_dim);
    const size_t need = kPartBase + attn_bytes + lplan.ws_bytes;
    if ((st = check_ws(workspace, workspace_bytes, need, fn)) != TB_OK)
        return st;
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    cudaStream_t s = (cudaStream_t)stream;

    // the step's structure: see StepStreams
    cudaError_t e = cudaSuccess;
    StepStreams ss(bank, s, false);  // the batch's attention takes every SM
    // tree attention of every sequence (after the rotary embedding of their tree keys)
    {
        const bool rope = kv0.rope_theta != 0.f;
        if (rope) {
            RopeParams rp{};
            int max_nodes = 1;
            for (int b = 0; b < batch; ++b) {
                rp.seq[b] = rope_seq(&seqs[b].kv, bank->d_desc + seqs[b].bank_id);
                max_nodes = Ns[b] > max_nodes ? Ns[b] : max_nodes;
            }
            if ((st = rope_enqueue(rp, &kv0, batch, 0, kv0.n_layers, max_nodes, ws, s, fn)) != TB_OK)
                return st;
        }
        if ((st = ss.before_attention(fn)) != TB_OK)
            return st;
        const char *err = "";
        e = attn_tc_launch_batch(as, batch, 0, kv0.n_layers, n_q_heads, reinterpret_cast<float *>(ws + kPartBase),
                                 reinterpret_cast<int *>(ws), nsm, s, &err, rope ? rope_table(ws) : nullptr,
                                 ss.merge_later());
        if (e == cudaErrorInvalidValue && err[0])
            return fail(TB_EINVAL, "%s: %s", fn, err);
        if (e != cudaSuccess)
            return cuda_fail(e, fn);
    }
    // LM head over every row of the batch, in chunks of up to 256 rows; in
    // typical mode each chunk gathers the draft logits of the edges whose
    // parent row it holds
    const TypRows tr = typ_rows(ws);
    const uint8_t *h8 = static_cast<const uint8_t *>(hidden);
    for (int r0 = 0; r0 < rows_total; r0 += 256) {
        const int rc = rows_total - r0 < 256 ? rows_total - r0 : 256;
        LmTypical lt{};
        if (typ) {
            lt.temperature = typ->temperature;
            lt.logz_t = tr.logz_t + r0;
            lt.ent_t = tr.ent_t + r0;
            int sr = 0;
            for (int b = 0; b < batch; ++b) {
                if (sr < r0 + rc && sr + Ns[b] > r0)
                    lt.gather.seq[lt.gather.n_seq++] = LmGatherSeq{bank->d_desc + seqs[b].bank_id,
                                                                   seqs[b].draft_tokens, tr.draft_logit + sr, sr - r0,
                                                                   Ns[b]};
                sr += Ns[b];
            }
        }
        // the chunks share the partials and counters: only the first overlaps the attention
        if ((st = lm_enqueue(h8 + (size_t)r0 * d_model * 2, rc, lm_head, d_model, vocab, argmax + r0, top1 + r0,
                             entropy + r0, ws, kPartBase + attn_bytes, ss.lm_stream(), fn, 0, typ ? &lt : nullptr,
                             ss.lm_pdl() && r0 == 0)) != TB_OK)
            return st;
    }
    if ((st = ss.before_accept(fn)) != TB_OK)
        return st;
    // acceptance + compaction, one launch
    AcceptParams ps[TB_MAX_BATCH];
    int r0 = 0;
    for (int b = 0; b < batch; ++b) {
        ps[b] = accept_params(bank, seqs[b].bank_id, seqs[b].draft_tokens, argmax + r0, vocab, seqs[b].kv.L,
                              seqs[b].result, reinterpret_cast<const int *>(ws));
        if (typ)
            add_typical(ps[b], typ, tr.logz_t + r0, tr.ent_t + r0, tr.draft_logit + r0);
        if (!(flags & TB_NO_COMPACT))
            add_compaction(ps[b], &seqs[b].kv);
        r0 += Ns[b];
    }
    e = accept_launch_batch(ps, batch, nsm, s, ss.accept_pdl());
    if (e != cudaSuccess)
        return cuda_fail(e, fn);
    if ((st = ss.merge(fn, true)) != TB_OK)
        return st;
    return ok();
}

extern "C" tb_status verify_step_batched(const tb_bank *bank, int batch, const tb_seq *seqs, int n_q_heads,
                                         const void *hidden, const void *lm_head, int d_model, int vocab,
                                         int32_t *argmax, float *top1, float *entropy, void *workspace,
                                         size_t workspace_bytes, int flags, tb_stream stream)
{
    return verify_step_batched_impl(bank, batch, seqs, n_q_heads, hidden, lm_head, d_model, vocab, argmax, top1,
                                    entropy, nullptr, workspace, workspace_bytes, flags, stream,
                                    "verify_step_batched");
}

extern "C" tb_status verify_step_batched_typical(const tb_bank *bank, int batch, const tb_seq *seqs, int n_q_heads,
                                                 const void *hidden, const void *lm_head, int d_model, int vocab,
                                                 int32_t *argmax, float *top1, float *entropy,
                                                 const tb_typical *params, void *workspace, size_t workspace_bytes,
                                                 int flags, tb_stream stream)
{
    const char *fn = "verify_step_batched_typical";
    if (!params)
        return fail(TB_EINVAL, "%s: typical-acceptance parameters are NULL", fn);
    return verify_step_batched_impl(bank, batch, seqs, n_q_heads, hidden, lm_head, d_model, vocab, argmax, top1,
                                    entropy, params, workspace, workspace_bytes, flags, stream, fn);
}

// ------------------------------------------------------------------ device-driven loop

static tb_status check_policy(const tb_bank *bank, const tb_policy *pol, const char *fn, int *n_max)
{
    if (!pol)
        return fail(TB_EINVAL, "%s: policy is NULL", fn);
    if (pol->n_rungs < 1 || pol->n_rungs > 8)
        return fail(TB_EINVAL, "%s: %d rungs (1..8)", fn, pol->n_rungs);
    if (pol->kind < TB_POLICY_HYSTERETIC_LADDER || pol->kind > TB_POLICY_THRESHOLD_LADDER)
        return fail(TB_EINVAL, "%s: policy kind %d", fn, pol->kind);
    if (pol->feature < TB_FEATURE_TRACE || pol->feature > TB_FEATURE_ENTROPY)
        return fail(TB_EINVAL, "%s: feature %d", fn, pol->feature);
    if (pol->kind == TB_POLICY_BINARY && (pol->n_rungs != 2 || !(pol->b <= pol->a)))
        return fail(TB_EINVAL, "%s: the binary policy takes 2 rungs and tau_off <= tau_on", fn);
    if (pol->kind != TB_POLICY_THRESHOLD_LADDER && !(std::isfinite(pol->a) && std::isfinite(pol->b)))
        return fail(TB_EINVAL, "%s: thresholds must be finite", fn);
    if (pol->kind == TB_POLICY_THRESHOLD_LADDER)
        for (int i = 0; i + 1 < pol->n_rungs; ++i)
            if (!std::isfinite(pol->edges[i]) || (i > 0 && pol->edges[i] < pol->edges[i - 1]))
                return fail(TB_EINVAL, "%s: ladder edges must be finite and ascending", fn);
    const bool uses_trace = pol->feature == TB_FEATURE_TRACE ||
                            (pol->feature == TB_FEATURE_PATH_VALUE && pol->n_heads > 0);
    if (pol->feature == TB_FEATURE_PATH_VALUE && (pol->n_heads < 0 || pol->n_heads > 8))
        return fail(TB_EINVAL, "%s: %d head probabilities per step (0..8)", fn, pol->n_heads);
    if (uses_trace && (!pol->trace || pol->n_trace < 1))
        return fail(TB_EINVAL, "%s: the feature needs a device trace with at least one entry", fn);
    int nm = 0;
    for (int r = 0; r < pol->n_rungs; ++r) {
        tb_status st = check_bank(bank, pol->bank_ids[r], fn);
        if (st != TB_OK)
            return st;
        const int n = bank->h_desc[pol->bank_ids[r]].n;
        nm = n > nm ? n : nm;
    }
    if (pol->node_stride != 0 && (pol->node_stride < nm || pol->node_stride > kMaxNodes))
        return fail(TB_EINVAL, "%s: node_stride %d below the largest tree (%d) or above %d", fn, pol->node_stride,
                    nm, kMaxNodes);
    *n_max = pol->node_stride != 0 ? pol->node_stride : nm;
    return TB_OK;
}

extern "C" tb_status verify_step_scheduled(const tb_bank *bank, const tb_policy *policy, tb_state *state,
                                           const tb_kv *kv, const void *q, int n_q_heads, const void *hidden,
                                           const void *lm_head, int d_model, int vocab, const int32_t *draft_tokens,
                                           void *attn_out, int32_t *argmax, float *top1, float *entropy,
                                           tb_result *result, void *workspace, size_t workspace_bytes, int flags,
                                           tb_stream stream)
{
    const char *fn = "verify_step_scheduled";
    if (!bank)
        return fail(TB_EINVAL, "%s: bank is NULL", fn);
    int N_max = 0;
    tb_status st = check_policy(bank, policy, fn, &N_max);
    if (st != TB_OK)
        return st;
    if (!state || (reinterpret_cast<uintptr_t>(state) & 3u))
        return fail(TB_EINVAL, "%s: state NULL or not 4-byte aligned", fn);
    if (!kv)
        return fail(TB_EINVAL, "%s: kv is NULL", fn);
    tb_kv kv0 = *kv;
    kv0.L = 0;  // the prefix length lives in *state
    if ((st = check_kv(&kv0, N_max, fn)) != TB_OK)
        return st;
    if ((st = check_rope(kv, fn)) != TB_OK)
        return st;
    if (n_q_heads < kv->n_kv_heads || n_q_heads % kv->n_kv_heads)
        return fail(TB_EINVAL, "%s: n_q_heads %d not a multiple of n_kv_heads %d", fn, n_q_heads, kv->n_kv_heads);
    if (N_max * (n_q_heads / kv->n_kv_heads) > 256)
        return fail(TB_EUNSUPPORTED, "%s: N_max * group = %d > 256", fn, N_max * (n_q_heads / kv->n_kv_heads));
    if ((long long)kv->n_layers * kv->n_kv_heads * ((N_max * (n_q_heads / kv->n_kv_heads) + 127) / 128) >
        kMaxAttnUnits)
        return fail(TB_EUNSUPPORTED, "%s: more than %d attention units", fn, kMaxAttnUnits);
    if (!q || !attn_out || !aligned16(q) || !aligned16(attn_out))
        return fail(TB_EINVAL, "%s: q / attn_out NULL or not 16-byte aligned", fn);
    if (!draft_tokens || !result)
        return fail(TB_EINVAL, "%s: draft_tokens / result is NULL", fn);
    LmPlan lplan;
    if ((st = lm_validate(hidden, N_max, lm_head, d_model, vocab, argmax, top1, entropy, fn, &lplan)) != TB_OK)
        return st;
    const int nsm = sm_count(bank->device);
    const size_t attn_bytes = attn_part_bytes(nsm, kv->head_dim);
    if ((st = check_ws(workspace, workspace_bytes, kPartBase + attn_bytes + lplan.ws_bytes, fn)) != TB_OK)
        return st;
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    cudaStream_t s = (cudaStream_t)stream;
    AttnSched sc{};
    sc.kv = kv;
    sc.n_rungs = policy->n_rungs;
    sc.N_max = N_max;
    sc.sched = reinterpret_cast<const int32_t *>(state);
    sc.q = q;
    sc.out = attn_out;
    for (int r = 0; r < policy->n_rungs; ++r)
        sc.rung_tree[r] = bank->d_desc + policy->bank_ids[r];
    StepStreams ss(bank, s, false);  // the scheduled attention takes every SM
    {
        if (kv->rope_theta != 0.f) {
            RopeParams rp{};
            rp.seq[0] = rope_seq(kv, sc.rung_tree[0]);
            rp.sched = sc.sched;
            rp.n_rungs = sc.n_rungs;
            rp.L_cap = kv->L_cap;
            for (int r = 0; r < sc.n_rungs; ++r)
                rp.rung_tree[r] = sc.rung_tree[r];
            if ((st = rope_enqueue(rp, kv, 1, 0, kv->n_layers, N_max, ws, s, fn)) != TB_OK)
                return st;
            sc.rope_tab = rope_table(ws);
        }
        if ((st = ss.before_attention(fn)) != TB_OK)
            return st;
        const char *err = "";
        cudaError_t e = attn_tc_launch_sched(sc, n_q_heads, reinterpret_cast<float *>(ws + kPartBase),
                                             reinterpret_cast<int *>(ws), nsm, s, &err, ss.merge_later());
        if (e == cudaErrorInvalidValue && err[0])
            return fail(TB_EINVAL, "%s: %s", fn, err);
        if (e != cudaSuccess)
            return cuda_fail(e, fn);
        if ((st = lm_enqueue(hidden, N_max, lm_head, d_model, vocab, argmax, top1, entropy, ws,
                             kPartBase + attn_bytes, ss.lm_stream(), fn, 0, nullptr, ss.lm_pdl())) != TB_OK)
            return st;
        if ((st = ss.merge(fn, false)) != TB_OK)
            return st;
        if ((st = ss.before_accept(fn)) != TB_OK)
            return st;
    }
    AcceptParams p = accept_params(bank, policy->bank_ids[0], draft_tokens, argmax, vocab, 0, result,
                                   reinterpret_cast<const int *>(ws));
    if (!(flags & TB_NO_COMPACT))
        add_compaction(p, kv);
    p.L_cap = kv->L_cap;
    p.sched = reinterpret_cast<int32_t *>(state);
    p.n_rungs = policy->n_rungs;
    for (int r = 0; r < policy->n_rungs; ++r)
        p.rung_tree[r] = sc.rung_tree[r];
    p.n_max = N_max;
    p.ticket = reinterpret_cast<int *>(ws + kTicketOff);
    p.pol_kind = policy->kind;
    p.pol_feature = policy->feature;
    p.n_trace = policy->n_trace;
    p.n_heads = policy->feature == TB_FEATURE_PATH_VALUE ? policy->n_heads : 0;
    p.pol_a = policy->a;
    p.pol_b = policy->b;
    for (int i = 0; i < 7; ++i)
        p.pol_edges[i] = policy->edges[i];
    p.trace = policy->trace;
    p.top1 = top1;
    p.entropy = entropy;
    cudaError_t e = accept_launch(p, nsm, s, ss.accept_pdl());
    if (e != cudaSuccess)
        return cuda_fail(e, fn);
    return ok();
}

// ------------------------------------------------------------------ per-step tree selection

extern "C" int tb_schedule_hysteretic_ladder(int current, int n_trees, double feature, double up_below,
                                             double down_above)
{
    if (n_trees < 1)
        return 0;
    int k = current < 0 ? 0 : (current >= n_trees ? n_trees - 1 : current);
    if (feature < up_below)
        k = k + 1 < n_trees ? k + 1 : n_trees - 1;
    else if (feature > down_above)
        k = k > 0 ? k - 1 : 0;
    return k;
}

extern "C" int tb_schedule_binary(int aggressive, double s, double tau_on, double tau_off)
{
    if (s > tau_on)
        return 1;
    if (s <= tau_off)
        return 0;
    return aggressive ? 1 : 0;
}

extern "C" int tb_schedule_threshold_ladder(double s, const double *edges, int n_trees)
{
    if (!edges || n_trees <= 1)
        return 0;
    int k = 0;
    while (k < n_trees - 1 && s >= edges[k])
        ++k;
    return k;
}
