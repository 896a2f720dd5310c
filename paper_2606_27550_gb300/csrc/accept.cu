// accept.cu -- greedy tree acceptance and KV-cache compaction (K3).
//
// Verification (Sec. 3.2, greedy form): a non-root node j "matches" when its
// draft token equals the target's greedy token after its parent,
// draft[j] == argmax[parent(j)].  Node i is accepted when every non-root node
// of its ancestor-or-self set matches; with the ancestor bitset anc[i] this is
// (anc[i] & ~match & ~root) == 0, one AND per node.  The accepted path ends at
// the deepest accepted node j* (smallest canonical id among equally deep
// ones); it is exactly the set bits of anc[j*] in increasing id order because
// canonical order puts every parent before its children.  accept_len =
// depth(j*) + 1 tokens are emitted: the accepted drafts plus the bonus token
// argmax[j*] (Sec. 5.1: tau counts tokens per draft-verify cycle).
//
// KV-cache update (Sec. 3.2): slot L + j takes slot L + path[j] for
// j < accept_len, in every layer and kv head.  path[j] >= j and path is
// increasing, so copying rows in increasing j never reads a row that an
// earlier copy overwrote; one warp copies one (layer, head, K|V) row set in
// that order, in chunks of eight rows (each chunk loads all of its source
// rows, then stores them; a warp barrier between chunks).
//
// Typical acceptance (the Medusa/Hydra rule the paper keeps, Sec. 5.1/5.2):
// edge j passes when p_T(draft[j] | parent) > min(eps, alpha e^(-H_T(parent))),
// with p_T = e^(z / T - logZ_T) from the LM head's tempered statistics and
// gathered draft logit.  Accepted nodes follow from the same bitset test;
// among the deepest the largest path log-likelihood sum ln p_T wins (smallest
// id on exact ties), and the bonus token is still argmax[j*].
//
// Every CTA recomputes the (tiny) acceptance itself, so acceptance and
// compaction run as one launch without a grid-wide barrier.
#include "kernels.cuh"

namespace tv {

// Slot L + j takes slot L + path[j] for 1 <= j < k (slot L + path[0] = L is the
// root itself).  path is strictly increasing with path[j] >= j, so in a chunk
// of consecutive j no copy reads a slot that a copy of a later chunk writes,
// and a chunk's writes land below every source of the later chunks: each chunk
// loads all of its source rows, then stores them.  A warp covers 512 bytes per
// pass: 512 / row_bytes rows side by side (row_bytes a multiple of 16, <= 512).
__device__ __forceinline__ void copy_rows(uint8_t *base, const int *path, int k, int row_bytes, int room, int lane,
                                          int *status)
{
    constexpr int kChunk = 8;
    const int lanes_per_row = row_bytes >> 4;
    const int rows_per_pass = 32 / lanes_per_row;
    const int r_in = lane / lanes_per_row;
    const int off = (lane - r_in * lanes_per_row) * 16;
    for (int j0 = 1; j0 < k; j0 += kChunk) {
        uint4 buf[kChunk];
#pragma unroll
        for (int m = 0; m < kChunk; ++m) {
            const int j = j0 + r_in + m * rows_per_pass;
            if (m * rows_per_pass < kChunk && j < k && j < j0 + kChunk) {
                const int src = path[j];
                if (src > j && src < room)
                    buf[m] = *reinterpret_cast<const uint4 *>(base + (size_t)src * row_bytes + off);
            }
        }
        __syncwarp();
#pragma unroll
        for (int m = 0; m < kChunk; ++m) {
            const int j = j0 + r_in + m * rows_per_pass;
            if (m * rows_per_pass < kChunk && j < k && j < j0 + kChunk) {
                const int src = path[j];
                if (src > j && src < room && in_bounds(j < room && off + 16 <= row_bytes, status))
                    *reinterpret_cast<uint4 *>(base + (size_t)j * row_bytes + off) = buf[m];
            }
        }
        __syncwarp();
    }
}

struct AcceptBatch {
    AcceptParams seq[TB_MAX_BATCH];
};

// A warp's registers with the tree of a step: lane l holds nodes l and l + 32
// (parent, ancestor set, depth, draft token; the tokens of existing nodes only).
struct TreeRegs {
    int n;
    int par[2], dep[2], tok[2];
    uint64_t anc[2];
    __device__ __forceinline__ void load(const TreeDesc *t, const int32_t *draft, int lane)
    {
        n = t->n;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int i = lane + 32 * h;
            par[h] = t->parent[i];
            dep[h] = t->depth[i];
            anc[h] = t->anc[i];
        }
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int i = lane + 32 * h;
            tok[h] = i < n && i < kMaxNodes ? draft[i] : 0;
        }
    }
    // the ancestor set of node j (every lane of the warp calls it)
    __device__ __forceinline__ uint64_t anc_of(int j) const
    {
        const uint64_t a0 = __shfl_sync(0xffffffffu, anc[0], j & 31);
        const uint64_t a1 = __shfl_sync(0xffffffffu, anc[1], j & 31);
        return j < 32 ? a0 : a1;
    }
};

// Asks L2 for the tree's cache rows (positions L + 1 .. L + n - 1) of the
// (layer, kv head, K|V) units this warp compacts: the copy then reads them
// from L2.  A prefetch is only a hint; it changes no data.
__device__ __forceinline__ void prefetch_tree_rows(const AcceptParams &p, int L, int n, int warp, int lane)
{
    const int units = p.n_layers * p.n_kv_heads * 2;
    const int warps_per_cta = blockDim.x >> 5;
    for (int unit = blockIdx.x * warps_per_cta + warp; unit < units; unit += gridDim.x * warps_per_cta) {
        const int which = unit & 1;
        const int lh = unit >> 1;
        const int head = lh % p.n_kv_heads, layer = lh / p.n_kv_heads;
        const uint8_t *base = (which ? p.v : p.k) + layer * p.layer_stride_b + head * p.head_stride_b +
                              (size_t)L * p.row_bytes;
        for (int j = 1 + lane; j < n && j < kMaxNodes && L + j < p.L_cap; j += 32)
            for (int off = 0; off < p.row_bytes; off += 128)
                asm volatile("prefetch.global.L2 [%0];" ::"l"(base + (size_t)j * p.row_bytes + off));
    }
}

// Per-step tree selection on the device (Sec. 4, "Path-value score" and
// "Policy"): the feature of the step just verified, then the next rung.
// Writes the state words rung, L, step, feature (bits), accept_len.
__device__ void policy_step(const AcceptParams &p, int rung, int L, int len, int jstar)
{
    const int step = p.sched[2];
    const int row = p.n_trace > 0 ? min(step, p.n_trace - 1) : 0;
    float f = 0.f;
    if (p.pol_feature == TB_FEATURE_TRACE) {
        f = p.trace[row];
    } else if (p.pol_feature == TB_FEATURE_PATH_VALUE) {
        // s = max(p0, g_1 .. g_D), g_d = p0 * p_1 * ... * p_d
        const float p0 = p.top1[jstar];
        float g = p0, sv = p0;
        for (int i = 0; i < p.n_heads; ++i) {
            g *= p.trace[(size_t)row * p.n_heads + i];
            sv = fmaxf(sv, g);
        }
        f = sv;
    } else {
        f = p.entropy[jstar];
    }
    const int nr = p.n_rungs;
    int next = rung;
    if (p.pol_kind == TB_POLICY_HYSTERETIC_LADDER) {
        if (f < p.pol_a)
            next = min(rung + 1, nr - 1);
        else if (f > p.pol_b)
            next = max(rung - 1, 0);
    } else if (p.pol_kind == TB_POLICY_BINARY) {
        next = f > p.pol_a ? 1 : (f <= p.pol_b ? 0 : (rung == 1 ? 1 : 0));
    } else {
        next = 0;
        while (next < nr - 1 && f >= p.pol_edges[next])
            ++next;
    }
    p.sched[0] = next;
    p.sched[1] = L + len;
    p.sched[2] = step + 1;
    p.sched[3] = __float_as_int(f);
    p.sched[4] = len;
}

// blockIdx.y selects the sequence; every CTA of a sequence recomputes its acceptance.
__global__ void __launch_bounds__(256) k3_accept_compact(const __grid_constant__ AcceptBatch pb)
{
    const AcceptParams &p = pb.seq[blockIdx.y];
    __shared__ int s_path[kMaxNodes];
    __shared__ float s_lp[kMaxNodes];
    __shared__ int s_len;
    __shared__ int s_rung, s_L, s_err;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    // Launched as a programmatic dependent of the step's LM head, it starts
    // while the LM head runs.  What no kernel of the step writes -- the tree,
    // the draft tokens, and the tree's cache rows the compaction may move (the
    // attention only reads them) -- is fetched before the wait below; the LM
    // head's statistics, the status word and every cache write come after it,
    // and so does the trigger that lets the split-unit merge start beside this
    // kernel.  Scheduled steps and a path from a previous kernel learn their
    // tree after the wait.
    TreeRegs tr;
    const bool early = !p.sched && !p.from_len;
    if (early) {
        if (warp == 0)
            tr.load(p.tree, p.draft, lane);
        if (p.n_layers > 0)
            prefetch_tree_rows(p, p.L, p.tree->n, warp, lane);
    }
    pdl_wait();
    pdl_trigger();

    const TreeDesc *tree = p.tree;
    const int32_t *draft = p.draft;
    int L = p.L;
    if (p.sched) {
        if (threadIdx.x == 0) {
            int rung = p.sched[0];
            const int Ls = p.sched[1];
            int err = TB_OK;
            if (rung < 0 || rung >= p.n_rungs) {
                err = TB_EINVAL;
                rung = 0;
            } else if (Ls < 0 || Ls + p.rung_tree[rung]->n > p.L_cap) {
                err = TB_ECAPACITY;
            }
            s_rung = rung;
            s_L = err == TB_OK ? Ls : 0;
            s_err = err;
        }
        __syncthreads();
        tree = p.rung_tree[s_rung];
        draft = p.draft + (size_t)s_rung * p.n_max;
        L = s_L;
    }

    if (p.from_len) {
        // path entries past accept_len are not read (a caller's array may end there)
        const int len = min(max(*p.from_len, 1), kMaxNodes);
        if (threadIdx.x < kMaxNodes)
            s_path[threadIdx.x] = threadIdx.x < len ? p.from_path[threadIdx.x] : (int)threadIdx.x;
        if (threadIdx.x == 0)
            s_len = len;
        __syncthreads();
    } else {
        if (warp == 0) {
            if (!early)
                tr.load(tree, draft, lane);
            const int n = tr.n;
            uint64_t match = 0;
            bool bad = false;
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int i = lane + 32 * h;
                bool m = false;
                if (i >= 1 && i < n && in_bounds(n <= kMaxNodes && tr.par[h] >= 0 && tr.par[h] < i,
                                                 const_cast<int *>(p.ws_status))) {
                    const int tok = tr.tok[h];
                    const bool bad_tok = (tok < 0 || tok >= p.vocab);
                    bad |= bad_tok;
                    if (!p.typical) {
                        m = (tok == p.argmax[tr.par[h]]);
                    } else {
                        const int u = tr.par[h];
                        float lp = -INFINITY;
                        if (!bad_tok) {
                            lp = p.draft_logit[i] * p.inv_t - p.logz_t[u];
                            const float thr = fminf(p.eps, p.alpha * expf(-p.ent_t[u]));
                            m = expf(lp) > thr;
                        }
                        s_lp[i] = lp;
                    }
                }
                const uint32_t bits = __ballot_sync(0xffffffffu, m);
                match |= (uint64_t)bits << (32 * h);
            }
            const bool any_bad = __any_sync(0xffffffffu, bad);
            int jstar;
            if (!p.typical) {
                // key = depth * 128 + (127 - id): the max is the deepest, smallest-id accepted node
                int best = 127;  // the root (depth 0, id 0) is always accepted
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int i = lane + 32 * h;
                    if (i < n) {
                        const uint64_t a = tr.anc[h];
                        if ((a & ~match & ~1ull) == 0ull) {
                            const int key = tr.dep[h] * 128 + (127 - i);
                            best = max(best, key);
                        }
                    }
                }
#pragma unroll
                for (int m = 16; m >= 1; m >>= 1)
                    best = max(best, __shfl_xor_sync(0xffffffffu, best, m));
                jstar = 127 - (best & 127);
            } else {
                __syncwarp();
                // accepted nodes, their depth and path log-likelihood (edges in increasing id)
                int dep[2];
                float ll[2];
                int bdep = 0;  // the root is always accepted
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int i = lane + 32 * h;
                    dep[h] = -1;
                    ll[h] = -INFINITY;
                    if (i < n) {
                        uint64_t a = tr.anc[h];
                        if ((a & ~match & ~1ull) == 0ull) {
                            float acc = 0.f;
                            a &= ~1ull;
                            while (a) {
                                acc += s_lp[__ffsll((long long)a) - 1];
                                a &= a - 1;
                            }
                            dep[h] = tr.dep[h];
                            ll[h] = acc;
                            bdep = max(bdep, dep[h]);
                        }
                    }
                }
#pragma unroll
                for (int m = 16; m >= 1; m >>= 1)
                    bdep = max(bdep, __shfl_xor_sync(0xffffffffu, bdep, m));
                float bll = -INFINITY;
#pragma unroll
                for (int h = 0; h < 2; ++h)
                    if (dep[h] == bdep)
                        bll = fmaxf(bll, ll[h]);
#pragma unroll
                for (int m = 16; m >= 1; m >>= 1)
                    bll = fmaxf(bll, __shfl_xor_sync(0xffffffffu, bll, m));
                int bid = kMaxNodes;
#pragma unroll
                for (int h = 0; h < 2; ++h)
                    if (dep[h] == bdep && ll[h] == bll)
                        bid = min(bid, lane + 32 * h);
#pragma unroll
                for (int m = 16; m >= 1; m >>= 1)
                    bid = min(bid, __shfl_xor_sync(0xffffffffu, bid, m));
                jstar = bid < n ? bid : 0;
            }
            const uint64_t pa = tr.anc_of(jstar);
            const int len = __popcll(pa);
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int i = lane + 32 * h;
                if ((pa >> i) & 1ull)
                    s_path[__popcll(pa & ((1ull << i) - 1ull))] = i;
            }
            if (lane == 0) {
                s_len = len;
                if (blockIdx.x == 0) {
                    tb_result *r = p.result;
                    r->accept_len = len;
                    r->bonus_token = p.argmax[jstar];
                    int st = TB_OK;
                    const int ws = p.ws_status ? *p.ws_status : 0;
                    if (p.sched && s_err != TB_OK)
                        st = s_err;
                    else if (ws & kStatusTimeout)
                        st = TB_ETIMEOUT;
                    else if (any_bad || (ws & (kStatusBadToken | kStatusBounds)))
                        st = TB_EINVAL;
                    r->new_L = (p.sched && s_err != TB_OK) ? p.sched[1] : L + len;
                    r->status = st;
                }
            }
            __syncwarp();
            if (blockIdx.x == 0)
                for (int i = lane; i < kMaxNodes; i += 32)
                    p.result->path[i] = (i < len) ? s_path[i] : -1;
        }
        __syncthreads();
    }

    const int k = s_len;
    const bool compact = p.n_layers > 0 && k > 1 && !(p.sched && s_err != TB_OK);
    if (compact) {
        const int units = p.n_layers * p.n_kv_heads * 2;
        const int warps_per_cta = blockDim.x >> 5;
        for (int unit = blockIdx.x * warps_per_cta + warp; unit < units; unit += gridDim.x * warps_per_cta) {
            const int which = unit & 1;
            const int lh = unit >> 1;
            const int head = lh % p.n_kv_heads, layer = lh / p.n_kv_heads;
            uint8_t *base = (which ? p.v : p.k) + layer * p.layer_stride_b + head * p.head_stride_b +
                            (size_t)L * p.row_bytes;
            if (in_bounds(layer < p.n_layers && head < p.n_kv_heads && k <= kMaxNodes,
                          const_cast<int *>(p.ws_status)))
                copy_rows(base, s_path, k, p.row_bytes, p.L_cap - L, lane, const_cast<int *>(p.ws_status));
        }
    }
    if (!p.sched)
        return;
    // ---------------- scheduled mode: the last CTA to arrive takes the policy step
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        const int ticket = atomicAdd(p.ticket, 1);
        if (ticket == (int)gridDim.x - 1) {
            *p.ticket = 0;
            if (s_err == TB_OK)
                policy_step(p, s_rung, L, k, s_path[k - 1]);
        }
    }
}

cudaError_t accept_launch_batch(const AcceptParams *ps, int n, int n_sm, cudaStream_t stream, bool pdl)
{
    if (n < 1 || n > TB_MAX_BATCH)
        return cudaErrorInvalidValue;
    AcceptBatch pb{};
    int grid = 1;
    for (int b = 0; b < n; ++b) {
        pb.seq[b] = ps[b];
        if (ps[b].n_layers > 0) {
            const int units = ps[b].n_layers * ps[b].n_kv_heads * 2;
            int gx = (units + 7) / 8;
            const int cap = (2 * n_sm + n - 1) / n;
            if (gx > cap)
                gx = cap;
            if (gx > grid)
                grid = gx;
        }
    }
    return launch_kernel(k3_accept_compact, dim3(grid, n), dim3(256), 0, stream, pdl, pb);
}

cudaError_t accept_launch(const AcceptParams &p, int n_sm, cudaStream_t stream, bool pdl)
{
    return accept_launch_batch(&p, 1, n_sm, stream, pdl);
}

TB_BOUNDS_COUNTER(bounds_violations_accept)

}  // namespace tv
