// sample.cu -- speculative sampling on the draft tree (K4).
//
// The rule of Sec. 2.1 -- a drafted token t is accepted with probability
// min(1, p(t) / q(t)); at the first rejection the replacement comes from
// norm(max(0, p - q)) -- applied at every node of the tree to its children in
// increasing id order, the residual taking the target's place after each
// rejected sibling.  The walk starts at the root with r = p_root = softmax(
// z_root / T); an accepted child becomes the current node (r = its own
// target); the walk stops at the node none of whose children is accepted and
// the token after it is drawn from r by inverse CDF.  Uniforms are inputs:
// unif[c] decides child c, unif[N + u] draws the token at the final node u.
//
// The residual after k rejected siblings at node u has a closed form.  With
// q = q_u, c_0 = 0, S_0 = 1 and, after each rejection, c <- c + S,
// S <- sum_v max(0, p(v) - c q(v)):
//     r_k = max(0, p - c_k q) / S_k
// (induction: max(0, max(0, a) / S - q) = max(0, a - S q) / S for S > 0, so
// max(0, r_k - q) = max(0, p - (c_k + S_k) q) / S_k and the new normaliser is
// S_{k+1} / S_k).  A rejection therefore needs one sum over the vocabulary
// and no residual array; the final draw uses the unnormalised max(0, p - c q)
// against uniform * its total.  S = 0 (the residual vanished) makes r = 0:
// every later child is rejected and the draw returns the last token, as the
// sequential update does.
//
// k4_spec_sample_cluster (vocabularies up to 131072): a cluster of 8 CTAs x
// 1024 threads, each thread holding E consecutive vocabulary entries of p_u
// and q_u in registers (loaded once per node), so a rejection costs a block
// reduction and one cluster barrier.  What the decisions read -- for every
// non-root node c with parent u, p_u(t_c), q_u(t_c) and unif[c] -- depends on
// the tree and the drafts only, so every CTA gathers all of it at the start
// (one round of dependent loads for the whole walk) and the slices of a node
// are loaded only when a child of it is rejected or the draw happens there.
// The control flow -- the children tried, the decisions, the number of
// cluster barriers -- depends only on those values (the same read-only words,
// turned into the same numbers by the same instructions in every CTA) and on
// the cluster sums (the same eight CTA partials added in the same order
// everywhere), so every CTA takes the same decisions and the same barriers
// whatever the inputs hold.
//
// k4_spec_sample (larger vocabularies): one CTA of 1024 threads; the residual
// is kept explicitly in the scratch row, one read-modify-write pass per
// rejection.
#include <math.h>

#include "kernels.cuh"

namespace tv {

namespace {

constexpr int kSampleThreads = 1024;

// Block-wide sum over the kSampleThreads threads; every thread gets the total.
__device__ float block_sum(float x, float *red)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int m = 16; m >= 1; m >>= 1)
        x += __shfl_xor_sync(0xffffffffu, x, m);
    if (lane == 0)
        red[warp] = x;
    __syncthreads();
    float t = red[lane];
#pragma unroll
    for (int m = 16; m >= 1; m >>= 1)
        t += __shfl_xor_sync(0xffffffffu, t, m);
    __syncthreads();
    return t;
}

// Exclusive prefix of x over the block (thread order) and the total.
__device__ float block_exclusive_scan(float x, float *red, float *total)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    float inc = x;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
        const float y = __shfl_up_sync(0xffffffffu, inc, d);
        if (lane >= d)
            inc += y;
    }
    if (lane == 31)
        red[warp] = inc;
    __syncthreads();
    if (warp == 0) {
        float w = red[lane];
#pragma unroll
        for (int d = 1; d < 32; d <<= 1) {
            const float y = __shfl_up_sync(0xffffffffu, w, d);
            if (lane >= d)
                w += y;
        }
        red[lane] = w;  // inclusive prefix of the warp totals
    }
    __syncthreads();
    const float before = (warp > 0 ? red[warp - 1] : 0.f) + (inc - x);
    *total = red[31];
    __syncthreads();
    return before;
}

}  // namespace

// r(v) of the current node: the explicit residual times 1 / zw, or the target
// p_u(v) = 2^(z_v * scale - off) with scale = log2(e) / T, off = log2(e) logZ_u.
struct Resid {
    const float *z;
    float scale, off;
    bool expl;
    float inv_zw;
    __device__ __forceinline__ float at(const float *resid, int v) const
    {
        return expl ? resid[v] * inv_zw : ex2_approx(fmaf(z[v], scale, -off));
    }
    __device__ __forceinline__ float4 at4(const float *resid, int v) const
    {
        if (expl) {
            const float4 w = *reinterpret_cast<const float4 *>(resid + v);
            return make_float4(w.x * inv_zw, w.y * inv_zw, w.z * inv_zw, w.w * inv_zw);
        }
        const float4 x = *reinterpret_cast<const float4 *>(z + v);
        return make_float4(ex2_approx(fmaf(x.x, scale, -off)), ex2_approx(fmaf(x.y, scale, -off)),
                           ex2_approx(fmaf(x.z, scale, -off)), ex2_approx(fmaf(x.w, scale, -off)));
    }
};

__global__ void __launch_bounds__(kSampleThreads) k4_spec_sample(const __grid_constant__ SampleParams p)
{
    __shared__ float red[32];
    __shared__ int s_par[kMaxNodes];
    __shared__ int s_draft[kMaxNodes];
    __shared__ int s_tok;
    const TreeDesc *t = p.tree;
    const int n = t->n;
    const int tid = threadIdx.x;
    if (!in_bounds(n >= 1 && n <= kMaxNodes, const_cast<int *>(p.ws_status)))
        return;
    if (tid < kMaxNodes) {
        s_par[tid] = tid < n ? t->parent[tid] : -2;
        s_draft[tid] = tid < n ? p.draft[tid] : 0;
    }
    if (tid == 0)
        s_tok = 0x7fffffff;
    __syncthreads();

    constexpr float kLog2e = 1.4426950408889634f;
    const float scale = p.inv_t * kLog2e;
    // rows are 16-byte aligned when V is a multiple of 4: vector passes
    const bool vec = (p.V & 3) == 0;
    int u = 0;
    Resid r{p.logits, scale, p.logz_t[0] * kLog2e, false, 1.f};
    bool bad = false;
    for (int hop = 0; hop < kMaxNodes; ++hop) {
        const float *qu = p.q + (size_t)u * p.V;
        r = Resid{p.logits + (size_t)u * p.V, scale, p.logz_t[u] * kLog2e, false, 1.f};
        int next = -1;
        for (int c = u + 1; c < n; ++c) {
            if (s_par[c] != u)
                continue;
            const int tok = s_draft[c];
            const bool valid = tok >= 0 && tok < p.V;
            bad |= !valid;
            const float rt = valid ? r.at(p.resid, tok) : 0.f;
            const float qt = valid ? qu[tok] : 0.f;
            const bool acc = qt > 0.f ? (p.unif[c] < rt / qt) : (rt > 0.f);
            if (acc) {
                next = c;
                break;
            }
            // rejected: r <- max(0, r - q_u), renormalised through 1 / zw
            float part = 0.f;
            if (vec) {
                for (int v = 4 * tid; v < p.V; v += 4 * kSampleThreads) {
                    const float4 rv = r.at4(p.resid, v);
                    const float4 qv = *reinterpret_cast<const float4 *>(qu + v);
                    const float4 w = make_float4(fmaxf(rv.x - qv.x, 0.f), fmaxf(rv.y - qv.y, 0.f),
                                                 fmaxf(rv.z - qv.z, 0.f), fmaxf(rv.w - qv.w, 0.f));
                    *reinterpret_cast<float4 *>(p.resid + v) = w;
                    part += (w.x + w.y) + (w.z + w.w);
                }
            } else {
                for (int v = tid; v < p.V; v += kSampleThreads) {
                    const float w = fmaxf(r.at(p.resid, v) - qu[v], 0.f);
                    p.resid[v] = w;
                    part += w;
                }
            }
            const float zw = block_sum(part, red);  // its barriers also publish p.resid to the block
            r.expl = true;
            r.inv_zw = zw > 0.f ? 1.f / zw : 0.f;
        }
        if (next < 0)
            break;
        u = next;
    }

    // inverse CDF of r at u over contiguous per-thread chunks (16-byte aligned for vector loads)
    const int per = vec ? ((p.V / 4 + kSampleThreads - 1) / kSampleThreads) * 4 : (p.V + kSampleThreads - 1) / kSampleThreads;
    const int v0 = min(p.V, tid * per), v1 = min(p.V, v0 + per);
    float loc = 0.f;
    if (vec) {
        for (int v = v0; v < v1; v += 4) {
            const float4 x = r.at4(p.resid, v);
            loc += ((x.x + x.y) + x.z) + x.w;
        }
    } else {
        for (int v = v0; v < v1; ++v)
            loc += r.at(p.resid, v);
    }
    float total;
    const float before = block_exclusive_scan(loc, red, &total);
    const float thr = p.unif[n + u] * total;
    if (v1 > v0 && before <= thr && thr < before + loc) {
        float cum = before;
        int pick = v1 - 1;
        for (int v = v0; v < v1; ++v) {
            cum += r.at(p.resid, v);
            if (cum > thr) {
                pick = v;
                break;
            }
        }
        atomicMin(&s_tok, pick);  // rounding can let two neighbouring chunks claim the threshold
    }
    __syncthreads();

    if (tid == 0) {
        tb_result *res = p.result;
        const uint64_t anc = t->anc[u];
        const int len = __popcll(anc);
        int pos = 0;
        for (int i = 0; i < n; ++i)
            if ((anc >> i) & 1ull)
                res->path[pos++] = i;
        for (int i = pos; i < kMaxNodes; ++i)
            res->path[i] = -1;
        res->accept_len = len;
        res->bonus_token = s_tok == 0x7fffffff ? p.V - 1 : s_tok;  // threshold at the total: the last token
        res->new_L = p.L + len;
        const int ws = p.ws_status ? *p.ws_status : 0;
        res->status = (ws & kStatusTimeout) ? TB_ETIMEOUT
                                            : ((bad || (ws & (kStatusBadToken | kStatusBounds))) ? TB_EINVAL : TB_OK);
    }
}

// ------------------------------------------------------------ cluster walk

constexpr int kWalkCtas = 8;  // portable cluster size
constexpr int kWalkThreads = kSampleThreads;

__device__ __forceinline__ uint32_t cluster_rank()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

// All threads of all CTAs of the cluster; orders shared and global memory at
// cluster scope (writes before it are visible to every CTA after it).  The
// non-.aligned form: the threads of a warp need not be converged here.
__device__ __forceinline__ void cluster_sync()
{
    asm volatile("barrier.cluster.arrive.release;\n\tbarrier.cluster.wait.acquire;" ::: "memory");
}

// The address of the shared variable at p in the shared memory of CTA `rank`.
__device__ __forceinline__ uint32_t dsmem(const void *p, uint32_t rank)
{
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_u32(p)), "r"(rank));
    return r;
}

__device__ __forceinline__ float ld_dsmem_f32(uint32_t a)
{
    float v;
    asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(a) : "memory");
    return v;
}

// Atomic minimum on a 32-bit shared variable of another CTA of the cluster
// (ordered for the others by the next cluster barrier).
__device__ __forceinline__ void red_min_dsmem_s32(uint32_t a, int v)
{
    asm volatile("red.relaxed.cluster.shared::cluster.min.s32 [%0], %1;" ::"r"(a), "r"(v) : "memory");
}

// Sum of x over the cluster.  Every thread of every CTA gets the same bits:
// the CTA partials are added in rank order by a butterfly, and a butterfly's
// partners add the same two values (addition commutes exactly).
__device__ float cluster_sum(float x, float *red, float *part_slot)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int m = 16; m >= 1; m >>= 1)
        x += __shfl_xor_sync(0xffffffffu, x, m);
    if (lane == 0)
        red[warp] = x;
    __syncthreads();
    if (warp == 0) {
        float t = red[lane];
#pragma unroll
        for (int m = 16; m >= 1; m >>= 1)
            t += __shfl_xor_sync(0xffffffffu, t, m);
        if (lane == 0)
            *part_slot = t;
    }
    cluster_sync();
    float y = lane < kWalkCtas ? ld_dsmem_f32(dsmem(part_slot, lane)) : 0.f;
#pragma unroll
    for (int m = 16; m >= 1; m >>= 1)
        y += __shfl_xor_sync(0xffffffffu, y, m);
    return y;
}

// This thread's E consecutive entries of p_u = 2^(z * scale - off) and q_u,
// zero past the vocabulary.  vec: rows 16-byte aligned (V a multiple of 4).
template <int E>
__device__ __forceinline__ void load_slice(const float *z, const float *q, int v0, int V, bool vec, float scale,
                                           float off, float (&pv)[E], float (&qv)[E])
{
    if (vec) {
#pragma unroll
        for (int j = 0; j < E; j += 4) {
            const int v = v0 + j;  // a multiple of 4, as is V: the whole vector is in range or none of it
            float4 a = make_float4(0.f, 0.f, 0.f, 0.f), b = a;
            if (v < V) {
                a = *reinterpret_cast<const float4 *>(z + v);
                b = *reinterpret_cast<const float4 *>(q + v);
            }
            const bool in = v < V;
            pv[j] = in ? ex2_approx(fmaf(a.x, scale, -off)) : 0.f;
            pv[j + 1] = in ? ex2_approx(fmaf(a.y, scale, -off)) : 0.f;
            pv[j + 2] = in ? ex2_approx(fmaf(a.z, scale, -off)) : 0.f;
            pv[j + 3] = in ? ex2_approx(fmaf(a.w, scale, -off)) : 0.f;
            qv[j] = b.x;
            qv[j + 1] = b.y;
            qv[j + 2] = b.z;
            qv[j + 3] = b.w;
        }
    } else {
#pragma unroll
        for (int j = 0; j < E; ++j) {
            const int v = v0 + j;
            pv[j] = v < V ? ex2_approx(fmaf(z[v], scale, -off)) : 0.f;
            qv[j] = v < V ? q[v] : 0.f;
        }
    }
}

template <int E>
__global__ void __cluster_dims__(kWalkCtas, 1, 1) __launch_bounds__(kWalkThreads, 1)
    k4_spec_sample_cluster(const __grid_constant__ SampleParams p)
{
    __shared__ float red[32];
    __shared__ float s_part[2];             // this CTA's partial of the last two cluster sums
    __shared__ uint64_t l_kids[kMaxNodes];  // the children of each node (bitset)
    __shared__ int l_ok[kMaxNodes];         // per non-root node c with parent u: draft token in [0, V),
    __shared__ float l_pt[kMaxNodes];       // ... p_u(t_c), q_u(t_c) and the uniform deciding c
    __shared__ float l_qt[kMaxNodes], l_uf[kMaxNodes];
    __shared__ int s_tok;                   // rank 0: the drawn token (minimum over the claiming threads)

    constexpr float kLog2e = 1.4426950408889634f;
    const float scale = p.inv_t * kLog2e;
    const uint32_t rank = cluster_rank();
    const int tid = threadIdx.x, lane = tid & 31;
    const TreeDesc *t = p.tree;
    const int n = t->n;
    if (!in_bounds(n >= 1 && n <= kMaxNodes, const_cast<int *>(p.ws_status)))
        return;  // the same tree in every CTA: the whole cluster returns before its first barrier
    if (tid < kMaxNodes)
        l_kids[tid] = 0;
    if (tid == 0)
        s_tok = 0x7fffffff;
    __syncthreads();
    // every CTA gathers what every decision of the walk reads: they depend on
    // the tree and the drafts only, so all of them are loaded at once, up front
    // (no CTA reads another's shared memory before the first cluster barrier)
    if (tid > 0 && tid < n && tid < kMaxNodes) {
        const int c = tid, pa = t->parent[c];
        if (pa >= 0 && pa < c) {  // canonical order: a parent precedes its children
            atomicOr(reinterpret_cast<unsigned long long *>(&l_kids[pa]), 1ull << c);
            const int tok = p.draft[c];
            const bool ok = tok >= 0 && tok < p.V;
            const float zt = ok ? p.logits[(size_t)pa * p.V + tok] : 0.f;
            l_ok[c] = ok;
            l_pt[c] = ok ? ex2_approx(fmaf(zt, scale, -p.logz_t[pa] * kLog2e)) : 0.f;
            l_qt[c] = ok ? p.q[(size_t)pa * p.V + tok] : 0.f;
            l_uf[c] = p.unif[c];
        }
    }
    __syncthreads();

    const bool vec = (p.V & 3) == 0 && ((reinterpret_cast<uintptr_t>(p.logits) | reinterpret_cast<uintptr_t>(p.q)) & 15) == 0;
    const int v0 = (static_cast<int>(rank) * kWalkThreads + tid) * E;
    float pv[E], qv[E];
    int u = 0, nsum = 0;
    bool bad = false, first = true, zero = false, have = false;  // have: pv, qv hold node u's slices
    float cc = 0.f, S = 1.f;
    for (int hop = 0; hop < kMaxNodes; ++hop) {
        uint64_t kids = l_kids[u];
        first = true;
        zero = false;
        have = false;
        cc = 0.f;
        S = 1.f;
        int next = -1;
        while (kids) {  // children in increasing id
            const int c = __ffsll(static_cast<long long>(kids)) - 1;
            kids &= kids - 1ull;
            const float pt = l_pt[c], qt = l_qt[c];
            bad |= !l_ok[c];
            const float rt = first ? pt : (zero ? 0.f : fmaxf(fmaf(-cc, qt, pt), 0.f) / S);
            if (qt > 0.f ? (l_uf[c] < rt / qt) : (rt > 0.f)) {
                next = c;
                break;
            }
            // rejected: c <- c + S, S <- sum_v max(0, p - c q) over node u's slices
            if (!have) {
                load_slice<E>(p.logits + (size_t)u * p.V, p.q + (size_t)u * p.V, v0, p.V, vec, scale,
                              p.logz_t[u] * kLog2e, pv, qv);
                have = true;
            }
            cc += S;
            float part = 0.f;
#pragma unroll
            for (int j = 0; j < E; ++j)
                part += fmaxf(fmaf(-cc, qv[j], pv[j]), 0.f);
            S = cluster_sum(part, red, &s_part[nsum & 1]);
            ++nsum;
            zero = !(S > 0.f);
            first = false;
        }
        if (next <= u)  // none accepted (ids of children exceed their parent's)
            break;
        u = next;
    }
    if (!have)
        load_slice<E>(p.logits + (size_t)u * p.V, p.q + (size_t)u * p.V, v0, p.V, vec, scale, p.logz_t[u] * kLog2e,
                      pv, qv);

    // inverse CDF of max(0, p - c q) (p itself before any rejection) at u
    float loc = 0.f;
#pragma unroll
    for (int j = 0; j < E; ++j) {
        pv[j] = first ? pv[j] : (zero ? 0.f : fmaxf(fmaf(-cc, qv[j], pv[j]), 0.f));
        loc += pv[j];
    }
    float cta_total;
    const float before = block_exclusive_scan(loc, red, &cta_total);
    if (tid == 0)
        s_part[nsum & 1] = cta_total;
    cluster_sync();
    // the CTA totals in rank order: base = those of the lower ranks, grand = all
    const float tot = lane < kWalkCtas ? ld_dsmem_f32(dsmem(&s_part[nsum & 1], lane)) : 0.f;
    float base = 0.f, grand = 0.f;
#pragma unroll
    for (int r = 0; r < kWalkCtas; ++r) {
        const float x = __shfl_sync(0xffffffffu, tot, r);
        if (r == static_cast<int>(rank))
            base = grand;
        grand += x;
    }
    const float thr = p.unif[n + u] * grand;
    const float c0 = base + before;
    if (loc > 0.f && c0 <= thr && thr < c0 + loc) {
        float cum = c0;
        int pick = -1, last = -1;
#pragma unroll
        for (int j = 0; j < E; ++j) {
            cum += pv[j];
            if (pv[j] > 0.f) {
                last = v0 + j;
                if (pick < 0 && cum > thr)
                    pick = v0 + j;
            }
        }
        // into rank 0's s_tok (rounding can let two neighbouring chunks claim the threshold)
        red_min_dsmem_s32(dsmem(&s_tok, 0), pick >= 0 ? pick : last);
    }
    cluster_sync();  // every claim has reached rank 0; no CTA touches another's shared memory after it
    if (rank == 0 && tid == 0) {
        const int tok = s_tok;
        tb_result *res = p.result;
        const uint64_t anc = t->anc[u];
        const int len = __popcll(anc);
        int pos = 0;
        for (int i = 0; i < kMaxNodes; ++i)
            if ((anc >> i) & 1ull)
                res->path[pos++] = i;
        for (int i = pos; i < kMaxNodes; ++i)
            res->path[i] = -1;
        res->accept_len = len;
        res->bonus_token = tok == 0x7fffffff ? p.V - 1 : tok;  // threshold at the total: the last token
        res->new_L = p.L + len;
        const int ws = p.ws_status ? *p.ws_status : 0;
        res->status = (ws & kStatusTimeout) ? TB_ETIMEOUT
                                            : ((bad || (ws & (kStatusBadToken | kStatusBounds))) ? TB_EINVAL : TB_OK);
    }
}

cudaError_t sample_launch(const SampleParams &p, cudaStream_t stream)
{
    if (p.V <= kWalkCtas * kWalkThreads * 4)
        k4_spec_sample_cluster<4><<<kWalkCtas, kWalkThreads, 0, stream>>>(p);
    else if (p.V <= kWalkCtas * kWalkThreads * 16)
        k4_spec_sample_cluster<16><<<kWalkCtas, kWalkThreads, 0, stream>>>(p);
    else
        k4_spec_sample<<<1, kSampleThreads, 0, stream>>>(p);
    const cudaError_t e = cudaGetLastError();
    if (e == cudaSuccess)
        count_launch();
    return e;
}

TB_BOUNDS_COUNTER(bounds_violations_sample)

}  // namespace tv
