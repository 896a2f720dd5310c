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
// One CTA of 1024 threads: the accept / reject decisions are scalar, a
// residual update is one pass over the vocabulary (read z and q, write the
// unnormalised residual to scratch, block-wide sum), the final draw is a
// block-wide exclusive scan over contiguous per-thread chunks.  Every thread
// evaluates the same decisions from the same values, so no broadcast is
// needed between them.  The target probabilities are e^(z / T - logZ_T) from
// the LM head's logits and tempered log-partition, evaluated as ex2 of a
// pre-scaled exponent; the vocabulary passes run on float4 when V is a
// multiple of 4 (one SM does all of them, so the per-element work is what
// the walk costs).
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
        res->status = (ws & kStatusTimeout) ? TB_ETIMEOUT : ((bad || (ws & kStatusBadToken)) ? TB_EINVAL : TB_OK);
    }
}

cudaError_t sample_launch(const SampleParams &p, cudaStream_t stream)
{
    k4_spec_sample<<<1, kSampleThreads, 0, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace tv
