// rope.cu -- rotary position embedding at the tree's position offsets.
//
// The TopologyBank stores each tree's position offsets (Sec. 1, 2.3): node i
// of a step sits at position L + depth(i).  With the base model's rotary
// embedding (Llama convention: theta_i = base^(-2i/d), element i paired with
// element i + d/2) the step's queries and tree keys are rotated at those
// positions; the prefix keys were rotated when they entered the cache.
//
//   k0_rope_table   one CTA per sequence: cos / sin of (L + depth) * theta_i
//                   for every depth of the tree and i < d/2, into the
//                   workspace.  The angle is formed and reduced to [-pi, pi]
//                   in double (positions reach 10^4-10^5 rad), then sin and
//                   cos are taken in float.  At most 64 x 64 entries, so the
//                   few double operations stay cheap on a part whose FP64
//                   rate is low.
//   k0_rope_tree_k  one warp per tree key row (layer, kv head, node): the
//                   row's pairs are rotated with the table and written back
//                   to the bf16 cache in place.
// The queries are rotated inside the attention kernel as they are staged
// into tensor memory (attention_tc.cu), with the same table.
#include <cuda_bf16.h>

#include "kernels.cuh"

namespace tv {

__global__ void __launch_bounds__(256) k0_rope_table(const __grid_constant__ RopeParams p)
{
    const RopeSeq &sq = p.seq[blockIdx.x];
    const TreeDesc *tree = sq.tree;
    int L = sq.L;
    if (p.sched) {
        const int rung = p.sched[0];
        if (rung < 0 || rung >= p.n_rungs || p.sched[1] < 0)
            return;
        tree = p.rung_tree[rung];
        L = p.sched[1];
    }
    const int h = p.d / 2;
    const int n = (tree->max_depth + 1) * h;
    float2 *tab = p.table + (size_t)blockIdx.x * kRopeTableEntries;
    constexpr double kTwoPi = 6.283185307179586476925286766559;
    for (int e = threadIdx.x; e < n; e += blockDim.x) {
        const int dep = e / h, i = e - dep * h;
        const double a = (double)(L + dep) * p.inv_freq[i];
        const double r = a - kTwoPi * rint(a * (1.0 / kTwoPi));
        float s, c;
        sincosf((float)r, &s, &c);
        tab[dep * kRopeMaxHalf + i] = make_float2(c, s);
    }
}

__global__ void __launch_bounds__(256) k0_rope_tree_k(const __grid_constant__ RopeParams p)
{
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const RopeSeq &sq = p.seq[blockIdx.z];
    const TreeDesc *tree = sq.tree;
    int L = sq.L;
    if (p.sched) {
        const int rung = p.sched[0], Ls = p.sched[1];
        if (rung < 0 || rung >= p.n_rungs || Ls < 0 || Ls + p.rung_tree[rung]->n > p.L_cap)
            return;  // no work this step (the acceptance kernel reports it)
        tree = p.rung_tree[rung];
        L = Ls;
    }
    const int j = blockIdx.x * 8 + warp;
    if (j >= tree->n)
        return;
    const int head = blockIdx.y % p.Hkv, layer = p.layer_begin + blockIdx.y / p.Hkv;
    __nv_bfloat16 *row = sq.k + (size_t)layer * sq.layer_stride + (size_t)head * sq.head_stride + (size_t)(L + j) * p.d;
    const float2 *tab = p.table + (size_t)blockIdx.z * kRopeTableEntries + tree->depth[j] * kRopeMaxHalf;
    const int h = p.d / 2;
    for (int i = lane; i < h; i += 32) {
        const float2 cs = tab[i];
        const float x1 = __bfloat162float(row[i]), x2 = __bfloat162float(row[i + h]);
        row[i] = __float2bfloat16_rn(x1 * cs.x - x2 * cs.y);
        row[i + h] = __float2bfloat16_rn(x2 * cs.x + x1 * cs.y);
    }
}

void rope_inv_freq(double theta, int d, double *inv_freq)
{
    for (int i = 0; i < d / 2; ++i)
        inv_freq[i] = pow((double)theta, -2.0 * i / d);
}

cudaError_t rope_launch(const RopeParams &p, int n_seq, int max_nodes, int n_layers, cudaStream_t stream)
{
    if (n_seq < 1 || n_seq > TB_MAX_BATCH || p.d > 2 * kRopeMaxHalf)
        return cudaErrorInvalidValue;
    k0_rope_table<<<n_seq, 256, 0, stream>>>(p);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess)
        return e;
    k0_rope_tree_k<<<dim3((max_nodes + 7) / 8, p.Hkv * n_layers, n_seq), 256, 0, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace tv
