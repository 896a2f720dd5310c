// rope.cu -- rotary position embedding at the tree's position offsets.
//
// The TopologyBank stores each tree's position offsets (Sec. 1, 2.3): node i
// of a step sits at position L + depth(i).  With the base model's rotary
// embedding (Llama convention: theta_i = base^(-2i/d), element i paired with
// element i + d/2) the step's queries and tree keys are rotated at those
// positions; the prefix keys were rotated when they entered the cache.
//
//   k0_rope_tree_k  one launch: a CTA per (tree node, 64 or 128 (layer, kv
//                   head) rows of it).  Every thread first loads its 8 pairs
//                   of two rows (16 bytes from each half: the long-context
//                   step's 1024 CTAs are about one wave), then 64 threads form the
//                   (cos, sin) of (L + depth) * theta_i for the node's depth
//                   while the loads are in flight: the angle is formed and
//                   reduced to [-pi, pi] in double (positions reach 10^4-10^5
//                   rad), sin and cos are taken in float.  The rotated pairs
//                   are written back to the bf16 cache in place.  The first
//                   node of each depth (canonical order: depths do not
//                   decrease with the id) also writes its table row to the
//                   workspace for the query rotation.  head_dim 64 or 128
//                   (template kD: kD / 16 threads per row).
// The queries are rotated inside the attention kernel as they are staged
// into tensor memory (attention_tc.cu), with the same table.
#include <cuda_bf16.h>

#include "kernels.cuh"

namespace tv {

constexpr int kRopeThreads = 256;      // kD / 16 threads per row of kD elements
constexpr int kRopeRowsPerThread = 2;  // two rows a CTA-width apart: four 16-byte loads in flight

constexpr int rope_rows_per_cta(int d)
{
    return kRopeThreads / (d / 16) * kRopeRowsPerThread;
}

template <int kD>
__global__ void __launch_bounds__(kRopeThreads) k0_rope_tree_k(const __grid_constant__ RopeParams p, int n_rows)
{
    static_assert(kD == 64 || kD == 128, "head_dim 64 or 128");
    constexpr int kTpr = kD / 16;  // threads per row, 8 pairs each
    constexpr int kRowsPerCta = rope_rows_per_cta(kD);
    __shared__ float2 cs[kRopeMaxHalf];
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
    const int j = blockIdx.x;
    if (j >= tree->n)
        return;
    const int dep = tree->depth[j];
    constexpr int kHalf = kD / 2;  // pairs of a row
    const int ch = (threadIdx.x % kTpr) * 8;
    __nv_bfloat16 *row[kRopeRowsPerThread];
    uint4 lo[kRopeRowsPerThread], hi[kRopeRowsPerThread];  // elements [ch, ch + 8) and [kHalf + ch, kHalf + ch + 8)
#pragma unroll
    for (int k = 0; k < kRopeRowsPerThread; ++k) {
        const int r = blockIdx.y * kRowsPerCta + k * (kRopeThreads / kTpr) + (int)(threadIdx.x / kTpr);
        row[k] = nullptr;
        lo[k] = hi[k] = make_uint4(0, 0, 0, 0);
        if (r < n_rows && in_bounds((long long)(L + j + 1) * (2 * kHalf) <= sq.head_stride && dep < kMaxNodes, nullptr)) {
            const int head = r % p.Hkv, layer = p.layer_begin + r / p.Hkv;
            row[k] = sq.k + (size_t)layer * sq.layer_stride + (size_t)head * sq.head_stride +
                     (size_t)(L + j) * (2 * kHalf);
            lo[k] = *reinterpret_cast<const uint4 *>(row[k] + ch);
            hi[k] = *reinterpret_cast<const uint4 *>(row[k] + kHalf + ch);
        }
    }
    if (threadIdx.x < kHalf) {
        const int i = threadIdx.x;
        constexpr double kTwoPi = 6.283185307179586476925286766559;
        const double a = (double)(L + dep) * p.inv_freq[i];
        const double red = a - kTwoPi * rint(a * (1.0 / kTwoPi));
        float sn, cn;
        sincosf((float)red, &sn, &cn);
        cs[i] = make_float2(cn, sn);
        if (blockIdx.y == 0 && (j == 0 || tree->depth[j - 1] != dep))
            p.table[(size_t)blockIdx.z * kRopeTableEntries + dep * kRopeMaxHalf + i] = make_float2(cn, sn);
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < kRopeRowsPerThread; ++k) {
        if (!row[k])
            continue;
        __nv_bfloat16 *x = reinterpret_cast<__nv_bfloat16 *>(&lo[k]), *y = reinterpret_cast<__nv_bfloat16 *>(&hi[k]);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const float2 c = cs[ch + e];
            const float x1 = __bfloat162float(x[e]), x2 = __bfloat162float(y[e]);
            x[e] = __float2bfloat16_rn(x1 * c.x - x2 * c.y);
            y[e] = __float2bfloat16_rn(x2 * c.x + x1 * c.y);
        }
        *reinterpret_cast<uint4 *>(row[k] + ch) = lo[k];
        *reinterpret_cast<uint4 *>(row[k] + kHalf + ch) = hi[k];
    }
}

void rope_inv_freq(double theta, int d, double *inv_freq)
{
    for (int i = 0; i < d / 2; ++i)
        inv_freq[i] = pow((double)theta, -2.0 * i / d);
}

cudaError_t rope_launch(const RopeParams &p, int n_seq, int max_nodes, int n_layers, cudaStream_t stream)
{
    if (n_seq < 1 || n_seq > TB_MAX_BATCH || (p.d != 64 && p.d != 128) || max_nodes < 1 || max_nodes > kMaxNodes)
        return cudaErrorInvalidValue;
    const int n_rows = n_layers * p.Hkv;
    const int per_cta = rope_rows_per_cta(p.d);
    const dim3 grid(max_nodes, (n_rows + per_cta - 1) / per_cta, n_seq);
    if (p.d == 64)
        k0_rope_tree_k<64><<<grid, kRopeThreads, 0, stream>>>(p, n_rows);
    else
        k0_rope_tree_k<128><<<grid, kRopeThreads, 0, stream>>>(p, n_rows);
    const cudaError_t e = cudaGetLastError();
    if (e == cudaSuccess)
        count_launch();
    return e;
}

TB_BOUNDS_COUNTER(bounds_violations_rope)

}  // namespace tv
