// attention.cu -- tree-masked attention over the KV cache (K1).
//
// Tree decoding (Sec. 3.2): each of the N draft-tree nodes attends to the
// whole prefix [0, L) and to the tree slots of its ancestors-or-self, given by
// the topology's ancestor bitset (the precompiled tree attention mask of
// Sec. 2.3, swapped per step by pointer, Sec. 4 "Cost").
//
// Work decomposition.  A unit is (layer, kv head, block of <= 64 query rows);
// the rows of a kv head are its N nodes x (Hq/Hkv) query heads.  Each unit is
// a sequence of 64-key tiles over [0, L + N).  The flattened (unit, tile)
// space is split evenly over a persistent grid (split-L, stream-K style), so
// every CTA streams the same number of K/V bytes whatever N, L and the head
// count are.  A CTA that covers a whole unit writes the normalised output;
// a unit split between CTAs is finished by whichever CTA arrives last at the
// unit's ticket counter (log-sum-exp merge of (m, l, O) partials); no CTA
// ever waits for another.
//
// This kernel serves head_dim 64 (head_dim 128 runs on the tcgen05 kernel of
// attention_tc.cu).  Per CTA: warp 4 streams 64-key K and V tiles with TMA (4-D tensor maps over
// the caller's cache, 128-byte swizzle, zero fill past L + N) through a
// 3-stage mbarrier ring; warps 0-3 own 16 query rows each and run the
// online-softmax flash loop on the tensor cores (mma.sync m16n8k16 bf16,
// f32 accumulate) with ldmatrix reads of the swizzled tiles.
#include "kernels.cuh"

namespace tv {

struct AttnParams {
    CUtensorMap tmap_k;  // (head_dim, L + N, Hkv, layers), box (64, 64, 1, 1), 128B swizzle
    CUtensorMap tmap_v;
    const __nv_bfloat16 *q;  // [n_layers][N][Hq][d], first entry = layer_begin
    __nv_bfloat16 *out;      // same layout
    const TreeDesc *tree;
    int L, N, Hq, Hkv, group, layer_begin, n_layers;
    int rows, row_blocks, T, n_units;
    long long total;
    int P;
    float scale_log2;
    float *part;    // [P][2][64 * d + 128]
    int *counters;  // [n_units]
    int *status;
};

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t (&r)[4])
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}

__device__ __forceinline__ void ldsm_x4_trans(uint32_t addr, uint32_t (&r)[4])
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}

__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1)
{
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ void consumer_sync()
{
    asm volatile("bar.sync 1, 128;" ::: "memory");
}

__device__ __forceinline__ long long seg_begin(const AttnParams &p, int c)
{
    return (long long)c * p.total / p.P;
}

// CTA whose tile range contains flattened tile t.
__device__ __forceinline__ int cta_of(const AttnParams &p, long long t)
{
    return (int)(((t + 1) * (long long)p.P - 1) / p.total);
}

// 128-byte-swizzled offset of 16-byte chunk `chunk` of 128-byte row `row`.
__device__ __forceinline__ uint32_t sw128(int row, int chunk)
{
    return (uint32_t)(row * 128 + ((chunk ^ (row & 7)) << 4));
}

template <int D>
__global__ void __launch_bounds__(160, 2) k1_tree_attention(const __grid_constant__ AttnParams p)
{
    constexpr int kStages = 3;
    constexpr int kHalves = D / 64;           // 64-column swizzle atoms per row
    constexpr int kTileBytes = 64 * D * 2;    // one K or V tile: 64 keys x D
    constexpr int kStageBytes = 2 * kTileBytes;
    constexpr int kKSteps = D / 16;           // k16 steps of the QK^T product
    constexpr int kNBlk = D / 8;              // n8 blocks of the output
    constexpr int kSlot = 64 * D + 128;       // floats per partial slot

    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t full_bar[kStages];
    __shared__ __align__(8) uint64_t empty_bar[kStages];
    __shared__ int abort_flag;
    __shared__ int ticket;
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int c = blockIdx.x;
    const long long t0 = seg_begin(p, c), t1 = seg_begin(p, c + 1);

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&full_bar[s], 1);
            mbar_init(&empty_bar[s], 4);
        }
        abort_flag = 0;
        fence_mbar_init();
        prefetch_tmap(&p.tmap_k);
        prefetch_tmap(&p.tmap_v);
    }
    __syncthreads();

    if (warp == 4) {
        // ------------------------------------------------ TMA producer
        if (lane == 0) {
            long long issued = 0;
            const long long n = t1 - t0;
            for (long long it = 0; it < n; ++it) {
                const int s = (int)(it % kStages);
                const uint32_t ph = (uint32_t)(it / kStages) & 1u;
                if (!mbar_wait_bounded(&empty_bar[s], ph ^ 1u, &abort_flag, p.status))
                    break;
                const long long t = t0 + it;
                const int u = (int)(t / p.T);
                const int j = (int)(t % p.T);
                const int head = (u / p.row_blocks) % p.Hkv;
                const int layer = p.layer_begin + u / (p.row_blocks * p.Hkv);
                uint8_t *sk = smem + (size_t)s * kStageBytes;
                uint8_t *sv = sk + kTileBytes;
                mbar_arrive_expect_tx(&full_bar[s], kStageBytes);
#pragma unroll
                for (int h = 0; h < kHalves; ++h) {
                    tma_load_4d(sk + h * 8192, &p.tmap_k, &full_bar[s], h * 64, j * 64, head, layer);
                    tma_load_4d(sv + h * 8192, &p.tmap_v, &full_bar[s], h * 64, j * 64, head, layer);
                }
                issued = it + 1;
            }
            if (issued < n)
                for (long long it = (issued > kStages ? issued - kStages : 0); it < issued; ++it)
                    mbar_wait_drain(&full_bar[it % kStages], (uint32_t)(it / kStages) & 1u);
        }
        return;
    }

    // ---------------------------------------------------- consumers (warps 0-3)
    const int g = lane >> 2, cq = lane & 3;
    long long t = t0;
    long long it = 0;
    bool aborted = false;
    while (t < t1 && !aborted) {
        const int u = (int)(t / p.T);
        const long long u_first = (long long)u * p.T, u_last = u_first + p.T;
        const long long seg_end = t1 < u_last ? t1 : u_last;
        const bool seg_first_of_cta = (t == t0);
        const int rb = u % p.row_blocks;
        const int head = (u / p.row_blocks) % p.Hkv;
        const int layer_rel = u / (p.row_blocks * p.Hkv);
        const int rows_here = min(64, p.rows - rb * 64);
        const bool active = warp * 16 < rows_here;

        // rows owned by this thread: r0 = warp*16 + g, r1 = r0 + 8 (within the block)
        const int lr0 = warp * 16 + g, lr1 = lr0 + 8;
        bool v0 = lr0 < rows_here, v1 = lr1 < rows_here;
        const int gr0 = rb * 64 + lr0, gr1 = rb * 64 + lr1;
        const int node0 = v0 ? gr0 / p.group : 0, node1 = v1 ? gr1 / p.group : 0;
        const int qh0 = head * p.group + gr0 % p.group, qh1 = head * p.group + gr1 % p.group;
        // the rows' query / output rows and tree entries
        if (!in_bounds(layer_rel < p.n_layers && c < p.P && (!v0 || (node0 < p.N && node0 < kMaxNodes && qh0 < p.Hq)) &&
                           (!v1 || (node1 < p.N && node1 < kMaxNodes && qh1 < p.Hq)),
                       p.status))
            v0 = v1 = false;
        const uint64_t anc0 = v0 ? p.tree->anc[node0] : 0ull;
        const uint64_t anc1 = v1 ? p.tree->anc[node1] : 0ull;

        uint32_t qa[kKSteps][4];
        {
            const __nv_bfloat16 *q0 = p.q + (((size_t)layer_rel * p.N + node0) * p.Hq + qh0) * D;
            const __nv_bfloat16 *q1 = p.q + (((size_t)layer_rel * p.N + node1) * p.Hq + qh1) * D;
#pragma unroll
            for (int kk = 0; kk < kKSteps; ++kk) {
                const int col = kk * 16 + 2 * cq;
                qa[kk][0] = v0 ? *reinterpret_cast<const uint32_t *>(q0 + col) : 0u;
                qa[kk][1] = v1 ? *reinterpret_cast<const uint32_t *>(q1 + col) : 0u;
                qa[kk][2] = v0 ? *reinterpret_cast<const uint32_t *>(q0 + col + 8) : 0u;
                qa[kk][3] = v1 ? *reinterpret_cast<const uint32_t *>(q1 + col + 8) : 0u;
            }
        }

        float o[kNBlk][4];
#pragma unroll
        for (int nb = 0; nb < kNBlk; ++nb)
            o[nb][0] = o[nb][1] = o[nb][2] = o[nb][3] = 0.f;
        float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
        const long long seg_start = t;

        for (; t < seg_end; ++t, ++it) {
            const int s = (int)(it % kStages);
            const uint32_t ph = (uint32_t)(it / kStages) & 1u;
            if (!mbar_wait_bounded(&full_bar[s], ph, &abort_flag, p.status)) {
                aborted = true;
                break;
            }
            if (active) {
                const uint32_t sk = smem_u32(smem + (size_t)s * kStageBytes);
                const uint32_t sv = sk + kTileBytes;
                const int key0 = (int)(t - u_first) * 64;

                float sc[8][4];
#pragma unroll
                for (int nb = 0; nb < 8; ++nb)
                    sc[nb][0] = sc[nb][1] = sc[nb][2] = sc[nb][3] = 0.f;
#pragma unroll
                for (int kk = 0; kk < kKSteps; ++kk) {
                    const int half = kk >> 2, cc0 = (kk & 3) * 2;
#pragma unroll
                    for (int nbp = 0; nbp < 4; ++nbp) {
                        const int mi = lane >> 3;
                        const int key = (nbp * 2 + (mi >> 1)) * 8 + (lane & 7);
                        uint32_t b[4];
                        ldsm_x4(sk + half * 8192 + sw128(key, cc0 + (mi & 1)), b);
                        mma_bf16_16816(sc[2 * nbp], qa[kk], b[0], b[1]);
                        mma_bf16_16816(sc[2 * nbp + 1], qa[kk], b[2], b[3]);
                    }
                }

                // scale to log2 units, apply the tree mask on tiles that reach past the prefix
                const bool need_mask = key0 + 64 > p.L;
                float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
                for (int nb = 0; nb < 8; ++nb) {
#pragma unroll
                    for (int e = 0; e < 2; ++e) {
                        float x0 = sc[nb][e] * p.scale_log2;
                        float x1 = sc[nb][2 + e] * p.scale_log2;
                        if (need_mask) {
                            const int key = key0 + nb * 8 + 2 * cq + e;
                            const int tj = key - p.L;
                            const bool in_tree = tj >= 0 && tj < p.N;
                            const bool ok0 = tj < 0 || (in_tree && ((anc0 >> tj) & 1ull));
                            const bool ok1 = tj < 0 || (in_tree && ((anc1 >> tj) & 1ull));
                            x0 = ok0 ? x0 : -INFINITY;
                            x1 = ok1 ? x1 : -INFINITY;
                        }
                        sc[nb][e] = x0;
                        sc[nb][2 + e] = x1;
                        mx0 = fmaxf(mx0, x0);
                        mx1 = fmaxf(mx1, x1);
                    }
                }
                mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
                mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
                mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
                mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
                const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
                const float mu0 = (mn0 == -INFINITY) ? 0.f : mn0;
                const float mu1 = (mn1 == -INFINITY) ? 0.f : mn1;
                const float al0 = ex2_approx(m0 - mu0), al1 = ex2_approx(m1 - mu1);
                m0 = mn0;
                m1 = mn1;
                float rs0 = 0.f, rs1 = 0.f;
#pragma unroll
                for (int nb = 0; nb < 8; ++nb) {
                    sc[nb][0] = ex2_approx(sc[nb][0] - mu0);
                    sc[nb][1] = ex2_approx(sc[nb][1] - mu0);
                    sc[nb][2] = ex2_approx(sc[nb][2] - mu1);
                    sc[nb][3] = ex2_approx(sc[nb][3] - mu1);
                    rs0 += sc[nb][0] + sc[nb][1];
                    rs1 += sc[nb][2] + sc[nb][3];
                }
                l0 = l0 * al0 + rs0;
                l1 = l1 * al1 + rs1;
#pragma unroll
                for (int nb = 0; nb < kNBlk; ++nb) {
                    o[nb][0] *= al0;
                    o[nb][1] *= al0;
                    o[nb][2] *= al1;
                    o[nb][3] *= al1;
                }

                // O += P V
#pragma unroll
                for (int kk = 0; kk < 4; ++kk) {
                    uint32_t pa[4];
                    pa[0] = pack_bf16x2(sc[2 * kk][0], sc[2 * kk][1]);
                    pa[1] = pack_bf16x2(sc[2 * kk][2], sc[2 * kk][3]);
                    pa[2] = pack_bf16x2(sc[2 * kk + 1][0], sc[2 * kk + 1][1]);
                    pa[3] = pack_bf16x2(sc[2 * kk + 1][2], sc[2 * kk + 1][3]);
#pragma unroll
                    for (int nbp = 0; nbp < kNBlk / 2; ++nbp) {
                        const int mi = lane >> 3;
                        const int key = kk * 16 + (mi & 1) * 8 + (lane & 7);
                        const int dblk = nbp * 2 + (mi >> 1);
                        uint32_t b[4];
                        ldsm_x4_trans(sv + (dblk >> 3) * 8192 + sw128(key, dblk & 7), b);
                        mma_bf16_16816(o[2 * nbp], pa, b[0], b[1]);
                        mma_bf16_16816(o[2 * nbp + 1], pa, b[2], b[3]);
                    }
                }
            }
            __syncwarp();
            if (lane == 0)
                mbar_arrive(&empty_bar[s]);
        }
        if (aborted)
            break;

        // ------------------------------------------------ segment epilogue
        l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
        l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
        l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
        l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
        const bool whole = (seg_start == u_first) && (seg_end == u_last);
        if (whole) {
            if (active) {
                const float i0 = 1.f / l0, i1 = 1.f / l1;
                __nv_bfloat16 *o0 = p.out + (((size_t)layer_rel * p.N + node0) * p.Hq + qh0) * D;
                __nv_bfloat16 *o1 = p.out + (((size_t)layer_rel * p.N + node1) * p.Hq + qh1) * D;
#pragma unroll
                for (int nb = 0; nb < kNBlk; ++nb) {
                    const int col = nb * 8 + 2 * cq;
                    if (v0)
                        *reinterpret_cast<uint32_t *>(o0 + col) = pack_bf16x2(o[nb][0] * i0, o[nb][1] * i0);
                    if (v1)
                        *reinterpret_cast<uint32_t *>(o1 + col) = pack_bf16x2(o[nb][2] * i1, o[nb][3] * i1);
                }
            }
            continue;
        }

        // partial: (O unnormalised, m, l) into this CTA's slot, then the unit ticket
        float *slot = p.part + ((size_t)c * 2 + (seg_first_of_cta ? 0 : 1)) * kSlot;
        if (active) {
#pragma unroll
            for (int nb = 0; nb < kNBlk; ++nb) {
                const int col = nb * 8 + 2 * cq;
                *reinterpret_cast<float2 *>(slot + lr0 * D + col) = make_float2(o[nb][0], o[nb][1]);
                *reinterpret_cast<float2 *>(slot + lr1 * D + col) = make_float2(o[nb][2], o[nb][3]);
            }
            if (cq == 0) {
                slot[64 * D + lr0] = m0;
                slot[64 * D + 64 + lr0] = l0;
                slot[64 * D + lr1] = m1;
                slot[64 * D + 64 + lr1] = l1;
            }
        }
        __threadfence();
        consumer_sync();
        const int c_lo = cta_of(p, u_first), c_hi = cta_of(p, u_last - 1);
        if (threadIdx.x == 0)
            ticket = atomicAdd(&p.counters[u], 1);
        consumer_sync();
        if (ticket != c_hi - c_lo) {
            continue;
        }
        __threadfence();
        // last arrival: merge every CTA's partial of unit u
        {
            const int r = threadIdx.x >> 1;        // 0..63
            const int c0 = (threadIdx.x & 1) * (D / 2);
            if (r < rows_here) {
                float M = -INFINITY;
                for (int cc = c_lo; cc <= c_hi; ++cc) {
                    const float *sl = p.part + ((size_t)cc * 2 + (seg_begin(p, cc) >= u_first ? 0 : 1)) * kSlot;
                    M = fmaxf(M, __ldcg(sl + 64 * D + r));
                }
                float acc[D / 2];
#pragma unroll
                for (int x = 0; x < D / 2; ++x)
                    acc[x] = 0.f;
                float lsum = 0.f;
                for (int cc = c_lo; cc <= c_hi; ++cc) {
                    const float *sl = p.part + ((size_t)cc * 2 + (seg_begin(p, cc) >= u_first ? 0 : 1)) * kSlot;
                    const float ms = __ldcg(sl + 64 * D + r);
                    const float w = (ms == -INFINITY) ? 0.f : ex2_approx(ms - M);
                    lsum += w * __ldcg(sl + 64 * D + 64 + r);
#pragma unroll
                    for (int x = 0; x < D / 2; x += 4) {
                        const float4 v = __ldcg(reinterpret_cast<const float4 *>(sl + r * D + c0 + x));
                        acc[x] += w * v.x;
                        acc[x + 1] += w * v.y;
                        acc[x + 2] += w * v.z;
                        acc[x + 3] += w * v.w;
                    }
                }
                const float inv = 1.f / lsum;
                const int grow = rb * 64 + r;
                const int node = grow / p.group;
                const int qh = head * p.group + grow % p.group;
                __nv_bfloat16 *op = p.out + (((size_t)layer_rel * p.N + node) * p.Hq + qh) * D + c0;
                if (in_bounds(node < p.N && qh < p.Hq && c_lo >= 0 && c_hi < p.P, p.status)) {
#pragma unroll
                    for (int x = 0; x < D / 2; x += 2)
                        *reinterpret_cast<uint32_t *>(op + x) = pack_bf16x2(acc[x] * inv, acc[x + 1] * inv);
                }
            }
            if (threadIdx.x == 0)
                p.counters[u] = 0;
        }
    }
}

// ----------------------------------------------------------------------------
// host side

size_t attn_slot_floats(int d)
{
    return (size_t)64 * d + 128;
}

AttnPlan attn_plan(int L, int N, int Hq, int Hkv, int n_layers, int n_sm)
{
    AttnPlan pl{};
    pl.group = Hq / Hkv;
    pl.rows = N * pl.group;
    pl.row_blocks = (pl.rows + 63) / 64;
    pl.T = (L + N + 63) / 64;
    pl.n_units = n_layers * Hkv * pl.row_blocks;
    pl.total = (long long)pl.n_units * pl.T;
    long long P = 2LL * n_sm;
    if (P > pl.total)
        P = pl.total;
    pl.P = (int)P;
    return pl;
}

size_t attn_smem_bytes(int d)
{
    return (size_t)3 * 2 * 64 * d * 2 + 1024;
}

cudaError_t attn_launch(const tb_kv *kv, const TreeDesc *d_tree, int N, int layer_begin, int n_layers,
                        const void *q, int Hq, void *out, float *part, int *counters, int *status, int n_sm,
                        cudaStream_t stream, const char **err)
{
    const int d = kv->head_dim;
    const AttnPlan pl = attn_plan(kv->L, N, Hq, kv->n_kv_heads, n_layers, n_sm);
    AttnParams p{};
    if (!make_tmap_kv(&p.tmap_k, kv->k, d, kv->L + N, kv->n_kv_heads, kv->n_layers, kv->head_stride,
                      kv->layer_stride, 64, err))
        return cudaErrorInvalidValue;
    if (!make_tmap_kv(&p.tmap_v, kv->v, d, kv->L + N, kv->n_kv_heads, kv->n_layers, kv->head_stride,
                      kv->layer_stride, 64, err))
        return cudaErrorInvalidValue;
    p.q = static_cast<const __nv_bfloat16 *>(q);
    p.out = static_cast<__nv_bfloat16 *>(out);
    p.tree = d_tree;
    p.L = kv->L;
    p.N = N;
    p.Hq = Hq;
    p.Hkv = kv->n_kv_heads;
    p.group = pl.group;
    p.layer_begin = layer_begin;
    p.n_layers = n_layers;
    p.rows = pl.rows;
    p.row_blocks = pl.row_blocks;
    p.T = pl.T;
    p.n_units = pl.n_units;
    p.total = pl.total;
    p.P = pl.P;
    p.scale_log2 = 1.4426950408889634f / sqrtf((float)d);
    p.part = part;
    p.counters = counters;
    p.status = status;
    // head_dim 128 runs on the tcgen05 kernel (attention_tc.cu); this one serves head_dim 64
    if (d != 64) {
        *err = "the mma.sync attention kernel serves head_dim 64 only";
        return cudaErrorInvalidValue;
    }
    cudaError_t e;
    if ((e = allow_max_smem((const void *)k1_tree_attention<64>)) != cudaSuccess)
        return e;
    k1_tree_attention<64><<<pl.P, 160, attn_smem_bytes(d), stream>>>(p);
    return cudaGetLastError();
}

TB_BOUNDS_COUNTER(bounds_violations_attention)

}  // namespace tv
