// lm_head.cu -- fused LM head with per-row greedy statistics (K2 + merge).
//
// For every tree row r: z = W h_r over the whole vocabulary, reduced on the
// fly to (max, argmax, s = sum e^(z-max), t = sum e^(z-max)(z-max)); logits
// never reach memory.  top1 = 1/s, entropy = ln s - t/s (nats).
// These are the verifier's greedy token, the base-LM top-1 probability p0 and
// the entropy feature that the EntMTP scheduler consumes (Sec. 4, "Path-value
// score" and "Cost": computed from the verifier logits already on chip).
//
// Design (swap-AB): one CTA per 128-entry vocab tile.  The tile of W
// ([128][64] bf16 per k-block, 128-byte swizzled by TMA) is the MMA's M=128 A
// operand; the tree rows ([R_pad][64] per k-block, same swizzle) are the
// N = R_pad B operand.  tcgen05.mma (kind::f16, f32 accumulate) builds the
// 128 x R_pad logit tile in TMEM over d_model/64 k-blocks fed by a multi-stage
// TMA ring.  Warp 0 lane 0 issues TMA, warp 1 lane 0 issues MMAs, then all
// eight warps read TMEM (lane = vocab entry; two warps per lane quadrant, each
// taking half of the columns), transpose through shared memory and reduce
// each row.  Per-tile statistics are merged in two levels by
// atomic arrival tickets (the last CTA of a group merges the group; the last
// group merges everything); no CTA ever waits for another.
//
// Typical-acceptance mode (kTyp): the same pass also yields, per row, the
// statistics of the tempered distribution softmax(z / T) -- its log-partition
// logZ_T = m / T + ln sum e^((z-m)/T) and entropy H_T -- and gathers the logit
// z_{parent(j)}[draft[j]] of every tree edge j straight from the tile's logits
// in shared memory (the Medusa/Hydra typical-acceptance inputs, Sec. 5.1/5.2).
// Warps 2-3, idle during the k-loop, find the edges whose token falls in this
// CTA's vocab tile meanwhile.
#include <math.h>
#include <stdlib.h>

#include "kernels.cuh"

namespace tv {

struct LmParams {
    CUtensorMap tmap_w;  // (d_model, vocab), box (64, 128), 128B swizzle
    CUtensorMap tmap_h;  // (d_model, rows),  box (64, R_pad), 128B swizzle
    int R, R_pad, D, V;
    int n_tiles, n_kblocks, stages, tmem_cols;
    int bps;             // 64-column boxes per pipeline stage
    int group_size, n_groups;
    float4 *part_tile;   // [n_tiles][R_pad]  (max, argmax bits, s, t)
    float4 *part_group;  // [n_groups][R_pad]
    int *counters;       // [n_groups + 1], zero between launches
    int *status;
    int expire_wait;     // test hook: the epilogue waits on a barrier nothing arrives on
    int32_t *argmax;
    float *top1;
    float *entropy;
    // typical-acceptance mode
    float inv_t;          // 1 / T
    float2 *part_tile_t;  // [n_tiles][R_pad]  (sT, tT)
    float2 *part_group_t; // [n_groups][R_pad]
    float *logz_t;        // [R] m / T + ln sT
    float *ent_t;         // [R] ln sT - tT / sT
    LmGather gather;
    float *logits_out;    // typical mode, optional: [R][V] fp32 logits
};

struct RowStat {
    float m;   // running max logit
    int idx;   // its vocab index (lowest on ties)
    float s;   // sum e^(z - m)
    float t;   // sum e^(z - m) (z - m)
    float sT;  // sum e^((z - m) / T)          (typical mode)
    float tT;  // sum e^((z - m) / T) (z - m) / T
};

constexpr float kLog2e = 1.4426950408889634f;

// Threads per CTA: warp 0 lane 0 issues TMA, warp 1 lane 0 the MMAs; all eight
// warps then share the epilogue (warps w and w + 4 read the same TMEM lane
// quadrant and split its columns) and the per-row scans.
constexpr int kLmThreads = 256;

__device__ __forceinline__ RowStat stat_empty()
{
    return RowStat{-INFINITY, 0x7fffffff, 0.f, 0.f, 0.f, 0.f};
}

// Combines the statistics of two disjoint vocab subsets.
template <bool kTyp>
__device__ __forceinline__ RowStat stat_merge(RowStat a, RowStat b, float inv_t)
{
    if (b.m > a.m || (b.m == a.m && b.idx < a.idx)) {
        RowStat x = a;
        a = b;
        b = x;
    }
    if (b.s == 0.f)
        return a;
    const float delta = b.m - a.m;  // <= 0
    const float e = ex2_approx(delta * kLog2e);
    a.s += b.s * e;
    a.t += (b.t + delta * b.s) * e;
    if constexpr (kTyp) {
        const float dT = delta * inv_t;
        const float eT = ex2_approx(dT * kLog2e);
        a.sT += b.sT * eT;
        a.tT += (b.tT + dT * b.sT) * eT;
    }
    return a;
}

template <bool kTyp>
__device__ __forceinline__ RowStat stat_shfl_xor(RowStat a, int mask)
{
    RowStat b;
    b.m = __shfl_xor_sync(0xffffffffu, a.m, mask);
    b.idx = __shfl_xor_sync(0xffffffffu, a.idx, mask);
    b.s = __shfl_xor_sync(0xffffffffu, a.s, mask);
    b.t = __shfl_xor_sync(0xffffffffu, a.t, mask);
    if constexpr (kTyp) {
        b.sT = __shfl_xor_sync(0xffffffffu, a.sT, mask);
        b.tT = __shfl_xor_sync(0xffffffffu, a.tT, mask);
    }
    return b;
}

__device__ __forceinline__ float4 stat_pack(RowStat a)
{
    return make_float4(a.m, __int_as_float(a.idx), a.s, a.t);
}

__device__ __forceinline__ RowStat stat_unpack(float4 v)
{
    return RowStat{v.x, __float_as_int(v.y), v.z, v.w, 0.f, 0.f};
}

// Threads per row for per-row scans by the CTA's threads: the largest power
// of two with tpr x R_pad <= blockDim.x, at most 8 (the transposed tile's row
// stride 128 + tpr is sized for 8).
__device__ __forceinline__ int threads_per_row(int R_pad)
{
    int tpr = 1;
    while (tpr < 8 && tpr * 2 * R_pad <= (int)blockDim.x)
        tpr *= 2;
    return tpr;
}

// Combines the statistics held by the tpr consecutive lanes of each row group.
template <bool kTyp>
__device__ __forceinline__ RowStat group_merge(RowStat st, int tpr, float inv_t)
{
    for (int m = 1; m < tpr; m <<= 1)
        st = stat_merge<kTyp>(st, stat_shfl_xor<kTyp>(st, m), inv_t);
    return st;
}

// Writes the draft-token logit of tree edge (sequence b, node j) when its
// parent row lies in this launch and its token in this CTA's vocab tile.
__device__ __forceinline__ bool gather_hit(const LmGather &g, int b, int j, int R, int v0, int nvalid, int *row,
                                           int *col)
{
    const LmGatherSeq &sq = g.seq[b];
    const int r = sq.row_base + sq.tree->parent[j];
    const int c = sq.draft[j] - v0;
    *row = r;
    *col = c;
    return r >= 0 && r < R && c >= 0 && c < nvalid;
}

// Merges count x R_pad partials (global, written by other CTAs): they are
// staged in shared memory, then every row is reduced by `tpr` threads in two
// independent passes (max / first argmax, then the rescaled sums), so there is
// no serial dependency chain per row.  Writes the merged partial (dst) or the
// final per-row outputs.
template <bool kTyp>
__device__ void merge_partials(const LmParams &p, const float4 *src, const float2 *src_t, int count, float4 *sbuf,
                               float4 *dst, float2 *dst_t)
{
    // staging with eight loads in flight per thread: the partials are in L2,
    // and a load-then-store loop would pay one round trip per element
    constexpr int kInFlight = 8;
    const int n = count * p.R_pad;
    for (int i0 = threadIdx.x; i0 < n; i0 += blockDim.x * kInFlight) {
        float4 v[kInFlight];
#pragma unroll
        for (int u = 0; u < kInFlight; ++u) {
            const int i = i0 + u * (int)blockDim.x;
            if (i < n)
                v[u] = __ldcg(src + i);
        }
#pragma unroll
        for (int u = 0; u < kInFlight; ++u) {
            const int i = i0 + u * (int)blockDim.x;
            if (i < n)
                sbuf[i] = v[u];
        }
    }
    __syncthreads();
    const int tpr = threads_per_row(p.R_pad);
    const int sub = threadIdx.x % tpr;
    for (int r0 = 0; r0 < p.R; r0 += (int)blockDim.x / tpr) {
        const int r = r0 + threadIdx.x / tpr;
        RowStat st = stat_empty();
        if (r < p.R) {
            for (int k = sub; k < count; k += tpr) {
                const float4 v = sbuf[k * p.R_pad + r];
                const int idx = __float_as_int(v.y);
                if (v.z > 0.f && (v.x > st.m || (v.x == st.m && idx < st.idx))) {
                    st.m = v.x;
                    st.idx = idx;
                }
            }
            if (st.idx != 0x7fffffff) {
                for (int k0 = sub; k0 < count; k0 += tpr * kInFlight) {
                    // the tempered sums are read once, straight from L2, eight at a time
                    float2 w[kInFlight];
                    if constexpr (kTyp) {
#pragma unroll
                        for (int u = 0; u < kInFlight; ++u) {
                            const int k = k0 + u * tpr;
                            w[u] = k < count ? __ldcg(src_t + (size_t)k * p.R_pad + r) : make_float2(0.f, 0.f);
                        }
                    }
#pragma unroll
                    for (int u = 0; u < kInFlight; ++u) {
                        const int k = k0 + u * tpr;
                        if (k >= count)
                            break;
                        const float4 v = sbuf[k * p.R_pad + r];
                        if (v.z > 0.f) {
                            const float delta = v.x - st.m;
                            const float e = ex2_approx(delta * kLog2e);
                            st.s += v.z * e;
                            st.t += (v.w + delta * v.z) * e;
                            if constexpr (kTyp) {
                                const float dT = delta * p.inv_t;
                                const float eT = ex2_approx(dT * kLog2e);
                                st.sT += w[u].x * eT;
                                st.tT += (w[u].y + dT * w[u].x) * eT;
                            }
                        }
                    }
                }
            }
        }
        st = group_merge<kTyp>(st, tpr, p.inv_t);
        if (sub == 0 && r < p.R) {
            if (dst) {
                dst[r] = stat_pack(st);
                if constexpr (kTyp)
                    dst_t[r] = make_float2(st.sT, st.tT);
            } else {
                p.argmax[r] = st.idx;
                p.top1[r] = 1.0f / st.s;
                p.entropy[r] = logf(st.s) - st.t / st.s;
                if constexpr (kTyp) {
                    const float ls = logf(st.sT);
                    p.logz_t[r] = st.m * p.inv_t + ls;
                    p.ent_t[r] = ls - st.tT / st.sT;
                }
            }
        }
    }
    __syncthreads();
}

template <bool kTyp>
__global__ void __launch_bounds__(kLmThreads, 1) k2_lm_head(const __grid_constant__ LmParams p)
{
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t full_bar[8];
    __shared__ __align__(8) uint64_t empty_bar[8];
    __shared__ __align__(8) uint64_t acc_bar;
    __shared__ __align__(8) uint64_t never_bar;
    __shared__ uint32_t tmem_slot;
    __shared__ int abort_flag;
    __shared__ int ticket;
    // typical mode: edges whose draft token lies in this tile, packed as
    // (seq << 24) | (node << 16) | (row << 7) | col; overflow -> rescan in the epilogue
    constexpr int kHitCap = 64;
    __shared__ int s_hit[kTyp ? kHitCap : 1];
    __shared__ int s_nhit;

    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int S = p.stages;
    const int B = p.bps;
    const uint32_t hb = (uint32_t)p.R_pad * 128u;  // one hidden-row box
    const uint32_t w_stage = 16384u * B, h_stage = hb * B;
    uint8_t *sW = smem;
    uint8_t *sH = smem + (size_t)S * w_stage;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int tile = blockIdx.x;
    const int v0 = tile * 128;
    const int nk = p.n_kblocks;  // stages of B boxes

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&full_bar[s], 1);
            mbar_init(&empty_bar[s], 1);
        }
        mbar_init(&acc_bar, 1);
        mbar_init(&never_bar, 1);
        abort_flag = 0;
        s_nhit = 0;
        fence_mbar_init();
        prefetch_tmap(&p.tmap_w);
        prefetch_tmap(&p.tmap_h);
    }
    if (warp == 1) {
        tmem_alloc(&tmem_slot, (uint32_t)p.tmem_cols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;

    if (warp == 0 && lane == 0) {
        // ---------------- TMA producer: one stage = B adjacent 64-column boxes of
        // W (128 rows) and of the hidden rows, so each W row is fetched as a
        // contiguous run of B x 128 bytes.
        // Tiles start their k-loop at different stages so that the CTAs in
        // flight read W rows at spread-out column offsets.
        const int rot = (int)(((long long)tile * 5) % nk);
        int issued = 0;
        for (int kb = 0; kb < nk; ++kb) {
            const int s = kb % S;
            const uint32_t ph = (uint32_t)(kb / S) & 1u;
            if (!mbar_wait_bounded(&empty_bar[s], ph ^ 1u, &abort_flag, p.status))
                break;
            const int kx = (kb + rot) % nk;
            mbar_arrive_expect_tx(&full_bar[s], w_stage + h_stage);
            for (int b = 0; b < B; ++b) {
                const int x = (kx * B + b) * 64;
                tma_load_2d(sW + (size_t)s * w_stage + (size_t)b * 16384, &p.tmap_w, &full_bar[s], x, v0);
                tma_load_2d(sH + (size_t)s * h_stage + (size_t)b * hb, &p.tmap_h, &full_bar[s], x, 0);
            }
            issued = kb + 1;
        }
        if (issued < nk) {
            // gave up: let the copies already in flight land before the CTA exits
            for (int kb = (issued > S ? issued - S : 0); kb < issued; ++kb)
                mbar_wait_drain(&full_bar[kb % S], (uint32_t)(kb / S) & 1u);
        }
    } else if (warp == 1 && lane == 0) {
        // ---------------- MMA issuer
        constexpr uint32_t kIdescM = 128;
        const uint32_t idesc = idesc_bf16_f32(kIdescM, p.R_pad);
        for (int kb = 0; kb < nk; ++kb) {
            const int s = kb % S;
            const uint32_t ph = (uint32_t)(kb / S) & 1u;
            if (!mbar_wait_bounded(&full_bar[s], ph, &abort_flag, p.status))
                break;
            tc_fence_after();
            for (int b = 0; b < B; ++b) {
                const uint32_t a_base = smem_u32(sW + (size_t)s * w_stage + (size_t)b * 16384);
                const uint32_t b_base = smem_u32(sH + (size_t)s * h_stage + (size_t)b * hb);
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    const uint64_t a = smem_desc_sw128(a_base + k * 32, 0, 1024);
                    const uint64_t bd = smem_desc_sw128(b_base + k * 32, 0, 1024);
                    tc_mma_f16_ss(tmem, a, bd, idesc, (kb | b | k) != 0 ? 1u : 0u);
                }
            }
            tc_commit(&empty_bar[s]);
        }
        tc_commit(&acc_bar);
    } else if (kTyp && warp >= 2) {
        // ---------------- edges to gather (warps 2.. are otherwise idle here)
        const int nvalid = min(128, p.V - v0);
        const int helpers = (int)blockDim.x - 64;
        for (int b = 0; b < p.gather.n_seq; ++b) {
            for (int j = 1 + (threadIdx.x - 64); j < p.gather.seq[b].n; j += helpers) {
                int row, col;
                if (gather_hit(p.gather, b, j, p.R, v0, nvalid, &row, &col)) {
                    const int slot = atomicAdd(&s_nhit, 1);
                    if (slot < kHitCap)
                        s_hit[slot] = (b << 24) | (j << 16) | (row << 7) | col;
                }
            }
        }
    }
    __syncwarp();

    // ---------------- epilogue: TMEM -> shared (transposed) -> per-row stats
    mbar_wait_bounded(p.expire_wait ? &never_bar : &acc_bar, 0, &abort_flag, p.status);
    tc_fence_after();
    __syncthreads();
    const bool ok = (abort_flag == 0);
    // logits[r][v] at r * ld + v; the row stride 128 + tpr keeps both the
    // column writes below and the per-row scans free of bank conflicts.
    const int tpr = threads_per_row(p.R_pad);
    const int ld = 128 + tpr;
    float *logits = reinterpret_cast<float *>(smem);  // aliases the drained ring
    if (ok) {
        // warps w and w + 4 read TMEM lane quadrant w % 4 (vocab rows 32 (w % 4) ..)
        // and split the columns (tree rows) in alternate 16-column chunks
        const int quad = warp & 3, half = warp >> 2, halves = (int)blockDim.x >> 7;
        const uint32_t row_addr = tmem + ((uint32_t)(32 * quad) << 16);
        for (int c0 = 16 * half; c0 < p.R_pad; c0 += 16 * halves) {
            uint32_t r[16];
            tmem_ld_32x32b_x16(row_addr + (uint32_t)c0, r);
            tmem_ld_wait();
#pragma unroll
            for (int j = 0; j < 16; ++j)
                logits[(c0 + j) * ld + 32 * quad + lane] = __uint_as_float(r[j]);
        }
    } else if (warp == 1 && lane == 0) {
        mbar_wait_drain(&acc_bar, 0);  // MMAs issued before giving up must finish before dealloc
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1)
        tmem_dealloc(tmem, (uint32_t)p.tmem_cols);
    if (!ok)
        return;

    // per-row statistics of this tile: tpr threads per row, two passes
    {
        const int sub = threadIdx.x % tpr;
        const int nvalid = min(128, p.V - v0);
        for (int r0 = 0; r0 < p.R; r0 += (int)blockDim.x / tpr) {
            const int r = r0 + threadIdx.x / tpr;
            RowStat st = stat_empty();
            if (r < p.R) {
                const float *row = logits + r * ld;
                for (int j = sub; j < nvalid; j += tpr) {
                    const float z = row[j];
                    if (z > st.m) {
                        st.m = z;
                        st.idx = v0 + j;
                    }
                }
                for (int j = sub; j < nvalid; j += tpr) {
                    const float dz = row[j] - st.m;
                    const float e = ex2_approx(dz * kLog2e);
                    st.s += e;
                    st.t += e * dz;
                    if constexpr (kTyp) {
                        const float dT = dz * p.inv_t;
                        const float eT = ex2_approx(dT * kLog2e);
                        st.sT += eT;
                        st.tT += eT * dT;
                    }
                }
            }
            st = group_merge<kTyp>(st, tpr, p.inv_t);
            if (sub == 0 && r < p.R) {
                p.part_tile[(size_t)tile * p.R_pad + r] = stat_pack(st);
                if constexpr (kTyp)
                    p.part_tile_t[(size_t)tile * p.R_pad + r] = make_float2(st.sT, st.tT);
            }
        }
        if constexpr (kTyp) {
            if (p.logits_out) {
                // whole logit rows for speculative sampling: 128 consecutive floats per row
                for (int e = threadIdx.x; e < p.R * 128; e += blockDim.x) {
                    const int r = e >> 7, j = e & 127;
                    if (j < nvalid)
                        p.logits_out[(size_t)r * p.V + v0 + j] = logits[r * ld + j];
                }
            }
            const int nhit = s_nhit;
            if (nhit <= kHitCap) {
                for (int i = threadIdx.x; i < nhit; i += blockDim.x) {
                    const int w = s_hit[i];
                    const int b = w >> 24, j = (w >> 16) & 0xff, row = (w >> 7) & 0x1ff, col = w & 0x7f;
                    p.gather.seq[b].out[j] = logits[row * ld + col];
                }
            } else {
                for (int b = 0; b < p.gather.n_seq; ++b)
                    for (int j = 1 + threadIdx.x; j < p.gather.seq[b].n; j += blockDim.x) {
                        int row, col;
                        if (gather_hit(p.gather, b, j, p.R, v0, nvalid, &row, &col))
                            p.gather.seq[b].out[j] = logits[row * ld + col];
                    }
            }
        }
    }

    // ---------------- two-level merge by arrival tickets
    __threadfence();
    __syncthreads();
    const int g = tile / p.group_size;
    const int g_first = g * p.group_size;
    const int g_count = min(p.group_size, p.n_tiles - g_first);
    if (threadIdx.x == 0)
        ticket = atomicAdd(&p.counters[g], 1);
    __syncthreads();
    if (ticket != g_count - 1)
        return;
    __threadfence();
    float4 *sbuf = reinterpret_cast<float4 *>(smem);
    merge_partials<kTyp>(p, p.part_tile + (size_t)g_first * p.R_pad, p.part_tile_t + (size_t)g_first * p.R_pad,
                         g_count, sbuf, p.part_group + (size_t)g * p.R_pad, p.part_group_t + (size_t)g * p.R_pad);
    if (threadIdx.x == 0)
        p.counters[g] = 0;
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0)
        ticket = atomicAdd(&p.counters[p.n_groups], 1);
    __syncthreads();
    if (ticket != p.n_groups - 1)
        return;
    __threadfence();
    merge_partials<kTyp>(p, p.part_group, p.part_group_t, p.n_groups, sbuf, nullptr, nullptr);
    if (threadIdx.x == 0)
        p.counters[p.n_groups] = 0;
}

// ----------------------------------------------------------------------------
// host side

static int ceil_div(int a, int b)
{
    return (a + b - 1) / b;
}

// 64-column boxes per pipeline stage.  Measured on GB300 (V=32000 and 128256,
// 26-200 rows): one or two boxes per stage are within 3%; four boxes cost
// stages and lose; so one box, the deepest ring.
static int lm_boxes_per_stage(int R_pad)
{
    (void)R_pad;
    return 1;
}

LmPlan lm_plan(int R, int D, int V)
{
    LmPlan pl{};
    pl.R_pad = ceil_div(R, 16) * 16;
    pl.n_tiles = ceil_div(V, 128);
    pl.bps = lm_boxes_per_stage(pl.R_pad);
    pl.n_kblocks = ceil_div(D, 64 * pl.bps);
    const int stage_bytes = (16384 + pl.R_pad * 128) * pl.bps;
    // Up to 64 rows two CTAs share an SM (110 KB each); wider rows need a
    // transpose buffer that leaves one CTA per SM, so its ring takes ~200 KB.
    const size_t transpose_bytes = (size_t)pl.R_pad * (128 + 8) * 4;
    const int budget = (transpose_bytes + 1024 <= 110 * 1024) ? 110 * 1024 : 200 * 1024;
    pl.stages = budget / stage_bytes;
    if (pl.stages > 8)
        pl.stages = 8;
    if (pl.stages < 2)
        pl.stages = 2;
    int cols = 32;
    while (cols < pl.R_pad)
        cols *= 2;
    pl.tmem_cols = cols;
    int gs = 1;
    while (gs * gs < pl.n_tiles)
        ++gs;
    pl.group_size = gs;
    pl.n_groups = ceil_div(pl.n_tiles, gs);
    size_t pipe = (size_t)pl.stages * stage_bytes;
    size_t tr = (size_t)pl.R_pad * (128 + 8) * 4;
    size_t mg = (size_t)(gs > pl.n_groups ? gs : pl.n_groups) * pl.R_pad * 16;
    size_t sm = pipe;
    if (tr > sm)
        sm = tr;
    if (mg > sm)
        sm = mg;
    pl.smem_bytes = sm + 1024;
    // (max, argmax, s, t) partials, then the tempered (sT, tT) partials of typical mode
    pl.ws_bytes = ((size_t)(pl.n_tiles + pl.n_groups) * pl.R_pad * (16 + 8) + 255) / 256 * 256;
    return pl;
}

cudaError_t lm_head_launch(const void *hidden, int R, const void *W, int D, int V, int32_t *argmax, float *top1,
                           float *entropy, void *parts, int *counters, int *status, cudaStream_t stream,
                           const char **err, int expire_wait, const LmTypical *typ)
{
    const LmPlan pl = lm_plan(R, D, V);
    LmParams p{};
    if (!make_tmap_2d(&p.tmap_w, W, (uint64_t)D, (uint64_t)V, (uint64_t)D * 2, 64, 128, err))
        return cudaErrorInvalidValue;
    if (!make_tmap_2d(&p.tmap_h, hidden, (uint64_t)D, (uint64_t)R, (uint64_t)D * 2, 64, (uint32_t)pl.R_pad, err))
        return cudaErrorInvalidValue;
    p.R = R;
    p.R_pad = pl.R_pad;
    p.D = D;
    p.V = V;
    p.n_tiles = pl.n_tiles;
    p.n_kblocks = pl.n_kblocks;
    p.bps = pl.bps;
    p.stages = pl.stages;
    p.tmem_cols = pl.tmem_cols;
    p.group_size = pl.group_size;
    p.n_groups = pl.n_groups;
    p.part_tile = static_cast<float4 *>(parts);
    p.part_group = p.part_tile + (size_t)pl.n_tiles * pl.R_pad;
    p.counters = counters;
    p.status = status;
    p.argmax = argmax;
    p.top1 = top1;
    p.entropy = entropy;
    p.expire_wait = expire_wait;
    p.part_tile_t = reinterpret_cast<float2 *>(p.part_group + (size_t)pl.n_groups * pl.R_pad);
    p.part_group_t = p.part_tile_t + (size_t)pl.n_tiles * pl.R_pad;
    if (typ) {
        p.inv_t = 1.0f / typ->temperature;
        p.logz_t = typ->logz_t;
        p.ent_t = typ->ent_t;
        p.gather = typ->gather;
        p.logits_out = typ->logits_out;
        cudaError_t e = allow_max_smem((const void *)k2_lm_head<true>);
        if (e != cudaSuccess)
            return e;
        k2_lm_head<true><<<pl.n_tiles, kLmThreads, pl.smem_bytes, stream>>>(p);
    } else {
        p.inv_t = 1.0f;
        cudaError_t e = allow_max_smem((const void *)k2_lm_head<false>);
        if (e != cudaSuccess)
            return e;
        k2_lm_head<false><<<pl.n_tiles, kLmThreads, pl.smem_bytes, stream>>>(p);
    }
    return cudaGetLastError();
}

}  // namespace tv
