// lm_head.cu -- fused LM head with per-row greedy statistics (K2 + merge).
//
// For every tree row r: z = W h_r over the whole vocabulary, reduced on the
// fly to (max, argmax, s = sum e^(z-max), t = sum e^(z-max)(z-max)); logits
// never reach memory.  top1 = 1/s, entropy = ln s - t/s (nats).
// These are the verifier's greedy token, the base-LM top-1 probability p0 and
// the entropy feature that the EntMTP scheduler consumes (Sec. 4, "Path-value
// score" and "Cost": computed from the verifier logits already on chip).
//
// Design (swap-AB, persistent).  The 128-entry vocab tiles are split into
// contiguous runs over a persistent grid (two CTAs per SM when their rings fit
// side by side, one otherwise); a CTA walks its run tile by tile.  The tile of W
// ([128][64] bf16 per k-block, 128-byte swizzled by TMA) is the MMA's M=128 A
// operand, the tree rows ([R_pad][64], same swizzle) the N = R_pad B operand;
// tcgen05.mma (kind::f16, f32 accumulate) builds the 128 x R_pad logit tile in
// TMEM.  Lane 0 of warps 0 and 10 issue TMA (alternate stages) into a ring
// that runs across tiles, warp 1 lane 0 the MMAs into one of two TMEM
// accumulators, and warps 2-9 drain the
// other accumulator meanwhile (32 tree rows at a time: TMEM -> shared memory
// transposed -> eight threads per row reduce its 128 logits), folding each
// tile into per-row running statistics of the CTA.  The CTAs' statistics are
// merged in two levels by atomic arrival tickets (the last CTA of a group
// merges the group; the last group merges everything); no CTA ever waits for
// another.
//
#include <atomic>
#include <math.h>
#include <stdlib.h>

#include "kernels.cuh"

namespace tv {

struct LmParams {
    CUtensorMap tmap_w;  // (d_model, vocab), box (64, 128), 128B swizzle
    CUtensorMap tmap_h;  // (d_model, rows),  box (64, R_pad) (R_pad / 2 for CTA pairs), 128B swizzle
    int R, R_pad, D, V;
    int n_tiles, nk, stages, acc_cols;  // tiles of 128 vocab entries (256 for CTA pairs)
    int P;               // CTAs
    int units;           // the tile split's units: CTAs, or CTA pairs
    int group_size, n_groups;
    size_t smem_avail;   // dynamic shared memory after alignment (the merges stage partials there)
    float4 *part_cta;    // [P][R_pad]  (max, argmax bits, s, t)
    float4 *part_group;  // [n_groups][R_pad]
    float2 *part_cta_t;  // [P][R_pad]  (sT, tT), typical mode
    float2 *part_group_t;
    int *counters;       // [n_groups + 1] group tickets, zero between launches
    int *status;
    int expire_wait;     // test hook: the epilogue waits on a barrier nothing arrives on
    int32_t *argmax;
    float *top1;
    float *entropy;
    // typical-acceptance mode
    float inv_t;          // 1 / T
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

// Threads per CTA: lane 0 of warps 0 and 10 issue TMA, warp 1 lane 0 the
// MMAs, warps 2-9 form the epilogue (warps w and w + 4 read the same TMEM
// lane quadrant w % 4 and split each 32-row chunk's columns); all eleven merge
// at the end.
constexpr int kLmThreads = 352;
constexpr int kLmProducer2 = 10;
constexpr int kEpiThreads = 256;
constexpr int kLmChunk = 32;             // tree rows per epilogue chunk
constexpr int kLmTpr = kEpiThreads / kLmChunk;  // threads per row in the chunk scans
constexpr int kChunkLd = 128 + kLmTpr;   // chunk row stride (floats): conflict-free writes and scans

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

// Threads per row for the merges of partial statistics by all of the CTA's
// threads: the largest power of two with tpr x R_pad <= blockDim.x, at most 8
// (a row's partials are few, so more threads per row would mostly idle).
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
    if (!in_bounds((size_t)n * sizeof(float4) <= p.smem_avail, p.status))
        return;
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

// Arrival ticket of this CTA on `counter` once its writes are done: the
// barrier orders every thread's writes before thread 0's fence (fences are
// cumulative), and the fence orders them before the atomic, so the CTA that
// draws the last ticket -- after a fence of its own -- reads all of them.
// Returns true in every thread of that CTA.
__device__ __forceinline__ bool arrive_last(int *counter, int expected, int *s_ticket)
{
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        const int t = atomicAdd(counter, 1);
        if (t == expected - 1)
            __threadfence();
        *s_ticket = t;
    }
    __syncthreads();
    return *s_ticket == expected - 1;
}

// Named barrier of the eight epilogue warps.
__device__ __forceinline__ void epi_sync()
{
    asm volatile("bar.sync 1, 256;" ::: "memory");
}

// First vocab tile of unit c's run.
__device__ __forceinline__ int lm_tile_begin(const LmParams &p, int c)
{
    return (int)((long long)c * p.n_tiles / p.units);
}

// Step j of a tile's k-loop reads k-block j + lm_rot (mod nk): the order is
// rotated by the tile index, so the CTAs in flight read their W rows at
// spread-out column offsets rather than all at the same one.
__device__ __forceinline__ int lm_rot(const LmParams &p, int tile)
{
    return (int)(((long long)tile * 5) % p.nk);
}

// A producer thread's position in the ring: the k-block sequence g = g0,
// g0 + 2, ... of a run, as (tile, k-block) and (ring slot, phase parity),
// advanced without divisions.
struct RingCursor {
    int tile, j, kb, rot, slot;
    uint32_t phase;
    __device__ RingCursor(const LmParams &p, int tile0, int g0) : tile(tile0), j(g0), slot(g0), phase(0)
    {
        // g0 is 0 or 1; the ring has at least two slots
        while (j >= p.nk) {
            j -= p.nk;
            ++tile;
        }
        rot = lm_rot(p, tile);
        kb = j + rot >= p.nk ? j + rot - p.nk : j + rot;
    }
    __device__ __forceinline__ void advance2(const LmParams &p, int S)
    {
        slot += 2;
        if (slot >= S) {
            slot -= S;
            phase ^= 1u;
        }
        j += 2;
        if (j >= p.nk) {
            while (j >= p.nk) {
                j -= p.nk;
                ++tile;
            }
            rot = lm_rot(p, tile);
        }
        kb = j + rot >= p.nk ? j + rot - p.nk : j + rot;
    }
};

// Waits, when it goes out of scope (every exit of the kernel), for the
// stream's previous kernel to complete.  In a verification step the LM head
// runs beside the attention without depending on it; this keeps the step's
// acceptance kernel, which waits for the LM head, ordered after the attention
// as well.
struct PdlWaitOnExit {
    __device__ ~PdlWaitOnExit() { pdl_wait(); }
};

// kPair: CTA pairs (clusters of two) share each MMA (tcgen05 cta_group::2, M =
// 256): a pair tile is 256 vocab entries, 128 per CTA, and each CTA stages only
// half of the tree rows, so a stage moves 16 KB of W plus half the rows' box
// through each SM's shared memory instead of the whole box.  The even CTA
// issues the MMAs; both CTAs' TMA loads complete on its stage barriers, its
// commits arrive on both CTAs' barriers, and both CTAs' epilogues release its
// accumulators.  Used for wide rows, where a CTA holds an SM alone.
template <bool kTyp, bool kPair>
__global__ void __launch_bounds__(kLmThreads, 2) k2_lm_head(const __grid_constant__ LmParams p)
{
    // the acceptance kernel that reads this kernel's outputs may be launched now
    pdl_trigger();
    PdlWaitOnExit pdl_exit;
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t full_bar[8];
    __shared__ __align__(8) uint64_t empty_bar[8];
    __shared__ __align__(8) uint64_t acc_full[2], acc_empty[2];
    __shared__ __align__(8) uint64_t drain_bar, never_bar;
    __shared__ uint32_t tmem_slot;
    __shared__ int abort_flag;
    // CTA pairs: the stage sequences each producer thread issued, this CTA's and the odd CTA's
    __shared__ long long s_gend[2], s_peer_gend[2];
    __shared__ int s_ticket, s_ok;
    // typical mode: edges whose draft token lies in the current tile, packed as
    // (seq << 24) | (node << 16) | (row << 7) | col; overflow -> rescan per chunk
    constexpr int kHitCap = 64;
    __shared__ int s_hit[kTyp ? kHitCap : 1];
    __shared__ int s_nhit;

    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int S = p.stages;
    // one 64-column box of this CTA's tree rows (half of them in a pair)
    const uint32_t hb = (uint32_t)(kPair ? p.R_pad / 2 : p.R_pad) * 128u;
    const uint32_t stage_bytes = 16384u + hb;
    uint8_t *ring = smem;
    float *chunk = reinterpret_cast<float *>(smem + (size_t)S * stage_bytes);  // [kLmChunk][kChunkLd]
    RowStat *run = reinterpret_cast<RowStat *>(chunk + kLmChunk * kChunkLd);   // [R_pad] running statistics

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int c = blockIdx.x;
    // the unit of the tile split: a CTA, or a pair; tiles are 128 (256 for a pair) vocab entries
    const uint32_t rank = kPair ? cluster_ctarank() : 0u;
    const bool leader = rank == 0;
    const int unit = kPair ? c >> 1 : c;
    const int tile0 = lm_tile_begin(p, unit), tile1 = lm_tile_begin(p, unit + 1);

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&full_bar[s], 1);
            mbar_init(&empty_bar[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&acc_full[b], 1);
            mbar_init(&acc_empty[b], (kEpiThreads / 32) * (kPair ? 2 : 1));  // a pair's epilogues release the even CTA's
        }
        mbar_init(&drain_bar, 1);
        mbar_init(&never_bar, 1);
        abort_flag = 0;
        s_gend[0] = s_gend[1] = s_peer_gend[0] = s_peer_gend[1] = 0;
        fence_mbar_init();
        prefetch_tmap(&p.tmap_w);
        prefetch_tmap(&p.tmap_h);
    }
    if (warp == 1) {
        if constexpr (kPair) {
            tmem_alloc_pair(&tmem_slot, 2u * (uint32_t)p.acc_cols);
            tmem_relinquish_pair();
        } else {
            tmem_alloc(&tmem_slot, 2u * (uint32_t)p.acc_cols);
            tmem_relinquish();
        }
    }
    for (int r = threadIdx.x; r < p.R_pad; r += blockDim.x)
        run[r] = stat_empty();
    tc_fence_before();
    __syncthreads();
    if constexpr (kPair)
        cluster_barrier();  // both CTAs' barriers are initialised before either CTA signals the other's
    tc_fence_after();
    const uint32_t tmem = tmem_slot;

    if (warp == 0 || warp == kLmProducer2) {
        // ---------------- TMA producers: one stage = one 64-column box of W
        // (128 rows) and of the tree rows; the ring runs across the run's tiles.
        // Warp 0 fills the even stages of the sequence, the last warp the odd
        // ones: one issuing thread alone streams W measurably slower.
        if (lane == 0) {
            const int mine = warp == 0 ? 0 : 1;
            const long long G = (long long)(tile1 - tile0) * p.nk;  // the run's k-blocks
            RingCursor cur(p, tile0, mine);  // this thread's steps g = mine, mine + 2, ...
            long long g_end = 0;
            bool ok = true;
            for (long long g = mine; g < G; g += 2, cur.advance2(p, S)) {
                const int s = cur.slot, tile = cur.tile, kb = cur.kb;
                if (!mbar_wait_bounded(&empty_bar[s], cur.phase ^ 1u, &abort_flag, p.status)) {
                    ok = false;
                    break;
                }
                if constexpr (kPair) {
                    // the stage's four boxes (W and tree rows of both CTAs) complete on the even CTA's barrier
                    if (leader)
                        mbar_arrive_expect_tx(&full_bar[s], 2 * stage_bytes);
                    const uint32_t fb = cluster_addr(&full_bar[s], 0);
                    tma_load_2d_pair(ring + (size_t)s * stage_bytes, &p.tmap_w, fb, kb * 64,
                                     tile * 256 + (int)rank * 128);
                    tma_load_2d_pair(ring + (size_t)s * stage_bytes + 16384, &p.tmap_h, fb, kb * 64,
                                     (int)rank * (p.R_pad / 2));
                } else {
                    mbar_arrive_expect_tx(&full_bar[s], stage_bytes);
                    tma_load_2d(ring + (size_t)s * stage_bytes, &p.tmap_w, &full_bar[s], kb * 64, tile * 128);
                    tma_load_2d(ring + (size_t)s * stage_bytes + 16384, &p.tmap_h, &full_bar[s], kb * 64, 0);
                }
                g_end = g + 1;
            }
            s_gend[mine] = g_end;
            // Gave up: this thread's copies in flight land before the CTA exits.  (In a
            // pair, the even CTA drains both CTAs' copies at the teardown.)
            if (!ok && !kPair)
                for (long long it = (g_end > S ? g_end - S : 0); it < g_end; ++it)
                    if ((it & 1) == mine)
                        mbar_wait_drain(&full_bar[it % S], (uint32_t)(it / S) & 1u);
        }
    } else if (warp == 1) {
        // ---------------- MMA issuer: the CTA's i-th tile accumulates into TMEM buffer i & 1
        // (in a pair, the even CTA issues for both)
        if (lane == 0 && leader) {
            const uint32_t idesc = idesc_bf16_f32(kPair ? 256 : 128, p.R_pad);
            int s = 0;          // ring slot of the next k-block
            uint32_t ph = 0;    // and its phase parity
            bool ok = true;
            for (int tile = tile0, i = 0; tile < tile1 && ok; ++tile, ++i) {
                const int b = i & 1;
                if (!mbar_wait_bounded(&acc_empty[b], ((uint32_t)(i >> 1) & 1u) ^ 1u, &abort_flag, p.status))
                    break;
                tc_fence_after();
                const uint32_t d = tmem + (uint32_t)(b * p.acc_cols);
                for (int j = 0; j < p.nk; ++j) {
                    if (!mbar_wait_bounded(&full_bar[s], ph, &abort_flag, p.status)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t a_base = smem_u32(ring + (size_t)s * stage_bytes);
                    const uint32_t b_base = a_base + 16384u;
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        const uint64_t ad = smem_desc_sw128(a_base + k * 32, 0, 1024);
                        const uint64_t bd = smem_desc_sw128(b_base + k * 32, 0, 1024);
                        if constexpr (kPair)
                            tc_mma_f16_ss_pair(d, ad, bd, idesc, (j != 0 || k != 0) ? 1u : 0u);
                        else
                            tc_mma_f16_ss(d, ad, bd, idesc, (j != 0 || k != 0) ? 1u : 0u);
                    }
                    if constexpr (kPair)
                        tc_commit_pair(&empty_bar[s]);
                    else
                        tc_commit(&empty_bar[s]);
                    if (++s == S) {
                        s = 0;
                        ph ^= 1u;
                    }
                }
                if (!ok)
                    break;
                if constexpr (kPair)
                    tc_commit_pair(&acc_full[b]);
                else
                    tc_commit(&acc_full[b]);
            }
            // arrives when every MMA issued above has retired (waited for before TMEM is released)
            if constexpr (kPair)
                tc_commit_pair(&drain_bar);
            else
                tc_commit(&drain_bar);
        }
    } else if (warp < kLmProducer2) {
        // ---------------- epilogue (warps 2-9)
        const int e = threadIdx.x - 64;
        const int q = warp & 3, half = (warp - 2) >> 2;
        const int vr = 32 * q + lane;                 // this thread's vocab entry within the tile (TMEM lane)
        const int sub = e % kLmTpr, rloc = e / kLmTpr;  // chunk scans: kLmTpr threads per row
        // the same verdict for all epilogue threads: did every wait so far succeed?
        auto agree = [&]() -> bool {
            epi_sync();
            if (e == 0)
                s_ok = (abort_flag == 0);
            epi_sync();
            return s_ok != 0;
        };
        for (int tile = tile0, i = 0; tile < tile1; ++tile, ++i) {
            const int b = i & 1;
            mbar_wait_bounded(p.expire_wait ? &never_bar : &acc_full[b], (uint32_t)(i >> 1) & 1u, &abort_flag,
                              p.status);
            if (!agree())
                break;
            tc_fence_after();
            // this CTA's 128 vocab entries (the odd CTA of a pair's last tile may have none)
            const int v0 = kPair ? tile * 256 + (int)rank * 128 : tile * 128, nvalid = min(128, p.V - v0);
            if constexpr (kTyp) {
                // the tree edges whose draft token lies in this tile
                if (e == 0)
                    s_nhit = 0;
                epi_sync();
                for (int bq = 0; bq < p.gather.n_seq; ++bq)
                    for (int j = 1 + e; j < p.gather.seq[bq].n; j += kEpiThreads) {
                        int row, col;
                        if (gather_hit(p.gather, bq, j, p.R, v0, nvalid, &row, &col)) {
                            const int h = atomicAdd(&s_nhit, 1);
                            if (h < kHitCap)
                                s_hit[h] = (bq << 24) | (j << 16) | (row << 7) | col;
                        }
                    }
                epi_sync();
            }
            const uint32_t acc = tmem + (uint32_t)(b * p.acc_cols) + ((uint32_t)(32 * q) << 16);
            for (int c0 = 0; c0 < p.R_pad; c0 += kLmChunk) {
                const int col = c0 + 16 * half;  // this warp's 16 tree rows of the chunk
                uint32_t v[16];
                if (col < p.R_pad) {
                    tmem_ld_32x32b_x16(acc + (uint32_t)col, v);
                    tmem_ld_wait();
                }
                if (c0 + kLmChunk >= p.R_pad) {
                    // last read of this accumulator: the MMAs of segment i + 2 may reuse it
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) {
                        if constexpr (kPair)
                            mbar_arrive_cluster(cluster_addr(&acc_empty[b], 0));
                        else
                            mbar_arrive(&acc_empty[b]);
                    }
                }
                if (col < p.R_pad) {
#pragma unroll
                    for (int j = 0; j < 16; ++j)
                        chunk[(16 * half + j) * kChunkLd + vr] = __uint_as_float(v[j]);
                }
                epi_sync();
                // rows c0 .. c0 + 31: two passes (max / first argmax, then the sums)
                const int r = c0 + rloc;
                RowStat st = stat_empty();
                if (r < p.R) {
                    const float *row = chunk + rloc * kChunkLd;
                    for (int j = sub; j < nvalid; j += kLmTpr) {
                        const float z = row[j];
                        if (z > st.m) {
                            st.m = z;
                            st.idx = v0 + j;
                        }
                    }
                    for (int j = sub; j < nvalid; j += kLmTpr) {
                        const float dz = row[j] - st.m;
                        const float ex = ex2_approx(dz * kLog2e);
                        st.s += ex;
                        st.t += ex * dz;
                        if constexpr (kTyp) {
                            const float dT = dz * p.inv_t;
                            const float eT = ex2_approx(dT * kLog2e);
                            st.sT += eT;
                            st.tT += eT * dT;
                        }
                    }
                }
                st = group_merge<kTyp>(st, kLmTpr, p.inv_t);
                if (sub == 0 && r < p.R)
                    run[r] = stat_merge<kTyp>(run[r], st, p.inv_t);
                if constexpr (kTyp) {
                    const int nhit = s_nhit;
                    if (nhit <= kHitCap) {
                        for (int h = e; h < nhit; h += kEpiThreads) {
                            const int w = s_hit[h];
                            const int row = (w >> 7) & 0x1ff;
                            if (row >= c0 && row < c0 + kLmChunk &&
                                in_bounds((w >> 24) < p.gather.n_seq && ((w >> 16) & 0xff) < p.gather.seq[w >> 24].n,
                                          p.status))
                                p.gather.seq[w >> 24].out[(w >> 16) & 0xff] = chunk[(row - c0) * kChunkLd + (w & 0x7f)];
                        }
                    } else {
                        for (int bq = 0; bq < p.gather.n_seq; ++bq)
                            for (int j = 1 + e; j < p.gather.seq[bq].n; j += kEpiThreads) {
                                int row, cc;
                                if (gather_hit(p.gather, bq, j, p.R, v0, nvalid, &row, &cc) && row >= c0 &&
                                    row < c0 + kLmChunk)
                                    p.gather.seq[bq].out[j] = chunk[(row - c0) * kChunkLd + cc];
                            }
                    }
                    if (p.logits_out) {
                        // whole logit rows for speculative sampling: 128 consecutive floats per row
                        for (int x = e; x < kLmChunk * 128; x += kEpiThreads) {
                            const int rr = x >> 7, j = x & 127;
                            if (c0 + rr < p.R && j < nvalid)
                                p.logits_out[(size_t)(c0 + rr) * p.V + v0 + j] = chunk[rr * kChunkLd + j];
                        }
                    }
                }
                epi_sync();  // the chunk buffer is rewritten next
            }
        }
        // this CTA's statistics for the final merge
        if (!abort_flag)
            for (int r = e; r < p.R; r += kEpiThreads) {
                p.part_cta[(size_t)c * p.R_pad + r] = stat_pack(run[r]);
                if constexpr (kTyp)
                    p.part_cta_t[(size_t)c * p.R_pad + r] = make_float2(run[r].sT, run[r].tT);
            }
    }

    // ---------------- teardown: every MMA has retired before TMEM is released
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        if (lane == 0)
            mbar_wait_drain(&drain_bar, 0);
        __syncwarp();
        if constexpr (!kPair)
            tmem_dealloc(tmem, 2u * (uint32_t)p.acc_cols);
    }
    if constexpr (kPair) {
        // Both CTAs' epilogues are done with TMEM and both have seen the MMAs retire
        // before the pair frees it.  Every copy either CTA issued lands before either
        // exits: normally the MMAs consumed them all; after a give-up, the even CTA
        // arms the stages only the odd CTA filled (at most a ring's worth ahead) and
        // drains the last ring's worth of stages of each producer thread, waiting
        // with the usual bound.
        if (!leader && threadIdx.x < 2)
            st_cluster_s64(cluster_addr(&s_peer_gend[threadIdx.x], 0), s_gend[threadIdx.x]);
        cluster_barrier();
        if (warp == 1) {
            tc_fence_after();
            tmem_dealloc_pair(tmem, 2u * (uint32_t)p.acc_cols);
        }
        if (leader && threadIdx.x < 2) {
            const long long mine = threadIdx.x, gl = s_gend[mine], go = s_peer_gend[mine];
            for (long long it = gl; it < go; ++it)
                if ((it & 1) == mine)
                    mbar_arrive_expect_tx(&full_bar[it % S], stage_bytes);
            const long long ge = gl > go ? gl : go;
            if (abort_flag || gl != go)
                for (long long it = (ge > S ? ge - S : 0); it < ge; ++it)
                    if ((it & 1) == mine)
                        mbar_wait_drain(&full_bar[it % S], (uint32_t)(it / S) & 1u);
        }
        cluster_barrier();
    }
    if (abort_flag)
        return;

    // ---------------- two-level merge of the CTAs' statistics by arrival tickets
    const int g = c / p.group_size;
    const int g_first = g * p.group_size;
    const int g_count = min(p.group_size, p.P - g_first);
    if (!arrive_last(&p.counters[g], g_count, &s_ticket))
        return;
    float4 *sbuf = reinterpret_cast<float4 *>(smem);  // the drained ring
    merge_partials<kTyp>(p, p.part_cta + (size_t)g_first * p.R_pad, p.part_cta_t + (size_t)g_first * p.R_pad, g_count,
                         sbuf, p.part_group + (size_t)g * p.R_pad, p.part_group_t + (size_t)g * p.R_pad);
    if (threadIdx.x == 0)
        p.counters[g] = 0;
    if (!arrive_last(&p.counters[p.n_groups], p.n_groups, &s_ticket))
        return;
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

LmPlan lm_plan(int R, int D, int V, int n_sm, int max_pairs)
{
    LmPlan pl{};
    if (n_sm < 1)
        n_sm = 1;
    pl.R_pad = ceil_div(R, 16) * 16;
    pl.n_kblocks = ceil_div(D, 64);
    int cols = 32;
    while (cols < pl.R_pad)
        cols *= 2;
    pl.acc_cols = cols;
    const size_t fixed = (size_t)kLmChunk * kChunkLd * 4 + (size_t)pl.R_pad * sizeof(RowStat);
    // Two CTAs share an SM when each still gets a ring of at least three stages
    // in half of its shared memory and four accumulators fit in TMEM: two
    // independent TMA pipelines per SM stream W faster than one deeper ring.
    const size_t pad = 1024 + 1024;  // alignment pad, static shared memory
    const size_t half = 112 * 1024;
    const size_t stage1 = 16384 + (size_t)pl.R_pad * 128;
    const int st2 = half > fixed + pad ? (int)((half - fixed - pad) / stage1) : 0;
    pl.ctas_per_sm = (st2 >= 3 && 4 * cols <= 512) ? 2 : 1;
    // Otherwise (wide rows, one CTA per SM) CTA pairs share each MMA: each CTA
    // stages half of the rows, so the rows cross each SM's shared memory once
    // per 256 vocab entries instead of once per 128.
    if (max_pairs < 0)
        max_pairs = n_sm / 2;
    pl.pair = pl.ctas_per_sm == 1 && max_pairs >= 1;
    pl.n_tiles = ceil_div(V, pl.pair ? 256 : 128);
    const size_t stage_bytes = 16384 + (size_t)(pl.pair ? pl.R_pad / 2 : pl.R_pad) * 128;
    const size_t budget = (pl.ctas_per_sm == 2 ? half : 227 * 1024) - fixed - pad;
    pl.stages = (int)(budget / stage_bytes);
    if (pl.stages > 8)
        pl.stages = 8;
    if (pl.stages < 2)
        pl.stages = 2;
    if (pl.pair) {
        pl.units = max_pairs < pl.n_tiles ? max_pairs : pl.n_tiles;
        pl.P = 2 * pl.units;
    } else {
        const int slots = pl.ctas_per_sm * n_sm;
        pl.P = slots < pl.n_tiles ? slots : pl.n_tiles;
        pl.units = pl.P;
    }
    int gs = 1;
    while (gs * gs < pl.P)
        ++gs;
    pl.group_size = gs;
    pl.n_groups = ceil_div(pl.P, gs);
    size_t sm = (size_t)pl.stages * stage_bytes + fixed;
    const size_t mg = (size_t)(gs > pl.n_groups ? gs : pl.n_groups) * pl.R_pad * 16;
    if (mg > sm)
        sm = mg;
    pl.smem_bytes = sm + 1024;
    // (max, argmax, s, t) and (sT, tT) partials of the CTAs and the groups.  The
    // workspace also covers the plan without pairs, which a launch takes when
    // no cluster of two can be resident.
    const int slots = pl.ctas_per_sm * n_sm, n128 = ceil_div(V, 128);
    const int p1 = slots < n128 ? slots : n128;
    int gs1 = 1;
    while (gs1 * gs1 < p1)
        ++gs1;
    const int ng1 = ceil_div(p1, gs1);
    const int parts = pl.P + pl.n_groups > p1 + ng1 ? pl.P + pl.n_groups : p1 + ng1;
    pl.n_counters = (pl.n_groups > ng1 ? pl.n_groups : ng1) + 1;
    pl.ws_bytes = ((size_t)parts * pl.R_pad * (16 + 8) + 255) / 256 * 256;
    return pl;
}

// Clusters of two CTAs of k2_lm_head<kTyp, true> with `smem` bytes each that
// can be resident at once (cached per shared-memory size; 0 if none).
template <bool kTyp>
static int lm_max_pairs(size_t smem, int n_sm)
{
    static std::atomic<int> cache[24];  // by smem / 16 KB; 0: not queried yet, else pairs + 1
    const size_t slot = smem / 16384 < 24 ? smem / 16384 : 23;
    int v = cache[slot].load(std::memory_order_relaxed);
    if (v > 0)
        return v - 1;
    int pairs = 0;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(2 * (n_sm / 2 > 0 ? n_sm / 2 : 1));
    cfg.blockDim = dim3(kLmThreads);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (allow_max_smem((const void *)k2_lm_head<kTyp, true>) != cudaSuccess ||
        cudaOccupancyMaxActiveClusters(&pairs, k2_lm_head<kTyp, true>, &cfg) != cudaSuccess) {
        (void)cudaGetLastError();
        pairs = 0;
    }
    if (pairs > n_sm / 2)
        pairs = n_sm / 2;
    cache[slot].store(pairs + 1, std::memory_order_relaxed);
    return pairs;
}

template <bool kTyp>
static cudaError_t lm_launch_as(LmParams &p, const LmPlan &pl, cudaStream_t stream, bool pdl)
{
    if (pl.pair) {
        cudaError_t e = allow_max_smem((const void *)k2_lm_head<kTyp, true>);
        if (e != cudaSuccess)
            return e;
        return launch_kernel_cluster(k2_lm_head<kTyp, true>, dim3(pl.P), dim3(kLmThreads), pl.smem_bytes, stream, pdl,
                                     2, p);
    }
    cudaError_t e = allow_max_smem((const void *)k2_lm_head<kTyp, false>);
    if (e != cudaSuccess)
        return e;
    return launch_kernel(k2_lm_head<kTyp, false>, dim3(pl.P), dim3(kLmThreads), pl.smem_bytes, stream, pdl, p);
}

cudaError_t lm_head_launch(const void *hidden, int R, const void *W, int D, int V, int32_t *argmax, float *top1,
                           float *entropy, void *parts, int *counters, int *status, int n_sm, cudaStream_t stream,
                           const char **err, int expire_wait, const LmTypical *typ, bool pdl)
{
    LmPlan pl = lm_plan(R, D, V, n_sm);
    if (pl.pair) {
        // as many pairs as can be resident at once (the SMs of a cluster share a GPC)
        const int mp = typ ? lm_max_pairs<true>(pl.smem_bytes, n_sm) : lm_max_pairs<false>(pl.smem_bytes, n_sm);
        if (mp != pl.units || mp < 1)
            pl = lm_plan(R, D, V, n_sm, mp);
    }
    LmParams p{};
    if (!make_tmap_2d(&p.tmap_w, W, (uint64_t)D, (uint64_t)V, (uint64_t)D * 2, 64, 128, err))
        return cudaErrorInvalidValue;
    if (!make_tmap_2d(&p.tmap_h, hidden, (uint64_t)D, (uint64_t)R, (uint64_t)D * 2, 64,
                      (uint32_t)(pl.pair ? pl.R_pad / 2 : pl.R_pad), err))
        return cudaErrorInvalidValue;
    p.R = R;
    p.R_pad = pl.R_pad;
    p.D = D;
    p.V = V;
    p.n_tiles = pl.n_tiles;
    p.nk = pl.n_kblocks;
    p.stages = pl.stages;
    p.acc_cols = pl.acc_cols;
    p.P = pl.P;
    p.units = pl.units;
    p.group_size = pl.group_size;
    p.n_groups = pl.n_groups;
    p.smem_avail = pl.smem_bytes - 1024;
    p.part_cta = static_cast<float4 *>(parts);
    p.part_group = p.part_cta + (size_t)pl.P * pl.R_pad;
    p.part_cta_t = reinterpret_cast<float2 *>(p.part_group + (size_t)pl.n_groups * pl.R_pad);
    p.part_group_t = p.part_cta_t + (size_t)pl.P * pl.R_pad;
    p.counters = counters;
    p.status = status;
    p.argmax = argmax;
    p.top1 = top1;
    p.entropy = entropy;
    p.expire_wait = expire_wait;
    if (typ) {
        p.inv_t = 1.0f / typ->temperature;
        p.logz_t = typ->logz_t;
        p.ent_t = typ->ent_t;
        p.gather = typ->gather;
        p.logits_out = typ->logits_out;
        return lm_launch_as<true>(p, pl, stream, pdl);
    }
    p.inv_t = 1.0f;
    return lm_launch_as<false>(p, pl, stream, pdl);
}

TB_BOUNDS_COUNTER(bounds_violations_lm_head)

}  // namespace tv
