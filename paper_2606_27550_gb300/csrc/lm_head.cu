// lm_head.cu -- fused LM head with per-row greedy statistics (K2 + merge).
//
// For every tree row r: z = W h_r over the whole vocabulary, reduced on the
// fly to (max, argmax, s = sum e^(z-max), t = sum e^(z-max)(z-max)); logits
// never reach memory.  top1 = 1/s, entropy = ln s - t/s (nats).
// These are the verifier's greedy token, the base-LM top-1 probability p0 and
// the entropy feature that the EntMTP scheduler consumes (Sec. 4, "Path-value
// score" and "Cost": computed from the verifier logits already on chip).
//
// Design (swap-AB, persistent).  A persistent grid (two CTAs per SM when
// their rings fit side by side; for wide rows, clusters of two CTAs that share
// each MMA) pulls 128-entry vocab tiles (256 for a pair) dynamically: every
// unit (CTA or pair) starts on its own tile, then takes the next tile from a
// global counter, so units that start late -- on SMs that other kernels of the
// step still hold -- simply take fewer tiles.  The tile of W ([128][64] bf16
// per k-block, 128-byte swizzled by TMA) is the MMA's M=128 A operand, the
// tree rows ([R_pad][64], same swizzle) the N = R_pad B operand; tcgen05.mma
// (kind::f16, f32 accumulate) builds the 128 x R_pad logit tile in TMEM.
// Lane 0 of warps 0 and 10 issue TMA (alternate stages) into a ring that runs
// across tiles, warp 1 lane 0 the MMAs into one of two TMEM accumulators, and
// warps 2-9 drain the other accumulator meanwhile (32 tree rows at a time:
// TMEM -> shared memory transposed -> eight threads per row reduce its 128
// logits) into the tile's per-row statistics, written to the tile's own slot.
// A second kernel, k2_lm_merge (one CTA per row, launched as a programmatic
// dependent that waits for the whole grid), merges every row's slots in slot
// order, so the results do not depend on which CTA took which tile; no CTA of
// the LM head ever waits for another.
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
    int units;           // the tile split's units: CTAs, or CTA pairs
    int n_slots;         // per-tile partials: one per tile (two per pair tile, one per CTA)
    float4 *part_tile;   // [n_slots][R_pad]  (max, argmax bits, s, t)
    float2 *part_tile_t; // [n_slots][R_pad]  (sT, tT), typical mode
    int *counters;       // [1] the tile counter, zero between launches
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
constexpr int kTileQ = 4;  // tile-queue entries (a power of two)
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

// Named barrier of the eight epilogue warps.
__device__ __forceinline__ void epi_sync()
{
    asm volatile("bar.sync 1, 256;" ::: "memory");
}

// Waits on a tile-queue barrier: in a pair, the odd CTA's entries are written
// by the even CTA, so the wait acquires at cluster scope.
template <bool kPair>
__device__ __forceinline__ bool lm_wait(uint64_t *bar, uint32_t parity, volatile int *abort, int *status)
{
    if constexpr (kPair)
        return mbar_wait_bounded_cluster(bar, parity, abort, status);
    else
        return mbar_wait_bounded(bar, parity, abort, status);
}

// Step j of a tile's k-loop reads k-block j + lm_rot (mod nk): the order is
// rotated by the tile index, so the CTAs in flight read their W rows at
// spread-out column offsets rather than all at the same one.
__device__ __forceinline__ int lm_rot(const LmParams &p, int tile)
{
    return (int)(((long long)tile * 5) % p.nk);
}

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
    __shared__ __align__(8) uint64_t tq_full[kTileQ], tq_empty[kTileQ];
    __shared__ int s_tile[kTileQ];  // the CTA's i-th vocab tile in entry i % kTileQ (-1: no more)
    __shared__ uint32_t tmem_slot;
    __shared__ int abort_flag;
    // CTA pairs: the stage sequences each producer thread issued, this CTA's and the odd CTA's
    __shared__ long long s_gend[2], s_peer_gend[2];
    __shared__ int s_ok;
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

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int c = blockIdx.x;
    // the unit of the tile split: a CTA, or a pair; tiles are 128 (256 for a pair) vocab entries
    const uint32_t rank = kPair ? cluster_ctarank() : 0u;
    const bool leader = rank == 0;
    const int unit = kPair ? c >> 1 : c;
    int *const tile_ctr = p.counters;

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
        for (int q = 0; q < kTileQ; ++q) {
            mbar_init(&tq_full[q], 1);
            mbar_init(&tq_empty[q], kPair ? 2 : 1);  // a pair's epilogues release the even CTA's entries
        }
        abort_flag = 0;
        s_gend[0] = s_gend[1] = s_peer_gend[0] = s_peer_gend[1] = 0;
        fence_mbar_init();
        prefetch_tmap(&p.tmap_w);
        prefetch_tmap(&p.tmap_h);
        // every unit starts on its own tile
        s_tile[0] = unit;
        mbar_arrive(&tq_full[0]);
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
            int s = mine;       // ring slot and phase parity of this thread's next k-block
            uint32_t ph = 0;
            long long g = 0;    // the current tile's first k-block in the CTA's sequence
            long long g_end = 0;
            bool ok = true;
            // tile scheduler (warp 0 of the even CTA): entry i + 1 of the queue is
            // published while tile i streams; its tile was fetched a tile earlier
            int pending = mine == 0 && leader ? atomicAdd(tile_ctr, 1) : -1;
            for (int i = 0; ok; ++i) {
                const int qe = i & (kTileQ - 1);  // tile-queue entry
                if (!lm_wait<kPair>(&tq_full[qe], (uint32_t)(i / kTileQ) & 1u, &abort_flag, p.status)) {
                    ok = false;
                    break;
                }
                const int tile = s_tile[qe];
                const bool sched = mine == 0 && leader && tile >= 0;
                bool published = false;
                auto publish = [&]() {
                    // entry i + 1: the tile fetched before, or -1 once the vocabulary is exhausted
                    const int nxt = pending >= 0 && pending + p.units < p.n_tiles ? pending + p.units : -1;
                    const int q1 = (i + 1) & (kTileQ - 1);
                    if (!mbar_wait_bounded(&tq_empty[q1], ((uint32_t)((i + 1) / kTileQ) & 1u) ^ 1u, &abort_flag,
                                           p.status))
                        return false;
                    s_tile[q1] = nxt;
                    if constexpr (kPair) {
                        st_cluster_s32(cluster_addr(&s_tile[q1], 1), nxt);
                        mbar_arrive_cluster(cluster_addr(&tq_full[q1], 1));
                    }
                    mbar_arrive(&tq_full[q1]);
                    pending = nxt >= 0 ? atomicAdd(tile_ctr, 1) : -1;
                    published = true;
                    return true;
                };
                if (tile < 0)
                    break;
                const int rot = lm_rot(p, tile);
                for (int j = (int)((g + mine) & 1); j < p.nk; j += 2) {
                    const int kb = j + rot >= p.nk ? j + rot - p.nk : j + rot;
                    if (!mbar_wait_bounded(&empty_bar[s], ph ^ 1u, &abort_flag, p.status)) {
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
                    g_end = g + j + 1;
                    s += 2;
                    if (s >= S) {
                        s -= S;
                        ph ^= 1u;
                    }
                    if (sched && !published && !publish()) {
                        ok = false;
                        break;
                    }
                }
                if (ok && sched && !published && !publish())
                    ok = false;
                g += p.nk;
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
            for (int i = 0; ok; ++i) {
                const int qe = i & (kTileQ - 1);  // tile-queue entry
                if (!mbar_wait_bounded(&tq_full[qe], (uint32_t)(i / kTileQ) & 1u, &abort_flag, p.status) ||
                    s_tile[qe] < 0)
                    break;
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
        for (int i = 0;; ++i) {
            const int b = i & 1;
            const int qe = i & (kTileQ - 1);  // tile-queue entry
            lm_wait<kPair>(&tq_full[qe], (uint32_t)(i / kTileQ) & 1u, &abort_flag, p.status);
            if (!agree())
                break;
            const int tile = s_tile[qe];
            epi_sync();  // every epilogue thread has read the entry
            if (e == 0) {
                if constexpr (kPair)
                    mbar_arrive_cluster(cluster_addr(&tq_empty[qe], 0));
                else
                    mbar_arrive(&tq_empty[qe]);
            }
            if (tile < 0)
                break;
            mbar_wait_bounded(p.expire_wait ? &never_bar : &acc_full[b], (uint32_t)(i >> 1) & 1u, &abort_flag,
                              p.status);
            if (!agree())
                break;
            tc_fence_after();
            // this CTA's 128 vocab entries (the odd CTA of a pair's last tile may have none)
            const int v0 = kPair ? tile * 256 + (int)rank * 128 : tile * 128, nvalid = min(128, p.V - v0);
            const int slot = kPair ? 2 * tile + (int)rank : tile;  // this CTA's partial of the tile
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
                if (sub == 0 && r < p.R) {
                    // the tile's statistics of row r, in the tile's own slot
                    p.part_tile[(size_t)slot * p.R_pad + r] = stat_pack(st);
                    if constexpr (kTyp)
                        p.part_tile_t[(size_t)slot * p.R_pad + r] = make_float2(st.sT, st.tT);
                }
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
}

// Final merge of the per-tile partials (K2 merge): one CTA per tree row.
// Thread k folds slots k, k + 256, ... in order -- the row's maximum and its
// lowest vocab index first, then the sums rescaled to that maximum -- and the
// 256 results combine in a fixed tree (warp butterflies, then the eight warps
// in order), so the outputs do not depend on which CTA of k2_lm_head took
// which tile.  Launched as a programmatic dependent of k2_lm_head: it waits for
// that grid (and what it waited for) to complete, then resets the tile counter
// for the next launch (every fetch has completed by then).  After a time-out
// recorded in the status word it writes nothing.
constexpr int kMergeThreads = 256;

template <bool kTyp>
__global__ void __launch_bounds__(kMergeThreads) k2_lm_merge(const __grid_constant__ LmParams p)
{
    pdl_trigger();  // the kernel that reads the outputs may be launched now
    pdl_wait();
    constexpr int kInFlight = 4;
    constexpr int kWarps = kMergeThreads / 32;
    __shared__ float s_m[kWarps], s_sum[kWarps][4];
    __shared__ int s_i[kWarps];
    const int r = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (r == 0 && tid == 0)
        p.counters[0] = 0;
    // a bounded wait of the LM head ran out: its partials are incomplete, the
    // outputs stay unwritten (the status word reports it)
    if (__ldcg(p.status) & kStatusTimeout)
        return;
    if (!in_bounds(r < p.R, p.status))
        return;
    // A thread's slots k = tid + 256 u.  Up to 256 x kInFlight slots (every
    // vocabulary up to 131072) its partials are loaded once and both passes
    // read registers; beyond that pass 2 reads them again.
    const bool held = p.n_slots <= kMergeThreads * kInFlight;
    float4 v[kInFlight];
    float2 w[kInFlight];
    // pass 1: maximum and its lowest vocab index (empty partials hold -inf, s = 0)
    float M = -INFINITY;
    int I = 0x7fffffff;
    for (int k0 = tid; k0 < p.n_slots; k0 += kMergeThreads * kInFlight) {
#pragma unroll
        for (int u = 0; u < kInFlight; ++u) {
            const int k = k0 + u * kMergeThreads;
            v[u] = k < p.n_slots ? __ldcg(p.part_tile + (size_t)k * p.R_pad + r)
                                 : make_float4(-INFINITY, __int_as_float(0x7fffffff), 0.f, 0.f);
            if constexpr (kTyp)
                w[u] = k < p.n_slots ? __ldcg(p.part_tile_t + (size_t)k * p.R_pad + r) : make_float2(0.f, 0.f);
        }
#pragma unroll
        for (int u = 0; u < kInFlight; ++u) {
            const int idx = __float_as_int(v[u].y);
            if (v[u].x > M || (v[u].x == M && idx < I)) {
                M = v[u].x;
                I = idx;
            }
        }
    }
    for (int m = 16; m >= 1; m >>= 1) {
        const float M2 = __shfl_xor_sync(0xffffffffu, M, m);
        const int I2 = __shfl_xor_sync(0xffffffffu, I, m);
        if (M2 > M || (M2 == M && I2 < I)) {
            M = M2;
            I = I2;
        }
    }
    if (lane == 0) {
        s_m[warp] = M;
        s_i[warp] = I;
    }
    __syncthreads();
    M = s_m[0];
    I = s_i[0];
    for (int wp = 1; wp < kWarps; ++wp)
        if (s_m[wp] > M || (s_m[wp] == M && s_i[wp] < I)) {
            M = s_m[wp];
            I = s_i[wp];
        }
    // pass 2: s, t (and the tempered sT, tT) relative to M
    float S = 0.f, T = 0.f, ST = 0.f, TT = 0.f;
    for (int k0 = tid; k0 < p.n_slots; k0 += kMergeThreads * kInFlight) {
        if (!held) {
#pragma unroll
            for (int u = 0; u < kInFlight; ++u) {
                const int k = k0 + u * kMergeThreads;
                v[u] = k < p.n_slots ? __ldcg(p.part_tile + (size_t)k * p.R_pad + r) : make_float4(0.f, 0.f, 0.f, 0.f);
                if constexpr (kTyp)
                    w[u] = k < p.n_slots ? __ldcg(p.part_tile_t + (size_t)k * p.R_pad + r) : make_float2(0.f, 0.f);
            }
        }
#pragma unroll
        for (int u = 0; u < kInFlight; ++u) {
            if (v[u].z > 0.f) {
                const float d = v[u].x - M;  // <= 0
                const float x = ex2_approx(d * kLog2e);
                S += v[u].z * x;
                T += (v[u].w + d * v[u].z) * x;
                if constexpr (kTyp) {
                    const float dT = d * p.inv_t;
                    const float xT = ex2_approx(dT * kLog2e);
                    ST += w[u].x * xT;
                    TT += (w[u].y + dT * w[u].x) * xT;
                }
            }
        }
    }
    for (int m = 16; m >= 1; m >>= 1) {
        S += __shfl_xor_sync(0xffffffffu, S, m);
        T += __shfl_xor_sync(0xffffffffu, T, m);
        if constexpr (kTyp) {
            ST += __shfl_xor_sync(0xffffffffu, ST, m);
            TT += __shfl_xor_sync(0xffffffffu, TT, m);
        }
    }
    if (lane == 0) {
        s_sum[warp][0] = S;
        s_sum[warp][1] = T;
        s_sum[warp][2] = ST;
        s_sum[warp][3] = TT;
    }
    __syncthreads();
    if (tid == 0) {
        S = T = ST = TT = 0.f;
        for (int wp = 0; wp < kWarps; ++wp) {
            S += s_sum[wp][0];
            T += s_sum[wp][1];
            ST += s_sum[wp][2];
            TT += s_sum[wp][3];
        }
        p.argmax[r] = I;
        p.top1[r] = 1.0f / S;
        p.entropy[r] = logf(S) - T / S;
        if constexpr (kTyp) {
            const float ls = logf(ST);
            p.logz_t[r] = M * p.inv_t + ls;
            p.ent_t[r] = ls - TT / ST;
        }
    }
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
    const size_t fixed = (size_t)kLmChunk * kChunkLd * 4;  // the epilogue's chunk buffer
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
    // per-tile partials: one per tile and CTA, merged by k2_lm_merge
    pl.n_slots = pl.pair ? 2 * pl.n_tiles : pl.n_tiles;
    pl.smem_bytes = (size_t)pl.stages * stage_bytes + fixed + 1024;
    // (max, argmax, s, t) and (sT, tT) partials.  The workspace also covers the
    // plan without pairs, which a launch takes when no cluster of two can be
    // resident.
    const int slots1 = ceil_div(V, 128);
    const int parts = pl.n_slots > slots1 ? pl.n_slots : slots1;
    pl.n_counters = 1;  // the tile counter
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

// k2_lm_head, then its merge as a programmatic dependent (launched while the
// LM head runs; it waits for it on the device).
template <bool kTyp>
static cudaError_t lm_launch_as(LmParams &p, const LmPlan &pl, cudaStream_t stream, bool pdl)
{
    cudaError_t e;
    if (pl.pair) {
        if ((e = allow_max_smem((const void *)k2_lm_head<kTyp, true>)) != cudaSuccess)
            return e;
        e = launch_kernel_cluster(k2_lm_head<kTyp, true>, dim3(pl.P), dim3(kLmThreads), pl.smem_bytes, stream, pdl,
                                  2, p);
    } else {
        if ((e = allow_max_smem((const void *)k2_lm_head<kTyp, false>)) != cudaSuccess)
            return e;
        e = launch_kernel(k2_lm_head<kTyp, false>, dim3(pl.P), dim3(kLmThreads), pl.smem_bytes, stream, pdl, p);
    }
    if (e != cudaSuccess)
        return e;
    return launch_kernel(k2_lm_merge<kTyp>, dim3(p.R), dim3(kMergeThreads), 0, stream, true, p);
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
    p.units = pl.units;
    p.n_slots = pl.n_slots;
    p.part_tile = static_cast<float4 *>(parts);
    p.part_tile_t = reinterpret_cast<float2 *>(p.part_tile + (size_t)pl.n_slots * pl.R_pad);
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
