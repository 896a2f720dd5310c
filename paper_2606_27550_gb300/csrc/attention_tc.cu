// attention_tc.cu -- tree-masked attention on the 5th-generation tensor cores
// (K1, head_dim 64 or 128: one kernel template, kD).
//
// Tree decoding (Sec. 3.2) with the ancestor-bitset mask (Sec. 2.3): the
// flattened (layer, kv head, row block) x key-tile space is split evenly over
// a persistent grid, with the contractions on tcgen05.  A CTA that covers a
// whole unit writes its output; a unit split
// between CTAs leaves one (O, m, l) partial per CTA, and a second small kernel
// (k1_merge_split, one warp per query row) combines them by log-sum-exp after
// the first one has finished (in a verification step, beside the acceptance
// kernel at the end of the step: nothing in the step reads the attention
// output):
//
//   S   = Q K^T   tcgen05.mma kind::f16, M = 128 query rows, N = 128 keys,
//                 K = kD = head_dim; Q (bf16) is the TMEM A operand, the K
//                 tile a 128-byte-swizzled K-major shared-memory operand; S
//                 accumulates in TMEM.
//   O  += P V     M = 128 rows, N = kD, K = 128 keys; P (bf16)
//                 is the TMEM A operand, the V tile an MN-major shared-memory
//                 operand; O accumulates in TMEM.
//
// One CTA per SM, 8 warps:
//   warps 0, 7   TMA producers: 128-key K tiles (warp 0) and V tiles (warp 7),
//                kD / 64 boxes of 64 x 128 each, through separate 3-stage rings:
//                QK^T releases a K slot, P V a V slot, so the next K tiles
//                never wait for a P V.
//   warp 1       TMEM allocation (512 columns) and the QK^T-issuing thread;
//                S is double-buffered, so the softmax of tile i overlaps
//                QK^T of tile i+1.
//   warp 6       the P V-issuing thread (O += P V of tile i as soon as P is
//                written; it releases the tile's stage).
//   warps 2-5    one thread per query row (TMEM lane): row max, exp2 with a
//                lazily rescaled reference maximum (O and l are rescaled only
//                when the maximum grows by more than 2^8), P written back to
//                TMEM, and the segment epilogue (normalise, or write a partial
//                for the merge).
// TMEM columns: S0 [0,128), S1 [128,256) with P0 / P1 aliased onto their first
// halves, O [256,256+kD), Q [384,384+kD/2).  Both QK^T and P V take their A operand
// from TMEM, so each MMA reads only the 128 x 16 B operand from shared memory.
// Query row r of a block sits in TMEM lane 32*(r%4) + r/4 so that the rows
// are spread over the four lane quadrants (all four SM sub-partitions share
// the softmax).
#include <string.h>

#include "kernels.cuh"

namespace tv {

namespace {

constexpr int kBN = 128;           // keys per tile
constexpr int kKStages = 3;        // K ring depth
constexpr int kVStages = 3;        // V ring depth
constexpr int kMaxStages = kKStages > kVStages ? kKStages : kVStages;
constexpr int kAtom = 128 * 128;   // one 64-column swizzle atom of a 128-row tile (16 KB)
constexpr int kTcThreads = 256;    // 8 warps: K loads, QK^T issuer, 4 softmax, P V issuer, V loads
// bytes of a K or V tile (128 keys x head_dim: kD / 64 atoms)
constexpr int tile_bytes(int d)
{
    return d / 64 * kAtom;
}
// floats per partial slot: O[128][kD], m[128], l[128]
constexpr int slot_floats(int d)
{
    return 128 * d + 256;
}
// TMEM columns.  P_b (bf16 pairs) overwrites the first half of S_b once the
// softmax has read S_b into registers; Q (bf16 pairs) is the A operand of QK^T.
constexpr uint32_t kColS0 = 0, kColS1 = 128, kColP0 = 0, kColP1 = 128, kColO = 256, kColQ = 384;
constexpr int kQPrefetchTiles = 3;  // tiles before a segment's end at which the next unit's q rows are prefetched
constexpr float kRescaleLog2 = 8.f;  // rescale O only when the row max grows by more than 2^8
constexpr int kWholeUnitMaxTiles = 6;  // see attn_tc_plan

// One sequence of a (possibly batched) launch: its own KV cache (tensor maps),
// prefix length, tree, queries and outputs.  Its tiles occupy
// [tile_base, tile_base + n_units * T) of the flattened tile space.
struct TcSeq {
    long long tile_base;
    const __nv_bfloat16 *q;  // [n_layers][nstride][Hq][head_dim]
    __nv_bfloat16 *out;      // same layout
    const TreeDesc *tree;
    int L, N, rows, row_blocks, T;
    int nstride;             // nodes per layer in q / out (N, or the largest tree of a scheduled loop)
};

struct TcParams {
    CUtensorMap tmap[2 * kMaxSeqPerLaunch];  // K, V of each sequence: (head_dim, L + N, Hkv, layers), box (64, 128, 1, 1)
    TcSeq seq[kMaxSeqPerLaunch];
    int n_seq, Hq, Hkv, group, layer_begin;
    long long total;
    int P;
    float scale_log2;
    float *part;
    int *status;
    // scheduled mode (sched != null): the tree and the prefix length come from
    // device memory (sched[0] = rung into rung_tree, sched[1] = L) and every
    // CTA derives the work split itself; seq[0] carries q, out and nstride
    const int32_t *sched;
    const TreeDesc *rung_tree[8];
    int n_rungs, n_layers, L_cap;
    int max_rows;  // query rows of the largest row block (the split merge's grid)
    int d;         // head_dim: the kernels' kD (host side: picks the instantiation)
    // rotary embedding (null: the queries are already rotated): per sequence a
    // table of (cos, sin) at position L + depth for every pair of head elements
    const float2 *rope_tab;
};

// Scheduled mode: the sequence of this step from the device state.  An
// out-of-range rung or a prefix that does not fit the cache gives no work
// (the acceptance kernel reports it).
__device__ void sched_plan(const TcParams &p, TcSeq *sq, long long *total)
{
    *sq = p.seq[0];
    sq->tile_base = 0;
    const int rung = p.sched[0], L = p.sched[1];
    const bool ok = rung >= 0 && rung < p.n_rungs && L >= 0;
    const TreeDesc *tr = p.rung_tree[ok ? rung : 0];
    const int N = tr->n;
    sq->tree = tr;
    sq->L = ok ? L : 0;
    sq->N = N;
    sq->rows = N * p.group;
    sq->row_blocks = (sq->rows + 127) / 128;
    sq->T = (sq->L + N + kBN - 1) / kBN;
    *total = (ok && L + N <= p.L_cap) ? (long long)p.n_layers * p.Hkv * sq->row_blocks * sq->T : 0;
}

// Sequence holding flattened tile t, searching forward from `b` (tiles are
// visited in increasing order by every role).  kBatched = false: sequence 0.
template <bool kBatched>
__device__ __forceinline__ int seq_at(const TcParams &p, long long t, int b)
{
    if constexpr (!kBatched) {
        return 0;
    } else {
        while (b + 1 < p.n_seq && t >= p.seq[b + 1].tile_base)
            ++b;
        return b;
    }
}

// CTAs the tile space is split over.  The host plans at most one CTA per
// tile; scheduled mode plans on the device with a grid of one CTA per SM, and
// a step with fewer tiles than that splits them over its first `total` CTAs
// only (the others get nothing), so that no CTA range inside the split is
// empty: the split merge combines the partials of consecutive CTAs.
__device__ __forceinline__ int tc_split_ctas(const TcParams &p, long long total)
{
    return (p.sched && total < p.P) ? (int)(total > 0 ? total : 1) : p.P;
}

// First flattened tile of CTA c's range (the ranges split the tile space
// evenly).  The quotients take 32-bit divisions whenever the operands fit.
__device__ __forceinline__ long long tc_seg_begin(long long total, int P, int c)
{
    const unsigned long long x = (unsigned long long)c * (unsigned long long)total;
    return x <= 0xffffffffull ? (long long)((uint32_t)x / (uint32_t)P) : (long long)(x / (unsigned long long)P);
}

// The CTA whose range holds tile t.
__device__ __forceinline__ int tc_cta_of(long long total, int P, long long t)
{
    if (total <= 0)
        return 0;
    const unsigned long long x = (unsigned long long)(t + 1) * (unsigned long long)P - 1ull;
    return x <= 0xffffffffull && (unsigned long long)total <= 0xffffffffull ? (int)((uint32_t)x / (uint32_t)total)
                                                                           : (int)(x / (unsigned long long)total);
}

// MN-major (N contiguous) 128-byte-swizzled operand: lbo = stride between
// 64-element column atoms, sbo = stride between groups of 8 K rows.
__device__ __forceinline__ uint64_t smem_desc_sw128_mn(uint32_t addr, uint32_t lbo, uint32_t sbo)
{
    return smem_desc_sw128(addr, lbo, sbo);
}

}  // namespace

// Allowed-key bits of 32 consecutive keys whose first has tree index tj0
// (key position minus the prefix length): bit c is set when key tj0 + c is a
// prefix key (tree index < 0) or an ancestor of the row's node (bit tj0 + c of
// its ancestor set anc, whose bits lie below the tree's node count).
__device__ __forceinline__ uint32_t tile_allow(int tj0, uint64_t anc)
{
    if (tj0 <= -32)
        return 0xffffffffu;
    if (tj0 >= 64)
        return 0u;
    if (tj0 >= 0)
        return (uint32_t)(anc >> tj0);
    const int pre = -tj0;  // 1 .. 31 prefix keys, then the tree from bit pre
    return ((1u << pre) - 1u) | (uint32_t)(anc << pre);
}

template <int kD, bool kBatched>
__global__ void __launch_bounds__(kTcThreads, 1) k1_tree_attention_tc(const __grid_constant__ TcParams p)
{
    static_assert(kD == 64 || kD == 128, "head_dim 64 or 128");
    constexpr int kTile = tile_bytes(kD);
    constexpr int kSlot = slot_floats(kD);
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t k_full[kMaxStages], k_empty[kMaxStages], v_full[kMaxStages], v_empty[kMaxStages];
    __shared__ __align__(8) uint64_t s_full[2], s_free[2], p_full[2], pv_done[2];
    __shared__ __align__(8) uint64_t q_full, o_free, drain_bar;
    __shared__ uint32_t tmem_slot;
    __shared__ int abort_flag;
    __shared__ TcSeq s_seq;
    __shared__ long long s_total;

    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sK = smem;                                // K ring: kKStages tiles
    uint8_t *sV = smem + (size_t)kKStages * kTile;     // V ring: kVStages tiles

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int c = blockIdx.x;
    // Launched as a programmatic dependent (a grid that leaves SMs free), the
    // kernel waits here for the stream's previous work (the previous step's
    // compaction writes the cache).  The step's LM head may then be launched:
    // it fills the SMs that attention CTAs leave free or release.
    pdl_wait();
    pdl_trigger();
    const TcSeq *seqs = p.seq;
    long long total = p.total;
    if (p.sched) {
        if (threadIdx.x == 0)
            sched_plan(p, &s_seq, &s_total);
        __syncthreads();
        seqs = &s_seq;
        total = s_total;
    }
    const int P = tc_split_ctas(p, total);
    const long long t0 = c < P ? tc_seg_begin(total, P, c) : total;
    const long long t1 = c < P ? tc_seg_begin(total, P, c + 1) : total;
    const long long n_tiles = t1 - t0;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kMaxStages; ++s) {
            mbar_init(&k_full[s], 1);
            mbar_init(&k_empty[s], 1);
            mbar_init(&v_full[s], 1);
            mbar_init(&v_empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&s_full[b], 1);
            mbar_init(&s_free[b], 4);
            mbar_init(&p_full[b], 4);
            mbar_init(&pv_done[b], 1);
        }
        mbar_init(&q_full, 4);
        mbar_init(&o_free, 4);
        mbar_init(&drain_bar, 2);  // one commit from each MMA issuer
        abort_flag = 0;
        fence_mbar_init();
        for (int b = 0; b < (kBatched ? p.n_seq : 1); ++b) {
            prefetch_tmap(&p.tmap[2 * b]);
            prefetch_tmap(&p.tmap[2 * b + 1]);
        }
    }
    if (warp == 1) {
        tmem_alloc(&tmem_slot, 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;

    if (warp == 0 || warp == 7) {
        // ------------------------------------------------------------ TMA producers
        // warp 0 streams the K tiles, warp 7 the V tiles, each through its own
        // half of the 3-stage ring: QK^T releases a K slot, P V a V slot.
        if (lane == 0) {
            const bool is_v = (warp == 7);
            uint64_t *full = is_v ? v_full : k_full;
            uint64_t *empty = is_v ? v_empty : k_empty;
            const int S = is_v ? kVStages : kKStages;
            uint8_t *ring = is_v ? sV : sK;
            long long issued = 0;
            int sb = 0;
            for (long long it = 0; it < n_tiles; ++it) {
                const int s = (int)(it % S);
                const uint32_t ph = (uint32_t)(it / S) & 1u;
                if (!mbar_wait_bounded(&empty[s], ph ^ 1u, &abort_flag, p.status))
                    break;
                const long long t = t0 + it;
                sb = seq_at<kBatched>(p, t, sb);
                const TcSeq &sq = seqs[sb];
                const long long tl = t - sq.tile_base;
                const int u = (int)(tl / sq.T);
                const int j = (int)(tl % sq.T);
                const int head = (u / sq.row_blocks) % p.Hkv;
                const int layer = p.layer_begin + u / (sq.row_blocks * p.Hkv);
                const CUtensorMap *m = &p.tmap[2 * sb + (is_v ? 1 : 0)];
                uint8_t *dst = ring + (size_t)s * kTile;
                mbar_arrive_expect_tx(&full[s], kTile);
#pragma unroll
                for (int a = 0; a < kD / 64; ++a)
                    tma_load_4d(dst + a * kAtom, m, &full[s], 64 * a, j * kBN, head, layer);
                issued = it + 1;
            }
            if (issued < n_tiles)
                for (long long it = (issued > S ? issued - S : 0); it < issued; ++it)
                    mbar_wait_drain(&full[it % S], (uint32_t)(it / S) & 1u);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ QK^T issuer
        if (lane == 0) {
            const uint32_t idesc_s = idesc_bf16_f32(128, kBN);
            int sg = -1, sb = 0;
            for (long long it = 0; it < n_tiles; ++it) {
                const long long t = t0 + it;
                sb = seq_at<kBatched>(p, t, sb);
                const bool first = (it == 0) || ((t - seqs[sb].tile_base) % seqs[sb].T == 0);
                if (first)
                    ++sg;
                const int s = (int)(it % kKStages);
                const int b = (int)(it & 1);
                // K landed; the softmax has read S_b (tile it - 2) and P V(it - 2) has read
                // the P that shares its columns; at a segment's first tile, its Q is staged
                if (!mbar_wait_bounded(&k_full[s], (uint32_t)(it / kKStages) & 1u, &abort_flag, p.status) ||
                    !mbar_wait_bounded(&s_free[b], ((uint32_t)(it >> 1) & 1u) ^ 1u, &abort_flag, p.status) ||
                    (it >= 2 &&
                     !mbar_wait_bounded(&pv_done[b], (uint32_t)((it - 2) >> 1) & 1u, &abort_flag, p.status)) ||
                    (first && !mbar_wait_bounded(&q_full, (uint32_t)sg & 1u, &abort_flag, p.status)))
                    break;
                tc_fence_after();
                const uint32_t k_base = smem_u32(sK + (size_t)s * kTile);
                const uint32_t s_col = b ? kColS1 : kColS0;
#pragma unroll
                for (int kk = 0; kk < kD / 16; ++kk) {
                    const uint32_t off = (uint32_t)(kk >> 2) * kAtom + (uint32_t)(kk & 3) * 32;
                    const uint64_t bdesc = smem_desc_sw128(k_base + off, 0, 1024);
                    tc_mma_f16_ts(tmem + s_col, tmem + kColQ + kk * 8, bdesc, idesc_s, kk > 0 ? 1u : 0u);
                }
                tc_commit(&s_full[b]);
                tc_commit(&k_empty[s]);
            }
            // arrives when every MMA issued above has retired (waited for before TMEM is released)
            tc_commit(&drain_bar);
        }
    } else if (warp == 6) {
        // ------------------------------------------------------------ P V issuer
        // A second issuing thread: each tcgen05.mma holds its issuer for about
        // 100 cycles at these shapes, so P V(i) issued here runs alongside
        // QK^T(i + 1) instead of queueing behind it, and the stage is released
        // that much sooner.
        if (lane == 0) {
            const uint32_t idesc_pv = idesc_bf16_f32(128, kD, false, true);
            int sg = -1, sb = 0;
            for (long long it = 0; it < n_tiles; ++it) {
                const long long t = t0 + it;
                sb = seq_at<kBatched>(p, t, sb);
                const bool first = (it == 0) || ((t - seqs[sb].tile_base) % seqs[sb].T == 0);
                if (first)
                    ++sg;
                const int b = (int)(it & 1);
                // P written; at a segment's first tile, the previous epilogue has read O
                if (!mbar_wait_bounded(&p_full[b], (uint32_t)(it >> 1) & 1u, &abort_flag, p.status) ||
                    (first && sg > 0 &&
                     !mbar_wait_bounded(&o_free, (uint32_t)(sg - 1) & 1u, &abort_flag, p.status)) ||
                    !mbar_wait_bounded(&v_full[it % kVStages], (uint32_t)(it / kVStages) & 1u, &abort_flag, p.status))
                    break;
                tc_fence_after();
                const uint32_t v_base = smem_u32(sV + (size_t)(it % kVStages) * kTile);
                const uint32_t p_col = b ? kColP1 : kColP0;
#pragma unroll
                for (int ks = 0; ks < kBN / 16; ++ks) {
                    const uint64_t bdesc = smem_desc_sw128_mn(v_base + ks * 2048, kAtom, 1024);
                    tc_mma_f16_ts(tmem + kColO, tmem + p_col + ks * 8, bdesc, idesc_pv, (first && ks == 0) ? 0u : 1u);
                }
                tc_commit(&v_empty[it % kVStages]);
                tc_commit(&pv_done[b]);
            }
            tc_commit(&drain_bar);
        }
    } else if (warp < 6) {
        // ------------------------------------------------------------ softmax / epilogue (warps 2-5)
        const int q4 = warp & 3;  // TMEM lane quadrant of this warp
        const uint32_t lane_addr = tmem + ((uint32_t)(32 * q4) << 16);
        const int rloc = 4 * lane + q4;  // query row of this thread within the block

        struct Seg {
            long long start, end, u_first, u_last;  // flattened tile indices
            int b, u, rb, head, layer_rel, rows_here, node, qh, L, N, ns, dep;
            bool valid;
            uint64_t anc;
            const __nv_bfloat16 *q;
            __nv_bfloat16 *out;
        };
        int sb = 0;
        auto describe = [&](long long t) {
            Seg g;
            sb = seq_at<kBatched>(p, t, sb);
            const TcSeq &sq = seqs[sb];
            g.b = sb;
            g.start = t;
            g.u = (int)((t - sq.tile_base) / sq.T);
            g.u_first = sq.tile_base + (long long)g.u * sq.T;
            g.u_last = g.u_first + sq.T;
            g.end = t1 < g.u_last ? t1 : g.u_last;
            g.rb = g.u % sq.row_blocks;
            g.head = (g.u / sq.row_blocks) % p.Hkv;
            g.layer_rel = g.u / (sq.row_blocks * p.Hkv);
            g.rows_here = min(128, sq.rows - g.rb * 128);
            g.valid = rloc < g.rows_here;
            const int grow = g.rb * 128 + rloc;
            g.node = g.valid ? grow / p.group : 0;
            g.qh = g.head * p.group + grow % p.group;
            // the row's query / output rows and tree entries
            if (g.valid)
                g.valid = in_bounds(g.layer_rel < p.n_layers && g.node < sq.N && g.node < sq.nstride &&
                                        g.node < kMaxNodes && g.qh < p.Hq,
                                    p.status);
            g.anc = g.valid ? sq.tree->anc[g.node] : 0ull;
            g.dep = g.valid ? sq.tree->depth[g.node] : 0;
            g.L = sq.L;
            g.N = sq.N;
            g.ns = sq.nstride;
            g.q = sq.q;
            g.out = sq.out;
            return g;
        };
        // Q row of this thread -> its TMEM lane as kD / 2 columns of bf16 pairs (the
        // A operand of QK^T); zeros for padding rows
        auto write_q = [&](const Seg &g) {
            const uint4 *src =
                reinterpret_cast<const uint4 *>(g.q + (((size_t)g.layer_rel * g.ns + g.node) * p.Hq + g.qh) * kD);
            if (!p.rope_tab) {
                // the whole row (2 kD bytes) in flight at once, then kD / 32 TMEM stores
                uint4 qv[kD / 8];
#pragma unroll
                for (int i = 0; i < kD / 8; ++i)
                    qv[i] = g.valid ? src[i] : make_uint4(0, 0, 0, 0);
#pragma unroll
                for (int qc = 0; qc < kD / 32; ++qc) {
                    uint32_t w[16];
#pragma unroll
                    for (int ch = 0; ch < 4; ++ch) {
                        const uint4 v = qv[qc * 4 + ch];
                        w[4 * ch] = v.x;
                        w[4 * ch + 1] = v.y;
                        w[4 * ch + 2] = v.z;
                        w[4 * ch + 3] = v.w;
                    }
                    tmem_st_32x32b_x16(lane_addr + kColQ + qc * 16, w);
                }
            } else {
                // pre-rotary query: element i pairs with i + kD / 2, rotated at position
                // L + depth(node) with the sequence's (cos, sin) table
                constexpr int kHalf = kD / 64;  // 32-element chunks per half row
                const float2 *tab = p.rope_tab + (size_t)g.b * kRopeTableEntries + (size_t)g.dep * kRopeMaxHalf;
#pragma unroll 1
                for (int qc = 0; qc < kHalf; ++qc) {
                    uint32_t wl[16], wh[16];
#pragma unroll
                    for (int ch = 0; ch < 4; ++ch) {
                        const uint4 lo = g.valid ? src[qc * 4 + ch] : make_uint4(0, 0, 0, 0);
                        const uint4 hi = g.valid ? src[(qc + kHalf) * 4 + ch] : make_uint4(0, 0, 0, 0);
                        const uint32_t lw[4] = {lo.x, lo.y, lo.z, lo.w}, hw[4] = {hi.x, hi.y, hi.z, hi.w};
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            const int i0 = 32 * qc + 8 * ch + 2 * e;
                            const float2 c0 = tab[i0], c1 = tab[i0 + 1];
                            const float a0 = __uint_as_float(lw[e] << 16), a1 = __uint_as_float(lw[e] & 0xffff0000u);
                            const float b0 = __uint_as_float(hw[e] << 16), b1 = __uint_as_float(hw[e] & 0xffff0000u);
                            wl[4 * ch + e] = pack_bf16x2(a0 * c0.x - b0 * c0.y, a1 * c1.x - b1 * c1.y);
                            wh[4 * ch + e] = pack_bf16x2(b0 * c0.x + a0 * c0.y, b1 * c1.x + a1 * c1.y);
                        }
                    }
                    tmem_st_32x32b_x16(lane_addr + kColQ + qc * 16, wl);
                    tmem_st_32x32b_x16(lane_addr + kColQ + (qc + kHalf) * 16, wh);
                }
            }
            tmem_st_wait();
            tc_fence_before();
            __syncwarp();
            if (lane == 0)
                mbar_arrive(&q_full);
        };
        long long it = 0;
        bool aborted = (n_tiles == 0);
        Seg g;
        if (!aborted) {
            g = describe(t0);
            write_q(g);
        }
        while (!aborted) {
            float m_ref = -INFINITY, l = 0.f;
            for (long long t = g.start; t < g.end; ++t, ++it) {
                const int b = (int)(it & 1);
                if (t + kQPrefetchTiles == g.end && g.end < t1) {
                    // the next unit's query rows are read from HBM when this segment ends
                    // (write_q below): ask for them in L2 a few tiles ahead
                    const Seg nx = describe(g.end);
                    if (nx.valid) {
                        const char *row = reinterpret_cast<const char *>(
                            nx.q + (((size_t)nx.layer_rel * nx.ns + nx.node) * p.Hq + nx.qh) * kD);
#pragma unroll
                        for (int off = 0; off < 2 * kD; off += 128)
                            asm volatile("prefetch.global.L2 [%0];" ::"l"(row + off));
                    }
                }
                if (!mbar_wait_bounded(&s_full[b], (uint32_t)(it >> 1) & 1u, &abort_flag, p.status)) {
                    aborted = true;
                    break;
                }
                tc_fence_after();
                const uint32_t sa = lane_addr + (b ? kColS1 : kColS0);
                const int key0 = (int)(t - g.u_first) * kBN;
                const bool masked = key0 + kBN > g.L;

                // pass 1: the whole S row (4 loads, one wait), masked row max
                float sc[kBN];
                {
                    uint32_t *r = reinterpret_cast<uint32_t *>(sc);
                    tmem_ld_32x32b_x32(sa, r);
                    tmem_ld_32x32b_x32(sa + 32, r + 32);
                    tmem_ld_32x32b_x32(sa + 64, r + 64);
                    tmem_ld_32x32b_x32(sa + 96, r + 96);
                    tmem_ld_wait();
                }
                float mx = -INFINITY;
                if (masked) {
                    // the row's allowed keys among the tile's 128 columns, 32 per word:
                    // prefix keys (tree index tj < 0) and the ancestors in the tree
                    uint32_t allow[kBN / 32];
#pragma unroll
                    for (int w = 0; w < kBN / 32; ++w)
                        allow[w] = tile_allow(key0 + 32 * w - g.L, g.anc);
#pragma unroll
                    for (int x = 0; x < kBN; ++x) {
                        sc[x] = ((allow[x >> 5] >> (x & 31)) & 1u) ? sc[x] : -INFINITY;
                        mx = fmaxf(mx, sc[x]);
                    }
                } else {
#pragma unroll
                    for (int x = 0; x < kBN; ++x)
                        mx = fmaxf(mx, sc[x]);
                }
                mx *= p.scale_log2;  // row max in log2 units (scale > 0)

                // lazily rescaled reference maximum
                float alpha = 1.f;
                bool rescale = false;
                if (t == g.start) {
                    m_ref = mx;
                } else if (mx > m_ref + kRescaleLog2) {
                    alpha = (m_ref == -INFINITY) ? 0.f : ex2_approx(m_ref - mx);
                    m_ref = mx;
                    rescale = true;
                }
                if (__any_sync(0xffffffffu, rescale)) {
                    // O holds the previous tiles' P V: wait for the last one, then scale in place
                    const long long jp = it - 1;
                    if (!mbar_wait_bounded(&pv_done[jp & 1], (uint32_t)(jp >> 1) & 1u, &abort_flag, p.status)) {
                        aborted = true;
                        break;
                    }
                    tc_fence_after();
                    l *= alpha;
#pragma unroll 1
                    for (int c0 = 0; c0 < kD; c0 += 32) {
                        uint32_t o[32];
                        tmem_ld_32x32b_x32(lane_addr + kColO + c0, o);
                        tmem_ld_wait();
#pragma unroll
                        for (int x = 0; x < 32; ++x)
                            o[x] = __float_as_uint(__uint_as_float(o[x]) * alpha);
                        tmem_st_32x32b_x32(lane_addr + kColO + c0, o);
                    }
                    tmem_st_wait();
                }
                // P buffer b was last read by O += P V of tile it - 2
                if (it >= 2 &&
                    !mbar_wait_bounded(&pv_done[b], (uint32_t)((it - 2) >> 1) & 1u, &abort_flag, p.status)) {
                    aborted = true;
                    break;
                }
                tc_fence_after();

                // pass 2: P = 2^(s * scale - m_ref) as bf16 pairs into TMEM (masked entries are
                // -inf and give 0), row sum into l
                const float mu = (m_ref == -INFINITY) ? 0.f : m_ref;
                const uint32_t pa = lane_addr + (b ? kColP1 : kColP0);
                float rs = 0.f;
#pragma unroll
                for (int c0 = 0; c0 < kBN; c0 += 32) {
                    uint32_t pk[16];
#pragma unroll
                    for (int x = 0; x < 16; ++x) {
                        const float p0 = ex2_approx(fmaf(sc[c0 + 2 * x], p.scale_log2, -mu));
                        const float p1 = ex2_approx(fmaf(sc[c0 + 2 * x + 1], p.scale_log2, -mu));
                        rs += p0 + p1;
                        pk[x] = pack_bf16x2(p0, p1);
                    }
                    tmem_st_32x32b_x16(pa + c0 / 2, pk);
                }
                l += rs;
                tmem_st_wait();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) {
                    mbar_arrive(&s_free[b]);
                    mbar_arrive(&p_full[b]);
                }
            }
            if (aborted)
                break;

            // Every QK^T of this segment has been consumed, so Q can take the next unit's rows
            // now, letting the next segment's first QK^T overlap this epilogue.
            const bool has_next = g.end < t1;
            Seg nx;
            if (has_next) {
                nx = describe(g.end);
                write_q(nx);
            }

            // ---------------------------------------------------- segment epilogue
            const long long jl = it - 1;
            if (!mbar_wait_bounded(&pv_done[jl & 1], (uint32_t)(jl >> 1) & 1u, &abort_flag, p.status))
                break;
            tc_fence_after();
            const bool whole = (g.start == g.u_first && g.end == g.u_last);
            float *slot = p.part + ((size_t)c * 2 + (g.start == t0 ? 0 : 1)) * kSlot;
            if (!whole && g.valid)
                g.valid = in_bounds(c < p.P && rloc < 128, p.status);
            {
                const float inv = 1.f / l;
                uint4 *dst =
                    reinterpret_cast<uint4 *>(g.out + (((size_t)g.layer_rel * g.ns + g.node) * p.Hq + g.qh) * kD);
                float4 *pdst = reinterpret_cast<float4 *>(slot + rloc * kD);
#pragma unroll 1
                for (int c0 = 0; c0 < kD; c0 += 32) {
                    uint32_t r[32];
                    tmem_ld_32x32b_x32(lane_addr + kColO + c0, r);
                    tmem_ld_wait();
                    if (!g.valid)
                        continue;
                    if (whole) {
#pragma unroll
                        for (int ch = 0; ch < 4; ++ch) {
                            uint4 v;
                            v.x = pack_bf16x2(__uint_as_float(r[8 * ch + 0]) * inv, __uint_as_float(r[8 * ch + 1]) * inv);
                            v.y = pack_bf16x2(__uint_as_float(r[8 * ch + 2]) * inv, __uint_as_float(r[8 * ch + 3]) * inv);
                            v.z = pack_bf16x2(__uint_as_float(r[8 * ch + 4]) * inv, __uint_as_float(r[8 * ch + 5]) * inv);
                            v.w = pack_bf16x2(__uint_as_float(r[8 * ch + 6]) * inv, __uint_as_float(r[8 * ch + 7]) * inv);
                            dst[c0 / 8 + ch] = v;
                        }
                    } else {
#pragma unroll
                        for (int x = 0; x < 8; ++x)
                            pdst[c0 / 4 + x] = make_float4(__uint_as_float(r[4 * x]), __uint_as_float(r[4 * x + 1]),
                                                           __uint_as_float(r[4 * x + 2]), __uint_as_float(r[4 * x + 3]));
                    }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0)
                mbar_arrive(&o_free);

            if (!whole && g.valid) {
                // partial (O in the slot already, m_ref, l); k1_merge_split finishes the unit
                slot[128 * kD + rloc] = m_ref;
                slot[128 * kD + 128 + rloc] = l;
            }
            if (!has_next)
                break;
            g = nx;
        }
    }

    // ---------------------------------------------------------------- teardown
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        if (lane == 0)
            mbar_wait_drain(&drain_bar, 0);
        __syncwarp();
        tmem_dealloc(tmem, 512);
    }
}

// Log-sum-exp merge of the partials of every unit split between CTAs.  A unit
// is split exactly when a CTA range starts inside it, so the grid runs over
// the CTA boundaries c = 1 .. P-1 (x) and groups of 8 query rows (y); the
// first boundary inside a unit handles it.  One warp per query row, each lane
// kD / 32 of the kD output columns, four slots' loads issued together; at most
// 64 registers per thread (four CTAs of 256 threads per SM).
//
// kAfterStep: launched as a programmatic dependent of a verification step's
// acceptance kernel.  The attention it merges has completed by then (the
// acceptance kernel proceeds only once the LM head has, and the LM head
// completes only after the attention), so it does not wait at entry and runs
// beside the acceptance kernel; at exit it waits for the acceptance kernel,
// so that the stream's next kernel also runs after the compaction.
// Otherwise it waits at entry for the stream's previous kernel.
struct PdlWaitOnExit {
    __device__ ~PdlWaitOnExit() { pdl_wait(); }
};

// kD / 32 consecutive floats of a partial row (one lane's columns)
template <int kCpl>
struct ColVec;
template <>
struct ColVec<4> {
    float v[4];
    __device__ __forceinline__ void load(const float *src)
    {
        const float4 x = __ldcg(reinterpret_cast<const float4 *>(src));
        v[0] = x.x, v[1] = x.y, v[2] = x.z, v[3] = x.w;
    }
};
template <>
struct ColVec<2> {
    float v[2];
    __device__ __forceinline__ void load(const float *src)
    {
        const float2 x = __ldcg(reinterpret_cast<const float2 *>(src));
        v[0] = x.x, v[1] = x.y;
    }
};

template <int kD, bool kBatched, bool kAfterStep>
__global__ void __launch_bounds__(256, 4) k1_merge_split(const __grid_constant__ TcParams p)
{
    constexpr int kSlot = slot_floats(kD);
    constexpr int kCpl = kD / 32;  // output columns per lane
    if constexpr (!kAfterStep)
        pdl_wait();
    pdl_trigger();
    PdlWaitOnExit pdl_exit;
    __shared__ TcSeq s_seq;
    __shared__ long long s_total;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const TcSeq *seqs = p.seq;
    long long total = p.total;
    if (p.sched) {
        if (threadIdx.x == 0)
            sched_plan(p, &s_seq, &s_total);
        __syncthreads();
        seqs = &s_seq;
        total = s_total;
    }
    const int P = tc_split_ctas(p, total);
    const int cb = blockIdx.x + 1;  // CTA range starting at tile t_c
    if (cb >= P)
        return;
    const long long tc = tc_seg_begin(total, P, cb);
    int b = 0;
    if constexpr (kBatched) {
        while (b + 1 < p.n_seq && tc >= seqs[b + 1].tile_base)
            ++b;
    }
    const TcSeq &sq = seqs[b];
    const int u = (int)((tc - sq.tile_base) / sq.T);
    const long long u_first = sq.tile_base + (long long)u * sq.T, u_last = u_first + sq.T;
    if (tc == u_first)
        return;  // the boundary is a unit boundary
    const int c_lo = tc_cta_of(total, P, u_first), c_hi = tc_cta_of(total, P, u_last - 1);
    if (cb != c_lo + 1)
        return;  // an earlier boundary inside this unit handles it
    const int nseg = c_hi - c_lo + 1;
    const int rb = u % sq.row_blocks;
    const int head = (u / sq.row_blocks) % p.Hkv;
    const int layer_rel = u / (sq.row_blocks * p.Hkv);
    const int rows_here = min(128, sq.rows - rb * 128);
    const int r = blockIdx.y * 8 + warp;
    if (r >= rows_here)
        return;
    {
        const int grow = rb * 128 + r;
        if (!in_bounds(c_lo >= 0 && c_hi < P && layer_rel < p.n_layers && grow / p.group < sq.nstride &&
                           head * p.group + grow % p.group < p.Hq,
                       p.status))
            return;
    }
    // lane j of each 32-slot block owns slot c_lo + j0 + j: its row pointer, max and weight
    float M = -INFINITY;
    for (int j0 = 0; j0 < nseg; j0 += 32) {
        const int cc = c_lo + j0 + lane;
        if (j0 + lane < nseg) {
            const float *sl = p.part + ((size_t)cc * 2 + (tc_seg_begin(total, P, cc) >= u_first ? 0 : 1)) * kSlot;
            M = fmaxf(M, __ldcg(sl + 128 * kD + r));
        }
    }
#pragma unroll
    for (int m = 16; m >= 1; m >>= 1)
        M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, m));
    float lsum = 0.f;
    float acc[kCpl] = {};
    for (int j0 = 0; j0 < nseg; j0 += 32) {
        const int cc = c_lo + j0 + lane;
        const float *sl = p.part;
        float w = 0.f;
        if (j0 + lane < nseg) {
            sl = p.part + ((size_t)cc * 2 + (tc_seg_begin(total, P, cc) >= u_first ? 0 : 1)) * kSlot;
            const float ms = __ldcg(sl + 128 * kD + r);
            w = (ms == -INFINITY) ? 0.f : ex2_approx(ms - M);
            lsum += w * __ldcg(sl + 128 * kD + 128 + r);
        }
        const unsigned long long row_ptr = reinterpret_cast<unsigned long long>(sl + r * kD);
        const int cnt = min(32, nseg - j0);
        for (int j1 = 0; j1 < cnt; j1 += 4) {
            ColVec<kCpl> v[4];
            float wk[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const int src = (j1 + k) & 31;
                // lane's column block of slot j0 + j1 + k
                const unsigned long long base = __shfl_sync(0xffffffffu, row_ptr, src) + 4ull * kCpl * lane;
                wk[k] = __shfl_sync(0xffffffffu, w, src);
                if (j1 + k < cnt)
                    v[k].load(reinterpret_cast<const float *>(base));
                else
#pragma unroll
                    for (int x = 0; x < kCpl; ++x)
                        v[k].v[x] = 0.f;
            }
#pragma unroll
            for (int k = 0; k < 4; ++k)
#pragma unroll
                for (int x = 0; x < kCpl; ++x)
                    acc[x] += wk[k] * v[k].v[x];
        }
    }
#pragma unroll
    for (int m = 16; m >= 1; m >>= 1)
        lsum += __shfl_xor_sync(0xffffffffu, lsum, m);
    const float inv = 1.f / lsum;
    const int grow = rb * 128 + r;
    const int node = grow / p.group;
    const int qh = head * p.group + grow % p.group;
    __nv_bfloat16 *orow = sq.out + (((size_t)layer_rel * sq.nstride + node) * p.Hq + qh) * kD;
    if constexpr (kCpl == 4)
        reinterpret_cast<uint2 *>(orow)[lane] =
            make_uint2(pack_bf16x2(acc[0] * inv, acc[1] * inv), pack_bf16x2(acc[2] * inv, acc[3] * inv));
    else
        reinterpret_cast<uint32_t *>(orow)[lane] = pack_bf16x2(acc[0] * inv, acc[1] * inv);
}

// ----------------------------------------------------------------------------
// host side

// The split-unit merge of an attention launch with parameters p, for head_dim
// kD.  after_step: see k1_merge_split.
template <int kD>
static cudaError_t merge_launch_d(const TcParams &p, bool batched, cudaStream_t stream, bool pdl, bool after_step)
{
    const dim3 grid(p.P - 1, (p.max_rows + 7) / 8);
    if (batched)
        return after_step ? launch_kernel(k1_merge_split<kD, true, true>, grid, dim3(256), 0, stream, pdl, p)
                          : launch_kernel(k1_merge_split<kD, true, false>, grid, dim3(256), 0, stream, pdl, p);
    return after_step ? launch_kernel(k1_merge_split<kD, false, true>, grid, dim3(256), 0, stream, pdl, p)
                      : launch_kernel(k1_merge_split<kD, false, false>, grid, dim3(256), 0, stream, pdl, p);
}

// Whether a CTA range of the launch starts inside a unit (the split merge then
// has work).  Scheduled mode plans on the device: assumed so.
static bool any_split(const TcParams &p)
{
    if (p.P <= 1)
        return false;
    if (p.sched)
        return true;
    int b = 0;
    for (int c = 1; c < p.P; ++c) {
        const long long t = (long long)((unsigned long long)c * (unsigned long long)p.total / (unsigned long long)p.P);
        while (b + 1 < p.n_seq && t >= p.seq[b + 1].tile_base)
            ++b;
        if ((t - p.seq[b].tile_base) % p.seq[b].T != 0)
            return true;
    }
    return false;
}

// The split-unit merge, when the launch split a unit (nothing to do otherwise).
static cudaError_t merge_launch(const TcParams &p, bool batched, cudaStream_t stream, bool pdl, bool after_step)
{
    if (!any_split(p))
        return cudaSuccess;
    return p.d == 64 ? merge_launch_d<64>(p, batched, stream, pdl, after_step)
                     : merge_launch_d<128>(p, batched, stream, pdl, after_step);
}

// The attention kernel for p.d, one CTA per SM (each holds 512 TMEM columns).
template <int kD, bool kBatched>
static cudaError_t attn_kernel_launch_d(const TcParams &p, cudaStream_t stream, bool pdl)
{
    cudaError_t e;
    if ((e = allow_max_smem((const void *)k1_tree_attention_tc<kD, kBatched>)) != cudaSuccess)
        return e;
    const size_t smem = (size_t)(kKStages + kVStages) * tile_bytes(kD) + 1024;
    return launch_kernel(k1_tree_attention_tc<kD, kBatched>, dim3(p.P), dim3(kTcThreads), smem, stream, pdl, p);
}

static cudaError_t attn_kernel_launch(const TcParams &p, bool batched, cudaStream_t stream, bool pdl)
{
    if (p.d == 64)
        return batched ? attn_kernel_launch_d<64, true>(p, stream, pdl) : attn_kernel_launch_d<64, false>(p, stream, pdl);
    return batched ? attn_kernel_launch_d<128, true>(p, stream, pdl) : attn_kernel_launch_d<128, false>(p, stream, pdl);
}

// The attention launch's parameters, kept for a split-unit merge enqueued later.
static void stash_merge(const TcParams &p, bool batched, AttnMerge *m)
{
    static_assert(sizeof(TcParams) <= sizeof(m->params), "AttnMerge holds the attention launch's parameters");
    memcpy(m->params, &p, sizeof p);
    m->batched = batched;
    m->pending = any_split(p);
}

bool attn_tc_supported(int d)
{
    return d == 64 || d == 128;
}

AttnPlan attn_tc_plan(int L, int N, int Hq, int Hkv, int n_layers, int n_sm)
{
    AttnPlan pl{};
    pl.group = Hq / Hkv;
    pl.rows = N * pl.group;
    pl.row_blocks = (pl.rows + 127) / 128;
    pl.T = (L + N + kBN - 1) / kBN;
    pl.n_units = n_layers * Hkv * pl.row_blocks;
    pl.total = (long long)pl.n_units * pl.T;
    long long P = n_sm;
    if (P > pl.total)
        P = pl.total;
    // A problem of one wave whose units are a few tiles long runs a whole unit
    // per CTA: a split would save those tiles' serial steps (about 1 us each on
    // one SM) but add the split merge's launch and round trips (measured on
    // GB300: whole units faster up to 5 tiles, even at 6-7).
    if (pl.total <= n_sm && pl.T <= kWholeUnitMaxTiles)
        P = pl.n_units;
    pl.P = (int)P;
    return pl;
}

size_t attn_tc_slot_floats(int d)
{
    return (size_t)slot_floats(d);
}

int attn_tc_units(const AttnSeq *seqs, int n_seq, int Hq, int Hkv, int n_layers)
{
    int units = 0;
    for (int b = 0; b < n_seq; ++b)
        units += attn_tc_plan(seqs[b].kv->L, seqs[b].N, Hq, Hkv, n_layers, 1).n_units;
    return units;
}

cudaError_t attn_tc_launch_batch(const AttnSeq *seqs, int n_seq, int layer_begin, int n_layers, int Hq, float *part,
                                 int *status, int n_sm, cudaStream_t stream, const char **err,
                                 const float2 *rope_tab, AttnMerge *merge_later)
{
    if (n_seq < 1 || n_seq > kMaxSeqPerLaunch) {
        *err = "too many sequences for one attention launch";
        return cudaErrorInvalidValue;
    }
    TcParams p{};
    long long tiles = 0;
    int max_rows = 0;
    const int Hkv = seqs[0].kv->n_kv_heads;
    const int d = seqs[0].kv->head_dim;
    if (!attn_tc_supported(d)) {
        *err = "head_dim 64 or 128";
        return cudaErrorInvalidValue;
    }
    for (int b = 0; b < n_seq; ++b) {
        const tb_kv *kv = seqs[b].kv;
        if (kv->head_dim != d || kv->n_kv_heads != Hkv) {
            *err = "the sequences of one attention launch share head_dim and kv heads";
            return cudaErrorInvalidValue;
        }
        const AttnPlan pl = attn_tc_plan(kv->L, seqs[b].N, Hq, Hkv, n_layers, n_sm);
        if (!make_tmap_kv(&p.tmap[2 * b], kv->k, d, kv->L + seqs[b].N, kv->n_kv_heads, kv->n_layers,
                          kv->head_stride, kv->layer_stride, kBN, err) ||
            !make_tmap_kv(&p.tmap[2 * b + 1], kv->v, d, kv->L + seqs[b].N, kv->n_kv_heads, kv->n_layers,
                          kv->head_stride, kv->layer_stride, kBN, err))
            return cudaErrorInvalidValue;
        TcSeq &sq = p.seq[b];
        sq.tile_base = tiles;
        sq.q = static_cast<const __nv_bfloat16 *>(seqs[b].q);
        sq.out = static_cast<__nv_bfloat16 *>(seqs[b].out);
        sq.tree = seqs[b].tree;
        sq.L = kv->L;
        sq.N = seqs[b].N;
        sq.rows = pl.rows;
        sq.row_blocks = pl.row_blocks;
        sq.T = pl.T;
        sq.nstride = seqs[b].N;
        tiles += pl.total;
        max_rows = pl.rows < 128 ? (pl.rows > max_rows ? pl.rows : max_rows) : 128;
    }
    p.n_seq = n_seq;
    p.Hq = Hq;
    p.Hkv = Hkv;
    p.group = Hq / Hkv;
    p.layer_begin = layer_begin;
    p.n_layers = n_layers;
    p.total = tiles;
    // one sequence: its plan (whole units for a short one-wave problem); a batch
    // splits its tiles evenly (units of different lengths)
    p.P = n_seq == 1 ? attn_tc_plan(seqs[0].kv->L, seqs[0].N, Hq, Hkv, n_layers, n_sm).P
                     : (int)(tiles < n_sm ? tiles : n_sm);
    p.d = d;
    p.scale_log2 = 1.4426950408889634f / sqrtf((float)d);
    p.part = part;
    p.status = status;
    p.rope_tab = rope_tab;
    p.max_rows = max_rows;
    const bool batched = n_seq > 1;
    cudaError_t e;
    // A grid that takes every SM starts when the stream's previous work is done,
    // so that all its CTAs start together (its work split is static); a grid
    // capped beside a longer LM head (merge_later->pdl_launch) is launched as a
    // programmatic dependent and its CTAs wait on SMs that are free already.
    const bool pdl = merge_later && merge_later->pdl_launch;
    if ((e = attn_kernel_launch(p, batched, stream, pdl)) != cudaSuccess)
        return e;
    if (merge_later) {
        stash_merge(p, batched, merge_later);
        return cudaSuccess;
    }
    // A plain dependent of the attention: launched as a programmatic one, its
    // CTAs would take the SMs that attention CTAs release and hold them until
    // the whole grid is done, away from an LM head beside it on another stream
    // (measured on GB300: the ragged batch's step 20 us longer).
    return merge_launch(p, batched, stream, false, false);
}

cudaError_t attn_tc_launch_sched(const AttnSched &sc, int Hq, float *part, int *status, int n_sm,
                                 cudaStream_t stream, const char **err, AttnMerge *merge_later)
{
    if (sc.n_rungs < 1 || sc.n_rungs > 8) {
        *err = "scheduled attention: 1..8 rungs";
        return cudaErrorInvalidValue;
    }
    const tb_kv *kv = sc.kv;
    const int d = kv->head_dim;
    if (!attn_tc_supported(d)) {
        *err = "head_dim 64 or 128";
        return cudaErrorInvalidValue;
    }
    TcParams p{};
    // the cache's whole capacity: keys past L + N are masked by the kernel
    if (!make_tmap_kv(&p.tmap[0], kv->k, d, kv->L_cap, kv->n_kv_heads, kv->n_layers, kv->head_stride,
                      kv->layer_stride, kBN, err) ||
        !make_tmap_kv(&p.tmap[1], kv->v, d, kv->L_cap, kv->n_kv_heads, kv->n_layers, kv->head_stride,
                      kv->layer_stride, kBN, err))
        return cudaErrorInvalidValue;
    TcSeq &sq = p.seq[0];
    sq.q = static_cast<const __nv_bfloat16 *>(sc.q);
    sq.out = static_cast<__nv_bfloat16 *>(sc.out);
    sq.tree = sc.rung_tree[0];
    sq.nstride = sc.N_max;
    sq.T = 1;
    sq.row_blocks = 1;
    p.n_seq = 1;
    p.Hq = Hq;
    p.Hkv = kv->n_kv_heads;
    p.group = Hq / kv->n_kv_heads;
    p.layer_begin = 0;
    p.n_layers = kv->n_layers;
    p.L_cap = kv->L_cap;
    p.P = n_sm;
    p.d = d;
    p.scale_log2 = 1.4426950408889634f / sqrtf((float)d);
    p.part = part;
    p.status = status;
    p.sched = sc.sched;
    p.rope_tab = sc.rope_tab;
    p.n_rungs = sc.n_rungs;
    for (int r = 0; r < sc.n_rungs; ++r)
        p.rung_tree[r] = sc.rung_tree[r];
    p.max_rows = sc.N_max * p.group < 128 ? sc.N_max * p.group : 128;
    cudaError_t e;
    if ((e = attn_kernel_launch(p, false, stream, false)) != cudaSuccess)
        return e;
    if (merge_later) {
        stash_merge(p, false, merge_later);
        return cudaSuccess;
    }
    return merge_launch(p, false, stream, false, false);
}

cudaError_t attn_tc_launch(const tb_kv *kv, const TreeDesc *d_tree, int N, int layer_begin, int n_layers,
                           const void *q, int Hq, void *out, float *part, int *status, int n_sm,
                           cudaStream_t stream, const char **err, const float2 *rope_tab, AttnMerge *merge_later)
{
    AttnSeq one{kv, d_tree, N, q, out};
    return attn_tc_launch_batch(&one, 1, layer_begin, n_layers, Hq, part, status, n_sm, stream, err, rope_tab,
                                merge_later);
}

cudaError_t attn_merge_launch(const AttnMerge &m, cudaStream_t stream, bool after_step)
{
    if (!m.pending)
        return cudaSuccess;
    TcParams p;
    memcpy(&p, m.params, sizeof p);
    return merge_launch(p, m.batched, stream, true, after_step);
}

TB_BOUNDS_COUNTER(bounds_violations_attention_tc)

}  // namespace tv
