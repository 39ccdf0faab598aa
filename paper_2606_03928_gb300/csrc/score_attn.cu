// Window attention score of VaSE-AttnV on tcgen05 tensor cores.
//
// For one unit (sequence s, KV head h) the score of cached slot i is
//     a_i = (1 / (G*W)) * sum_r softmax_i(q_r . k_i / sqrt(d))
// over the G*W cached window queries r of the unit's query heads, with the
// softmax over all N = K + B cached keys (Eq. (1) and Eq. (2), Sec. 2; the
// queries are cached and the scores non-causal, per the footnote of Eq. (2)).
// Pooling is left to the selection kernel.
//
// Decomposition: the work items (layer slot, unit) are dealt to CTA groups; a
// group is one CTA, or a cluster of C CTAs sharing one unit, each CTA owning a
// contiguous range of 128-token tiles that a TMA warp streams in (128-byte
// swizzle).  Two passes over the tiles, each on the tensor cores:
//   pass A  S^T = Q K_tile^T (M = 128 window rows, N = 128 tokens): TMEM lane =
//           window row, so every consumer thread keeps an online (max, sum of
//           exp2) of its own row with no cross-lane traffic.  The reference of the
//           sum is the maximum of the row's first chunk; it is raised only for a
//           chunk whose sum against it passes 2^64, so most chunks take no maximum.  Short windows
//           (G*W < 128) are replicated across the 128 lanes and each copy takes
//           a slice of the tile's tokens.  The per-row statistics are then
//           merged across copies, warps and (through distributed shared
//           memory) the CTAs of the cluster.
//   pass B  S = K_tile Q^T (M = 128 tokens, N = window rows): TMEM lane =
//           token, so each thread accumulates sum_r exp2(s_ri - m'_r) of its token
//           alone, m'_r = m_r + log2(l_r * G*W) folding the softmax denominator
//           and the 1/(G*W) mean into the exponent.
// Consumers: four warpgroups, each owning one 128-column TMEM accumulator, wherever the
// window fits 128 rows (each tile is one item per pass, dealt to the groups in turn) or
// has 512 rows (a tile's products then fill all 512 TMEM columns in either pass, and each
// group owns one 128-row block in both passes; pass B writes four partial scores that
// the selection adds).  A group's next product waits only for that group, and sixteen
// consumer warps cover the TMEM-load and exp2 latencies that eight left exposed.  In
// between (256 window rows) two groups share two 256-column accumulators.
// A single-CTA group that takes several items runs them as phases: phase k
// interleaves pass B of item k-1 (K re-read from L2, kept there by an
// evict-last hint on the pass-A read) with pass A of item k (K read from HBM),
// so the HBM stream never waits for a pass-B sweep.
#include <cfloat>

#include "kernels.cuh"
#include "ptx.cuh"

namespace vase {

namespace {

// Consumer warpgroups: kG = 2 (group g takes the items i with i % 2 == g, alternating over the accumulator
// buffers) or kG = 4 (one buffer each: at 512 window rows a tile's products are four 128 x 128 items in both
// passes, and group g always takes row block g).  Plus a TMA warp and two MMA-issue warps (even / odd items).
constexpr int kMaxGroups = 4;
constexpr int kMaxMma = 4;
// MMA-issue warps: warp x issues the items i with i % mma_warps == x, so each accumulator buffer (item i uses
// buffer i % nbuf) is only ever issued into by one warp.
__host__ __device__ constexpr int score_mma_warps(int) { return 2; }
__host__ __device__ constexpr int score_threads(int groups) { return 128 * groups + 32 + 32 * score_mma_warps(groups); }
constexpr int kMaxBufs = 4;
constexpr int kMaxStages = 8;
constexpr uint32_t kTileBytes = kTileTokens * kRowBytes;  // 32 KB: two 64-column panels of 128 rows
constexpr uint32_t kPanelBytes = kTileTokens * 128;       // 16 KB

struct ScoreSmem {
    uint32_t q_off, k_off, bar_off, slot_off, pm_off, pl_off, xm_off, xl_off, rowm_off, total;
};

__host__ __device__ inline ScoreSmem score_layout(int q_rows, int q_bufs, int n_rbA, int GWp, int cluster,
                                                   int stages, int stage_bytes, int groups) {
    ScoreSmem L;
    uint32_t o = 0;
    L.q_off = o;
    o += static_cast<uint32_t>(q_bufs) * q_rows * kRowBytes;
    L.k_off = o;
    o += static_cast<uint32_t>(stages) * stage_bytes;
    L.bar_off = o;
    o += 8 * (2 + 2 * kMaxGroups + (1 + kMaxMma) * stages + 2 * kMaxBufs);
    o = (o + 15u) & ~15u;
    L.slot_off = o;
    o += 16;
    L.pm_off = o;
    o += 4u * n_rbA * 128 * groups;  // [group][sub][128 lanes]
    L.pl_off = o;
    o += 4u * n_rbA * 128 * groups;
    L.xm_off = o;
    o += 4u * cluster * GWp;
    L.xl_off = o;
    o += 4u * cluster * GWp;
    L.rowm_off = o;
    o += 4u * GWp;
    L.total = o;
    return L;
}

// 2^x on the SFU (ex2.approx.ftz: relative error about 2^-22), no range fix-up.
__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// (m, l) <- merge of two online-softmax partials in the exp2 domain.
__device__ __forceinline__ void merge_ml(float& m, float& l, float m2, float l2) {
    const float mn = fmaxf(m, m2);
    if (mn == -INFINITY) return;
    l = l * exp2f(m - mn) + l2 * exp2f(m2 - mn);
    m = mn;
}

// One chunk of a row's online (max, sum of exp2) in pass A.  Once the row has a reference m (the maximum of
// its first chunk), a chunk is summed against it with no chunk maximum: (m, l) stays a valid pair as long as
// no exp2 overflows, and a sum above 2^64 (or inf) sends the chunk through the exact path, which raises m.
template <int CW, bool kPacked>
__device__ __forceinline__ void row_stats_chunk(const float (&v)[CW], float cs, float& m, float& l) {
    if (m != -INFINITY) {
        if constexpr (kPacked) {  // (the four-group consumers) packed pairs: fewer issued instructions
            const float2 cs2 = make_float2(cs, cs), nm2 = make_float2(-m, -m);
            float2 b0 = make_float2(0.f, 0.f), b1 = make_float2(0.f, 0.f);
#pragma unroll
            for (int q = 0; q < CW; q += 4) {
                const float2 x0 = __ffma2_rn(make_float2(v[q], v[q + 1]), cs2, nm2);
                const float2 x1 = __ffma2_rn(make_float2(v[q + 2], v[q + 3]), cs2, nm2);
                b0 = __fadd2_rn(b0, make_float2(ex2(x0.x), ex2(x0.y)));
                b1 = __fadd2_rn(b1, make_float2(ex2(x1.x), ex2(x1.y)));
            }
            const float sum = (b0.x + b0.y) + (b1.x + b1.y);
            if (sum <= 0x1p64f) {
                l += sum;
                return;
            }
        } else {
        float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
#pragma unroll
        for (int q = 0; q < CW; q += 4) {
            s0 += ex2(fmaf(v[q], cs, -m));
            s1 += ex2(fmaf(v[q + 1], cs, -m));
            s2 += ex2(fmaf(v[q + 2], cs, -m));
            s3 += ex2(fmaf(v[q + 3], cs, -m));
        }
        const float sum = (s0 + s1) + (s2 + s3);
        if (sum <= 0x1p64f) {
            l += sum;
            return;
        }
        }
    }
    float cm0 = v[0], cm1 = v[1], cm2 = v[2], cm3 = v[3];
#pragma unroll
    for (int q = 4; q < CW; q += 4) {
        cm0 = fmaxf(cm0, v[q]);
        cm1 = fmaxf(cm1, v[q + 1]);
        cm2 = fmaxf(cm2, v[q + 2]);
        cm3 = fmaxf(cm3, v[q + 3]);
    }
    const float mn = fmaxf(m, fmaxf(fmaxf(cm0, cm1), fmaxf(cm2, cm3)) * cs);
    if (mn != -INFINITY) {
        float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
#pragma unroll
        for (int q = 0; q < CW; q += 4) {
            s0 += ex2(fmaf(v[q], cs, -mn));
            s1 += ex2(fmaf(v[q + 1], cs, -mn));
            s2 += ex2(fmaf(v[q + 2], cs, -mn));
            s3 += ex2(fmaf(v[q + 3], cs, -mn));
        }
        l = l * ex2(m - mn) + ((s0 + s1) + (s2 + s3));
        m = mn;
    }
}

// Work item w of the launch: layer slot w / units, unit w % units.
struct ScoreItem {
    int slot, unit;
    int64_t k_row;  // first cache row of the unit
    int64_t q_row;  // first window-query row of the unit's query heads
};

__device__ __forceinline__ ScoreItem score_item(const ScoreAttnParams& p, int w) {
    ScoreItem it;
    it.slot = w / p.units;
    it.unit = w - it.slot * p.units;
    const int layer = p.batch.layer[it.slot];
    const int seq = it.unit / p.Hkv;
    const int head = it.unit - seq * p.Hkv;
    it.k_row = static_cast<int64_t>(layer) * p.layer_rows + static_cast<int64_t>(it.unit) * p.N;
    it.q_row = static_cast<int64_t>(layer) * p.q_layer_rows +
               (static_cast<int64_t>(seq) * p.Hq + static_cast<int64_t>(head) * p.G) * p.W;
    return it;
}

// Tile t of a phase with nA pass-A tiles and nB pass-B tiles (each 0 or n): the first `lead` pass-B
// tiles, then pairs of one pass-A and one pass-B tile in the orders A B, B A, A B, ... (so that the two
// consumer groups, which take alternate items, each get both kinds), then the last `lead` pass-A tiles.
// Returns true for a pass-A tile; j is the tile's index within its pass.
__device__ __forceinline__ bool phase_tile(int t, int nA, int nB, int lead, int& j) {
    if (nB == 0) {
        j = t;
        return true;
    }
    if (nA == 0 || t < lead) {
        j = t;
        return false;
    }
    const int u = t - lead;
    if (u < 2 * (nB - lead)) {
        const int pr = u >> 1;
        const bool isA = (u & 1) == (pr & 1);
        j = isA ? pr : lead + pr;
        return isA;
    }
    j = t - nB;
    return true;
}

// kHeadMax: GQA max-aggregation (per-head sums in pass B, the largest kept); a template argument so that the
// default mean keeps its pass-B loop free of the head bookkeeping.
// kEarly: with two accumulator buffers (one per group) the next MMA into a buffer waits for its consumer, so
// the buffer is released as soon as the item's last TMEM load has landed; with four, each group already has a
// second buffer in flight and the release follows the item's arithmetic (measured faster there).  A template
// argument so that each form compiles to its own loop.
template <bool kHeadMax, bool kEarly, int kG>
__global__ void __launch_bounds__(score_threads(kG), 1)
    score_attn_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap qmap,
                      const ScoreAttnParams p) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    constexpr int stage_bytes = kTileBytes;
    constexpr int kConsumers = 128 * kG;
    constexpr int kThreads = score_threads(kG);
    constexpr int kM = score_mma_warps(kG);
    const ScoreSmem Ly = score_layout(p.q_rows, p.q_bufs, p.n_rbA, p.GWp, p.cluster, p.stages, stage_bytes, kG);

    uint8_t* q_s = smem + Ly.q_off;
    uint8_t* st_s = smem + Ly.k_off;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + Ly.bar_off);
    uint64_t* q_full = bars;                      // [2]
    uint64_t* q_empty = bars + 2;                 // [2][kG]
    uint64_t* k_full = bars + 2 + 2 * kMaxGroups; // [stages]
    uint64_t* k_empty = k_full + p.stages;        // [stages][kM]
    uint64_t* t_full = k_empty + kM * p.stages;   // [nbuf]
    uint64_t* t_empty = t_full + kMaxBufs;        // [nbuf]
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + Ly.slot_off);
    float* pm = reinterpret_cast<float*>(smem + Ly.pm_off);      // [group][n_rbA][128] running max per lane
    float* pl = reinterpret_cast<float*>(smem + Ly.pl_off);      // [group][n_rbA][128] running sum per lane
    float* xm = reinterpret_cast<float*>(smem + Ly.xm_off);      // [C][GWp] cluster inbox
    float* xl = reinterpret_cast<float*>(smem + Ly.xl_off);
    float* rowm = reinterpret_cast<float*>(smem + Ly.rowm_off);  // [GWp] m'_r: row max + log2(row sum * G*W)

    const int tid = threadIdx.x;
    const int warp = tid >> 5;
    const int lane = tid & 31;
    const int C = p.cluster;
    const int rank = static_cast<int>(blockIdx.x) % C;
    const int group = static_cast<int>(blockIdx.x) / C;
    // items group, group + groups, ... (one item per group whenever C > 1)
    const int n_w = group < p.work ? (p.work - group + p.groups - 1) / p.groups : 0;
    const int GWp = p.GWp;
    const int NB = p.NB;
    const int head_rows = p.head_rows;  // W when kHeadMax: rows per query head
    const int n_rb = p.n_rb;
    const int n_rbA = p.n_rbA;
    const int R = p.rep;                 // copies of the window rows across the 128 pass-A lanes
    const int bufcols = p.buf_cols;      // TMEM columns per accumulator buffer
    const int nbuf = p.nbuf;             // accumulator buffers (2 or 4): item i uses buffer i & bmask, use i >> bshift
    const int bmask = nbuf - 1;
    const int bshift = nbuf == 4 ? 2 : 1;
    const int t_begin = rank * p.tiles_per_cta;
    const int t_end = min(p.n_tiles, t_begin + p.tiles_per_cta);
    const int n_my = max(0, t_end - t_begin);
    const int lead = min(p.lead, n_my);
    const uint32_t q_bytes = static_cast<uint32_t>(p.q_rows) * kRowBytes;
    // With one accumulator per tile and no more stages than accumulators, a stage is free as soon as the MMA
    // of its tile has completed, which the TMA warp reads from the accumulator's full barrier (the buffer
    // cannot be reused before the stage is reloaded, so the parity is unambiguous).  Otherwise each MMA warp
    // commits a release of the stage after its last product of the tile: the stage is free when the products that
    // read it complete, whatever the consumers are doing (measured 2402 -> 2349 us per eight layers at G*W = 512,
    // where the stage was released when each consumer group began its last item of the tile).
    const bool mma_release = n_rbA == 1 && n_rb == 1 && p.stages <= nbuf;

    if (tid == 0) {
        // A consumer group waits for the accumulators of its own items, which come from one MMA warp whose
        // commits complete in issue order.  A K stage is released on one barrier per MMA warp (its commit after
        // its last product of the tile) and a window-row buffer on one per consumer group (once the group has
        // seen the last of its items that read it); the TMA warp waits for the owners of each.
        for (int b = 0; b < 2; ++b) {
            mbar_init(&q_full[b], 1);
            for (int g = 0; g < kG; ++g) mbar_init(&q_empty[kG * b + g], 128);
        }
        for (int s = 0; s < p.stages; ++s) {
            mbar_init(&k_full[s], 1);
            for (int x = 0; x < kM; ++x) mbar_init(&k_empty[kM * s + x], 1);  // MMA warp x's commit after its last product of the tile
        }
        for (int b = 0; b < nbuf; ++b) {
            mbar_init(&t_full[b], 1);     // the MMA warp's commit
            mbar_init(&t_empty[b], 128);  // the 128 threads of the group that owns the item
        }
        fence_mbar_init();
    }
    for (int i = tid; i < n_rbA * kConsumers; i += kThreads) {
        pm[i] = -INFINITY;
        pl[i] = 0.f;
    }
    const int tma_warp = kConsumers / 32;
    const int mma_warp = tma_warp + 1;  // .. mma_warp + kM - 1
    if (warp == tma_warp) {
        tmem_alloc(tmem_slot, static_cast<uint32_t>(p.tmem_cols));
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t taddr = *tmem_slot;
    if (C > 1) cluster_sync();  // every peer is running before any DSMEM store

    bool ok = true;

    if (warp == tma_warp) {
        // ---------------------------------------------------------------- TMA warp: window rows and K tiles
        if (C > 1) cluster_arrive();  // this warp takes no part in the statistics exchange
        if (lane == 0) {
            tma_prefetch_desc(&kmap);
            tma_prefetch_desc(&qmap);
            const uint64_t keep = l2_policy_evict_last();   // pass-A reads: read again by pass B
            const uint64_t drop = l2_policy_evict_first();  // pass-B reads: last use
            // Owners of the tile in each stage (bit x = MMA warp x, two bits per stage) and of the pass-B items that
            // read each window-row buffer (bit g = consumer group g, kG bits per buffer), and the parity of the next
            // phase of every per-owner empty barrier.
            uint32_t slot_owners = 0, kpar = 0, q_owners = 0, qpar = 0;
            int ld = 0, g = 0, st_pos = 0;
            for (int k = 0; k <= n_w; ++k) {
                const int nA = k < n_w ? n_my : 0;
                const int nB = k > 0 ? n_my : 0;
                const ScoreItem itA = score_item(p, group + min(k, n_w - 1) * p.groups);
                const ScoreItem itB = score_item(p, group + max(k - 1, 0) * p.groups);
                uint32_t b_owners = 0;
                for (int t = 0; t < nA + nB; ++t) {
                    int j;
                    const bool isA = phase_tile(t, nA, nB, lead, j);
                    const int n_sub = isA ? n_rbA : n_rb;
                    uint32_t owners = 0;  // MMA warps with an item of the tile
                    for (int i = 0; i < n_sub; ++i) owners |= 1u << ((g + i) & (kM - 1));
                    if (!isA)
                        for (int i = 0; i < n_sub; ++i) b_owners |= 1u << ((g + i) & (kG - 1));
                    const int ls = st_pos;
                    if (ld >= p.stages && mma_release) {
                        const int i = ld - p.stages;  // one item per tile: the item of the stage's last load
                        if (ok) ok = mbar_wait(&t_full[i & bmask], (i >> bshift) & 1, p.err, kErrScoreKEmpty);
                    } else if (ld >= p.stages) {
                        const uint32_t prev = (slot_owners >> (kM * ls)) & ((1u << kM) - 1u);
                        for (int x = 0; x < kM; ++x) {
                            if (!((prev >> x) & 1u)) continue;
                            const int bit = kM * ls + x;
                            if (ok) ok = mbar_wait(&k_empty[bit], (kpar >> bit) & 1u, p.err, kErrScoreKEmpty);
                            kpar ^= 1u << bit;
                        }
                    }
                    slot_owners = (slot_owners & ~(((1u << kM) - 1u) << (kM * ls))) | (owners << (kM * ls));
                    if (isA && j == 0) {
                        // window rows of item k: R copies of the GWp rows (pass A lanes), or q_rows rows
                        const int qb = k & (p.q_bufs - 1);
                        if (k >= 2) {  // item k - 2 is done with the buffer
                            const uint32_t prev = (q_owners >> (kG * qb)) & ((1u << kG) - 1u);
                            for (int grp = 0; grp < kG; ++grp) {
                                if (!((prev >> grp) & 1u)) continue;
                                const int bit = kG * qb + grp;
                                if (ok) ok = mbar_wait(&q_empty[bit], (qpar >> bit) & 1u, p.err, kErrScoreQ);
                                qpar ^= 1u << bit;
                            }
                        }
                        uint8_t* qd = q_s + qb * q_bytes;
                        const int q_panel = p.q_rows * 128;
                        mbar_arrive_expect_tx(&q_full[qb], q_bytes);
                        for (int panel = 0; panel < 2; ++panel) {
                            if (R > 1) {
                                for (int c = 0; c < R; ++c)
                                    tma_load_2d(qd + panel * q_panel + c * GWp * 128, &qmap, panel * 64,
                                                static_cast<int32_t>(itA.q_row), &q_full[qb]);
                            } else {
                                for (int r0 = 0; r0 < p.q_rows; r0 += p.q_box)
                                    tma_load_2d(qd + panel * q_panel + r0 * 128, &qmap, panel * 64,
                                                static_cast<int32_t>(itA.q_row + r0), &q_full[qb]);
                            }
                        }
                    }
                    const int64_t base = isA ? itA.k_row : itB.k_row;
                    const int32_t row = static_cast<int32_t>(base + static_cast<int64_t>(t_begin + j) * kTileTokens);
                    uint8_t* st = st_s + ls * stage_bytes;
                    mbar_arrive_expect_tx(&k_full[ls], kTileBytes);
                    tma_load_2d_hint(st, &kmap, 0, row, &k_full[ls], isA ? keep : drop);
                    tma_load_2d_hint(st + kPanelBytes, &kmap, 64, row, &k_full[ls], isA ? keep : drop);
                    ++ld;
                    g += n_sub;
                    if (++st_pos == p.stages) st_pos = 0;
                }
                // the pass-B items of this phase read item k - 1's window rows; item k + 1 takes that buffer
                if (k >= 1 && k + 1 < n_w) {
                    const int qb = (k - 1) & (p.q_bufs - 1);
                    q_owners = (q_owners & ~(((1u << kG) - 1u) << (kG * qb))) | (b_owners << (kG * qb));
                }
            }
            // drain: every load has been consumed (and so has landed) before the CTA leaves
            for (int ls = 0; ls < p.stages && ls < ld; ++ls) {
                if (mma_release) {
                    const int i = ls + (ld - 1 - ls) / p.stages * p.stages;  // the stage's last load
                    mbar_wait(&t_full[i & bmask], (i >> bshift) & 1, p.err, kErrScoreDrain);
                    continue;
                }
                const uint32_t prev = (slot_owners >> (kM * ls)) & ((1u << kM) - 1u);
                for (int x = 0; x < kM; ++x) {
                    const int bit = kM * ls + x;
                    if ((prev >> x) & 1u) mbar_wait(&k_empty[bit], (kpar >> bit) & 1u, p.err, kErrScoreDrain);
                }
            }
        }
        __syncwarp();
        if (C > 1) cluster_wait();
    } else if (warp >= mma_warp && warp < mma_warp + kM) {
        // ---------------------------------------------------------------- MMA warps: one elected lane issues
        // Warp mma_warp + x issues the items i with i % 2 == x (the items of consumer group x).  Each issuing
        // thread runs a serial wait / issue / commit loop whose overhead exceeds the MMAs' own time on the tensor
        // pipe; two such loops overlap that overhead.  The whole warp runs the loop, so descriptors and ring
        // positions stay warp-uniform, and one lane chosen by elect.sync issues each tcgen05.mma / commit.
        if (C > 1) cluster_arrive();
        {
            const int mine = warp - mma_warp;
            const uint32_t idescA = idesc_bf16_f32(128, 128);
            const uint32_t idescB = idesc_bf16_f32(128, static_cast<uint32_t>(NB));
            const uint32_t q_panel = static_cast<uint32_t>(p.q_rows) * 128u;  // bytes per 64-column panel
            const uint64_t qdesc0 = sw128_kmajor_desc(smem_u32(q_s));
            const uint64_t kdesc = sw128_kmajor_desc(smem_u32(st_s));
            // start-address steps (16-byte units) of the eight K = 16 slices of d = 128
            uint32_t koff[8], qoff[8];
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {
                koff[kk] = ((kk >> 2) * kPanelBytes + (kk & 3) * 32) >> 4;
                qoff[kk] = ((kk >> 2) * q_panel + (kk & 3) * 32) >> 4;
            }
            int s = 0, s_phase = 0;        // K stage ring position
            int g = 0;                     // item counter
            const int n_items = n_w * n_my * (n_rbA + n_rb);
            for (int k = 0; k <= n_w; ++k) {
                const int nA = k < n_w ? n_my : 0;
                const int nB = k > 0 ? n_my : 0;
                for (int t = 0; t < nA + nB; ++t) {
                    int j;
                    const bool isA = phase_tile(t, nA, nB, lead, j);
                    const int n_sub = isA ? n_rbA : n_rb;
                    // Both warps wait for every phase of every full barrier, in order, owned tile or not: a parity
                    // wait cannot tell phase P from phase P + 2, so no phase may be skipped.
                    const int qb = (isA ? k : k - 1) & (p.q_bufs - 1);
                    if (isA && j == 0 && ok) ok = mbar_wait(&q_full[qb], (k >> 1) & 1, p.err, kErrScoreQ);
                    if (ok) ok = mbar_wait(&k_full[s], s_phase, p.err, kErrScoreKFull);
                    bool owns = false;
                    for (int i = 0; i < n_sub; ++i) owns |= ((g + i) & (kM - 1)) == mine;
                    if (owns) {  // this warp owns an item of the tile
                        const uint64_t qdesc = qdesc0 + ((static_cast<uint32_t>(qb) * q_bytes) >> 4);
                        const uint64_t kt = kdesc + ((static_cast<uint32_t>(s) * stage_bytes) >> 4);
                        for (int sub = 0; sub < n_sub; ++sub) {
                            const int gi = g + sub;
                            if ((gi & (kM - 1)) != mine) continue;
                            const int buf = gi & bmask;
                            const int use = gi >> bshift;
                            if (use > 0 && ok) ok = mbar_wait(&t_empty[buf], (use - 1) & 1, p.err, kErrScoreTEmpty);
                            ok = __all_sync(0xffffffffu, ok);
                            tc_fence_after();
                            const uint32_t d = taddr + static_cast<uint32_t>(buf * bufcols);
                            if (elect_one()) {
                                if (ok) {
                                    if (isA) {
                                        // A = window rows of row block `sub` (128 lanes), B = the tile's tokens
                                        const uint64_t qa = qdesc + ((static_cast<uint32_t>(sub) * 128u * 128u) >> 4);
#pragma unroll
                                        for (int kk = 0; kk < 8; ++kk)
                                            tc_mma_bf16(d, qa + qoff[kk], kt + koff[kk], idescA, kk > 0 ? 1u : 0u);
                                    } else {
                                        // A = the tile's tokens (128 lanes), B = window rows of row block `sub`
                                        const uint64_t qb_ = qdesc + ((static_cast<uint32_t>(sub) * NB * 128u) >> 4);
#pragma unroll
                                        for (int kk = 0; kk < 8; ++kk)
                                            tc_mma_bf16(d, kt + koff[kk], qb_ + qoff[kk], idescB, kk > 0 ? 1u : 0u);
                                    }
                                    tc_commit(&t_full[buf]);
                                } else {
                                    // keep every phase moving; the data is garbage and the error word is set
                                    mbar_arrive(&t_full[buf]);
                                }
                            }
                            __syncwarp();
                        }
                        if (!mma_release) {
                            // the stage is free once this warp's products of the tile have read it
                            if (elect_one()) {
                                if (ok) tc_commit(&k_empty[kM * s + mine]);
                                else mbar_arrive(&k_empty[kM * s + mine]);
                            }
                            __syncwarp();
                        }
                    }
                    g += n_sub;
                    if (++s == p.stages) {
                        s = 0;
                        s_phase ^= 1;
                    }
                }
            }
            // drain: the consumers have read every accumulator of this warp, so its MMAs have completed
            for (int b = mine; b < nbuf; b += kM) {
                const int uses = (n_items - b + nbuf - 1) / nbuf;
                if (uses > 0) mbar_wait(&t_empty[b], (uses - 1) & 1, p.err, kErrScoreDrain);
            }
        }
        __syncwarp();
        if (C > 1) cluster_wait();
    } else {
        // ---------------------------------------------------------------- consumer warpgroups
        const int grp = tid >> 7;   // group g takes the items i with i % kG == g
        const int L = tid & 127;    // TMEM lane
        const uint32_t lane_base = static_cast<uint32_t>((warp & 3) * 32) << 16;
        const float cs = p.scale_log2;
        // pass-A lane mapping: row (L mod rows_per_copy) of row block `sub`, token columns [c0, c0 + cw)
        const int rows_per_copy = R > 1 ? GWp : 128;
        const int copy = L / rows_per_copy;
        const int cw = 128 / R;
        const int c0 = copy * cw;
        float* pmg = pm + grp * n_rbA * 128;
        float* plg = pl + grp * n_rbA * 128;
        constexpr bool early = kEarly;
        constexpr int kCW = kG == 4 ? 32 : 64;  // pass-A columns per TMEM load (registers are scarcer at kG = 4)
        const bool own_block = kG == 4 && n_rbA == kG;  // one row block per group in both passes (n_rb == n_rbA)

        int st_pos = 0;  // K stage ring position
        int item = 0;    // accumulator counter
        for (int k = 0; k <= n_w; ++k) {
            const int nA = k < n_w ? n_my : 0;
            const int nB = k > 0 ? n_my : 0;
            const ScoreItem itB = score_item(p, group + max(k - 1, 0) * p.groups);
            bool owned_b = false;  // this group owns a pass-B item of the phase
            float* const attn_out = p.attn + static_cast<int64_t>(itB.slot) * n_rb * p.units * p.N;
            for (int t = 0; t < nA + nB; ++t) {
                int j;
                const bool isA = phase_tile(t, nA, nB, lead, j);
                const int s = st_pos;
                const int tile = t_begin + j;
                if (isA) {
                    // ------------------------------------ pass A: row statistics
                    const int tok0 = tile * kTileTokens;
                    // (kG = 4 with four row blocks: a tile's four items are this group's row block and three others')
                    const int item0 = item;
                    item += n_rbA;
                    for (int sub = own_block ? grp : 0; sub < n_rbA; sub += own_block ? kG : 1) {
                        const int it = item0 + sub;
                        if (!own_block && (it & (kG - 1)) != grp) continue;
                        const int buf = it & bmask;
                        if (ok) ok = mbar_wait(&t_full[buf], (it >> bshift) & 1, p.err, kErrScoreTFull);
                        tc_fence_after();
                        float m = pmg[sub * 128 + L];
                        float l = plg[sub * 128 + L];
                        // online (max, sum of exp2) over this lane's token columns, kCW (or 32) at a time
                        for (int c = 0; c < cw; c += kCW) {
                            float v[kCW];
                            const int width = cw - c >= kCW ? kCW : 32;
                            if constexpr (kCW == 64) {
                                if (width == 64) {
                                    tmem_ld64(taddr + lane_base + static_cast<uint32_t>(buf * bufcols + c0 + c), v);
                                } else {
                                    float h[32];
                                    tmem_ld32(taddr + lane_base + static_cast<uint32_t>(buf * bufcols + c0 + c), h);
#pragma unroll
                                    for (int q = 0; q < 32; ++q) {
                                        v[q] = h[q];
                                        v[q + 32] = -INFINITY;
                                    }
                                }
                            } else {
                                tmem_ld32(taddr + lane_base + static_cast<uint32_t>(buf * bufcols + c0 + c),
                                          *reinterpret_cast<float(*)[32]>(v));
                            }
                            if (early && c + kCW >= cw) {  // the item's last load has landed
                                tc_fence_before();
                                mbar_arrive(&t_empty[buf]);
                            }
                            const int nvalid = min(width, p.N - (tok0 + c0 + c));
                            if (nvalid < kCW) {
#pragma unroll
                                for (int q = 0; q < kCW; ++q)
                                    if (q >= nvalid) v[q] = -INFINITY;
                            }
                            row_stats_chunk<kCW, kG == 4>(v, cs, m, l);
                        }
                        pmg[sub * 128 + L] = m;
                        plg[sub * 128 + L] = l;
                        if (!early) {
                            tc_fence_before();
                            mbar_arrive(&t_empty[buf]);
                        }
                    }
                } else {
                    // ------------------------------------ pass B: per-token accumulation
                    // With two row blocks (G*W > 256) the two consecutive items of a tile belong to different
                    // groups; each group writes its own partial sum (attn part `grp`) and the selection kernel
                    // adds the parts.
                    const int token = tile * kTileTokens + L;
                    float acc = 0.f;
                    bool mine = false;
                    const int item0 = item;
                    item += n_rb;
                    for (int sub = own_block ? grp : 0; sub < n_rb; sub += own_block ? kG : 1) {
                        const int it = item0 + sub;
                        if (!own_block && (it & (kG - 1)) != grp) continue;
                        mine = true;
                        const int buf = it & bmask;
                        if (ok) ok = mbar_wait(&t_full[buf], (it >> bshift) & 1, p.err, kErrScoreTFull);
                        owned_b = true;
                        if (sub >= n_rb - kG) {
                            // item k - 1's last pass-B tile: this group is done with its window rows
                            if (j == nB - 1 && k + 1 < n_w) mbar_arrive(&q_empty[kG * ((k - 1) & (p.q_bufs - 1)) + grp]);
                        }
                        tc_fence_after();
                        if (!kHeadMax) {
                            // 32 columns at a time, two register sets: the load of the next set is in flight
                            // while this one is summed
                            const uint32_t col0 = taddr + lane_base + static_cast<uint32_t>(buf * bufcols);
                            const int nch = NB / 32;
                            uint32_t ra[32], rb[32];
                            auto sum32 = [&](const uint32_t (&r)[32], int c) {
                                const float4* m4 = reinterpret_cast<const float4*>(rowm + sub * NB + c);
                                if constexpr (kG == 4) {  // packed pairs (FFMA2, FADD2): fewer issued instructions
                                    const float2 cs2 = make_float2(cs, cs);
                                    float2 b0 = make_float2(0.f, 0.f), b1 = make_float2(0.f, 0.f);
#pragma unroll
                                    for (int q = 0; q < 8; ++q) {
                                        const float4 mm = m4[q];
                                        const float2 x0 = __ffma2_rn(make_float2(__uint_as_float(r[4 * q]), __uint_as_float(r[4 * q + 1])), cs2, make_float2(-mm.x, -mm.y));
                                        const float2 x1 = __ffma2_rn(make_float2(__uint_as_float(r[4 * q + 2]), __uint_as_float(r[4 * q + 3])), cs2, make_float2(-mm.z, -mm.w));
                                        b0 = __fadd2_rn(b0, make_float2(ex2(x0.x), ex2(x0.y)));
                                        b1 = __fadd2_rn(b1, make_float2(ex2(x1.x), ex2(x1.y)));
                                    }
                                    acc += (b0.x + b0.y) + (b1.x + b1.y);
                                    return;
                                }
                                float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
#pragma unroll
                                for (int q = 0; q < 8; ++q) {
                                    const float4 mm = m4[q];
                                    a0 += ex2(fmaf(__uint_as_float(r[4 * q]), cs, -mm.x));
                                    a1 += ex2(fmaf(__uint_as_float(r[4 * q + 1]), cs, -mm.y));
                                    a2 += ex2(fmaf(__uint_as_float(r[4 * q + 2]), cs, -mm.z));
                                    a3 += ex2(fmaf(__uint_as_float(r[4 * q + 3]), cs, -mm.w));
                                }
                                acc += (a0 + a1) + (a2 + a3);
                            };
                            // (early) the accumulator is released as soon as its last chunk is in registers
                            auto release = [&]() {
                                if (!early) return;
                                tc_fence_before();
                                mbar_arrive(&t_empty[buf]);
                            };
                            if constexpr (kG == 4) {
                                // one register set (the 608-thread block leaves 96 registers a thread); the other
                                // groups' warps cover the load latency
                                for (int ch = 0; ch < nch; ++ch) {
                                    tmem_ld32_issue(col0 + 32 * ch, ra);
                                    tmem_wait_ld32(ra);
                                    if (ch + 1 == nch) release();
                                    sum32(ra, 32 * ch);
                                }
                            } else {
                            tmem_ld32_issue(col0, ra);
                            tmem_wait_ld32(ra);
                            if (nch == 1) release();
                            for (int ch = 0; ch < nch; ch += 2) {
                                if (ch + 1 < nch) tmem_ld32_issue(col0 + 32 * (ch + 1), rb);
                                sum32(ra, 32 * ch);
                                if (ch + 1 < nch) {
                                    tmem_wait_ld32(rb);
                                    if (ch + 2 < nch) tmem_ld32_issue(col0 + 32 * (ch + 2), ra);
                                    else release();  // rb holds the last chunk
                                    sum32(rb, 32 * (ch + 1));
                                    if (ch + 2 < nch) {
                                        tmem_wait_ld32(ra);
                                        if (ch + 3 >= nch) release();  // ra holds the last chunk
                                    }
                                }
                            }
                            }
                        } else {
                        // GQA max-aggregation: the sum runs per query head (W consecutive window rows, whole
                        // heads per row block) and the token keeps the largest head sum
                        float head_sum = 0.f;
                        int head_end = kHeadMax ? sub * NB + head_rows : 0;
                        for (int c = 0; c < NB; c += kCW) {
                            float v[kCW];
                            const int width = NB - c >= kCW ? kCW : 32;
                            if constexpr (kCW == 64) {
                                if (width == 64) {
                                    tmem_ld64(taddr + lane_base + static_cast<uint32_t>(buf * bufcols + c), v);
                                } else {
                                    float h[32];
                                    tmem_ld32(taddr + lane_base + static_cast<uint32_t>(buf * bufcols + c), h);
#pragma unroll
                                    for (int q = 0; q < 32; ++q) v[q] = h[q];
                                }
                            } else {
                                tmem_ld32(taddr + lane_base + static_cast<uint32_t>(buf * bufcols + c),
                                          *reinterpret_cast<float(*)[32]>(v));
                            }
                            if (early && c + kCW >= NB) {  // the item's last load has landed
                                tc_fence_before();
                                mbar_arrive(&t_empty[buf]);
                            }
                            const float4* m4 = reinterpret_cast<const float4*>(rowm + sub * NB + c);
#pragma unroll
                            for (int q = 0; q < kCW / 4; ++q) {
                                if (q < width / 4) {
                                    if (sub * NB + c + 4 * q == head_end) {  // the same in every thread
                                        acc = fmaxf(acc, head_sum);
                                        head_sum = 0.f;
                                        head_end += head_rows;
                                    }
                                    const float4 mm = m4[q];
                                    head_sum += (ex2(fmaf(v[4 * q], cs, -mm.x)) + ex2(fmaf(v[4 * q + 1], cs, -mm.y))) +
                                                (ex2(fmaf(v[4 * q + 2], cs, -mm.z)) + ex2(fmaf(v[4 * q + 3], cs, -mm.w)));
                                }
                            }
                        }
                        acc = fmaxf(acc, head_sum);
                        }
                        if (!early) {
                            tc_fence_before();
                            mbar_arrive(&t_empty[buf]);
                        }
                    }
                    // no item in the last pass-B tile: the group's last one (if any) was waited for earlier
                    if (!mine && owned_b && j == nB - 1 && k + 1 < n_w)
                        mbar_arrive(&q_empty[kG * ((k - 1) & (p.q_bufs - 1)) + grp]);
                    if (mine && token < p.N) {
                        const int part = n_rb > 1 ? grp : 0;
                        attn_out[(static_cast<int64_t>(part) * p.units + itB.unit) * p.N + token] = acc;
                    }
                }
                if (++st_pos == p.stages) st_pos = 0;
            }
            if (k == n_w) break;
            // ------------------------------------ item k's row statistics: groups, copies, then the cluster
            // (every pass-B tile of item k - 1 is done, so rowm is free)
            named_bar(1, kConsumers);
            for (int r = tid; r < GWp; r += kConsumers) {
                float m = -INFINITY, l = 0.f;
                for (int g = 0; g < kG; ++g) {
                    const float* gm = pm + g * n_rbA * 128;
                    const float* gl = pl + g * n_rbA * 128;
                    if (R > 1) {
                        for (int c = 0; c < R; ++c) merge_ml(m, l, gm[c * GWp + r], gl[c * GWp + r]);
                    } else {
                        merge_ml(m, l, gm[(r >> 7) * 128 + (r & 127)], gl[(r >> 7) * 128 + (r & 127)]);
                    }
                }
                if (C > 1) {
                    for (int peer = 0; peer < C; ++peer) {
                        st_cluster_f32(map_to_rank(&xm[rank * GWp + r], static_cast<uint32_t>(peer)), m);
                        st_cluster_f32(map_to_rank(&xl[rank * GWp + r], static_cast<uint32_t>(peer)), l);
                    }
                } else {
                    const bool real = r < p.GW;
                    rowm[r] = real ? m + log2f(l * static_cast<float>(p.fold_rows)) : INFINITY;
                }
            }
            if (C > 1) {
                cluster_arrive();
                cluster_wait();
                for (int r = tid; r < GWp; r += kConsumers) {
                    float m = -INFINITY, l = 0.f;
                    for (int c = 0; c < C; ++c) merge_ml(m, l, xm[c * GWp + r], xl[c * GWp + r]);
                    const bool real = r < p.GW;
                    rowm[r] = real ? m + log2f(l * static_cast<float>(p.fold_rows)) : INFINITY;
                }
            }
            named_bar(1, kConsumers);
            // every read of the partial statistics is done: restart this thread's own entries for item k + 1
            for (int sub = 0; sub < n_rbA; ++sub) {
                pmg[sub * 128 + L] = -INFINITY;
                plg[sub * 128 + L] = 0.f;
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == tma_warp) tmem_dealloc(taddr, static_cast<uint32_t>(p.tmem_cols));
}

}  // namespace

size_t score_attn_smem_bytes(int q_rows, int q_bufs, int n_rbA, int GWp, int cluster, int stages, int groups) {
    return score_layout(q_rows, q_bufs, n_rbA, GWp, cluster, stages, kTileBytes, groups).total + 1024;
}

cudaError_t score_attn_set_attributes(size_t smem_bytes, int cluster) {
    for (auto fn : {score_attn_kernel<false, false, 2>, score_attn_kernel<true, false, 2>,
                    score_attn_kernel<false, true, 2>, score_attn_kernel<true, true, 2>,
                    score_attn_kernel<false, true, 4>, score_attn_kernel<true, true, 4>}) {
        cudaError_t e =
            cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem_bytes));
        if (e == cudaSuccess && cluster > 8) e = cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

cudaError_t launch_score_attn(const CUtensorMap& kmap, const CUtensorMap& qmap, const ScoreAttnParams& p,
                              size_t smem_bytes, cudaStream_t s) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(p.cluster) * static_cast<unsigned>(p.groups), 1, 1);
    cfg.blockDim = dim3(static_cast<unsigned>(score_threads(p.cgroups)), 1, 1);
    cfg.dynamicSmemBytes = smem_bytes;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = static_cast<unsigned>(p.cluster);
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    // four groups own one buffer each (their next product waits for them: early release); two groups with two
    // buffers each release after the arithmetic, with one buffer each as soon as the last load has landed
    if (p.cgroups == 4)
        return p.head_rows > 0 ? cudaLaunchKernelEx(&cfg, score_attn_kernel<true, true, 4>, kmap, qmap, p)
                               : cudaLaunchKernelEx(&cfg, score_attn_kernel<false, true, 4>, kmap, qmap, p);
    if (p.nbuf == 2)
        return p.head_rows > 0 ? cudaLaunchKernelEx(&cfg, score_attn_kernel<true, true, 2>, kmap, qmap, p)
                               : cudaLaunchKernelEx(&cfg, score_attn_kernel<false, true, 2>, kmap, qmap, p);
    return p.head_rows > 0 ? cudaLaunchKernelEx(&cfg, score_attn_kernel<true, false, 2>, kmap, qmap, p)
                           : cudaLaunchKernelEx(&cfg, score_attn_kernel<false, false, 2>, kmap, qmap, p);
}

}  // namespace vase
