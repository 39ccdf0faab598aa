// Window attention score of VaSE-AttnV on tcgen05 tensor cores.
//
// For one unit (sequence s, KV head h) the score of cached slot i is
//     a_i = (1 / (G*W)) * sum_r softmax_i(q_r . k_i / sqrt(d))
// over the G*W cached window queries r of the unit's query heads, with the
// softmax over all N = K + B cached keys (Eq. (1) and Eq. (2), Sec. 2; the
// queries are cached and the scores non-causal, per the footnote of Eq. (2)).
// Pooling is left to the selection kernel.
//
// Decomposition: a cluster of C CTAs per unit, each owning a contiguous range
// of 128-token tiles that a producer warp streams in with TMA (128-byte
// swizzle).  Two passes over the tiles, each on the tensor cores:
//   pass A  S^T = Q K_tile^T (M = 128 window rows, N = 128 tokens): TMEM lane =
//           window row, so every consumer thread keeps an online (max, sum of
//           exp2) of its own row with no cross-lane traffic.  Short windows
//           (G*W < 128) are replicated across the 128 lanes and each copy takes
//           a slice of the tile's tokens.  The per-row statistics are then
//           merged across copies, warps and (through distributed shared
//           memory) the CTAs of the cluster.
//   pass B  S = K_tile Q^T (M = 128 tokens, N = window rows): TMEM lane =
//           token, so each thread accumulates sum_r exp2(s_ri - m_r) / l_r of its
//           token alone.
// K tiles are re-read for pass B (from L2 for all but the largest units).
#include <cfloat>

#include "kernels.cuh"
#include "ptx.cuh"

namespace vase {

namespace {

constexpr int kGroups = 2;                      // consumer warpgroups; group g takes the items i with i % 2 == g
constexpr int kConsumers = 128 * kGroups;
constexpr int kThreads = kConsumers + 64;       // + a TMA warp and an MMA-issue warp
constexpr int kMaxBufs = 4;
constexpr uint32_t kTileBytes = kTileTokens * kRowBytes;  // 32 KB: two 64-column panels of 128 rows
constexpr uint32_t kPanelBytes = kTileTokens * 128;       // 16 KB

struct ScoreSmem {
    uint32_t q_off, k_off, bar_off, slot_off, pm_off, pl_off, xm_off, xl_off, rowm_off, roww_off, total;
};

__host__ __device__ inline ScoreSmem score_layout(int q_rows, int n_rbA, int GWp, int cluster, int stages,
                                                   int stage_bytes) {
    ScoreSmem L;
    uint32_t o = 0;
    L.q_off = o;
    o += static_cast<uint32_t>(q_rows) * kRowBytes;
    L.k_off = o;
    o += static_cast<uint32_t>(stages) * stage_bytes;
    L.bar_off = o;
    o += 8 * (1 + 2 * stages + 2 * kMaxBufs);
    o = (o + 15u) & ~15u;
    L.slot_off = o;
    o += 16;
    L.pm_off = o;
    o += 4u * n_rbA * kConsumers;  // [group][sub][128 lanes]
    L.pl_off = o;
    o += 4u * n_rbA * kConsumers;
    L.xm_off = o;
    o += 4u * cluster * GWp;
    L.xl_off = o;
    o += 4u * cluster * GWp;
    L.rowm_off = o;
    o += 4u * GWp;
    L.roww_off = o;
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

__global__ void __launch_bounds__(kThreads, 1)
    score_attn_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap qmap,
                      const ScoreAttnParams p) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    constexpr int stage_bytes = kTileBytes;
    const ScoreSmem Ly = score_layout(p.q_rows, p.n_rbA, p.GWp, p.cluster, p.stages, stage_bytes);

    uint8_t* q_s = smem + Ly.q_off;
    uint8_t* st_s = smem + Ly.k_off;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + Ly.bar_off);
    uint64_t* q_full = bars;
    uint64_t* k_full = bars + 1;
    uint64_t* k_empty = bars + 1 + p.stages;
    uint64_t* t_full = bars + 1 + 2 * p.stages;  // [nbuf]
    uint64_t* t_empty = t_full + kMaxBufs;        // [nbuf]
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + Ly.slot_off);
    float* pm = reinterpret_cast<float*>(smem + Ly.pm_off);      // [group][n_rbA][128] running max per lane
    float* pl = reinterpret_cast<float*>(smem + Ly.pl_off);      // [group][n_rbA][128] running sum per lane
    float* xm = reinterpret_cast<float*>(smem + Ly.xm_off);      // [C][GWp] cluster inbox
    float* xl = reinterpret_cast<float*>(smem + Ly.xl_off);
    float* rowm = reinterpret_cast<float*>(smem + Ly.rowm_off);  // [GWp] row max (scaled, exp2 domain)
    float* roww = reinterpret_cast<float*>(smem + Ly.roww_off);  // [GWp] 1 / (row sum * G*W)

    const int tid = threadIdx.x;
    const int warp = tid >> 5;
    const int lane = tid & 31;
    const int unit = blockIdx.y;
    const int rank = blockIdx.x;
    const int slot = blockIdx.z;  // layer slot of the batch
    const int layer = p.batch.layer[slot];
    float* const attn_out = p.attn + static_cast<int64_t>(slot) * p.n_rb * p.units * p.N;
    const int C = p.cluster;
    const int GWp = p.GWp;
    const int NB = p.NB;
    const int n_rb = p.n_rb;
    const int n_rbA = p.n_rbA;
    const int R = p.rep;                 // copies of the window rows across the 128 lanes in pass A
    const int bufcols = p.buf_cols;      // TMEM columns per accumulator buffer
    const int nbuf = p.nbuf;             // accumulator buffers (2 or 4)
    const int t_begin = rank * p.tiles_per_cta;
    const int t_end = min(p.n_tiles, t_begin + p.tiles_per_cta);
    const int n_my = max(0, t_end - t_begin);
    const int64_t k_row = static_cast<int64_t>(layer) * p.layer_rows + static_cast<int64_t>(unit) * p.N;
    const int seq = unit / p.Hkv;
    const int head = unit - seq * p.Hkv;
    const int64_t q_row = static_cast<int64_t>(layer) * p.q_layer_rows +
                          (static_cast<int64_t>(seq) * p.Hq + static_cast<int64_t>(head) * p.G) * p.W;
    const int itemsA = n_my * n_rbA;
    const int itemsB = n_my * n_rb;

    if (tid == 0) {
        mbar_init(q_full, 1);
        for (int s = 0; s < p.stages; ++s) {
            mbar_init(&k_full[s], 1);
            mbar_init(&k_empty[s], 1 + kConsumers);  // the last MMA commit + every consumer thread
        }
        for (int b = 0; b < nbuf; ++b) {
            mbar_init(&t_full[b], 1);
            mbar_init(&t_empty[b], 128);  // the 128 threads of the group that owns the item
        }
        fence_mbar_init();
    }
    for (int i = tid; i < n_rbA * kConsumers; i += kThreads) {
        pm[i] = -INFINITY;
        pl[i] = 0.f;
    }
    const int tma_warp = kConsumers / 32;
    const int mma_warp = tma_warp + 1;
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
    const int total_loads = 2 * n_my;

    if (warp == tma_warp) {
        // ---------------------------------------------------------------- TMA warp: window rows, then K tiles
        if (C > 1) cluster_arrive();  // this warp takes no part in the statistics exchange
        if (lane == 0) {
            tma_prefetch_desc(&kmap);
            tma_prefetch_desc(&qmap);
            // window rows: R copies of the GWp rows (pass A lanes), or q_rows rows when R == 1
            const int q_panel = p.q_rows * 128;
            mbar_arrive_expect_tx(q_full, static_cast<uint32_t>(p.q_rows) * kRowBytes);
            for (int panel = 0; panel < 2; ++panel) {
                if (R > 1) {
                    for (int c = 0; c < R; ++c)
                        tma_load_2d(q_s + panel * q_panel + c * GWp * 128, &qmap, panel * 64,
                                    static_cast<int32_t>(q_row), q_full);
                } else {
                    for (int r0 = 0; r0 < p.q_rows; r0 += p.q_box)
                        tma_load_2d(q_s + panel * q_panel + r0 * 128, &qmap, panel * 64,
                                    static_cast<int32_t>(q_row + r0), q_full);
                }
            }
            // K tiles of pass A, then again for pass B (second read served by L2)
            for (int ld = 0; ld < total_loads; ++ld) {
                const int ls = ld % p.stages;
                const int ln = ld / p.stages;
                if (ln > 0 && ok) ok = mbar_wait(&k_empty[ls], (ln - 1) & 1, p.err, kErrScoreKEmpty);
                const int tile = t_begin + (ld % n_my);
                const int32_t row = static_cast<int32_t>(k_row + static_cast<int64_t>(tile) * kTileTokens);
                uint8_t* st = st_s + ls * stage_bytes;
                mbar_arrive_expect_tx(&k_full[ls], kTileBytes);
                tma_load_2d(st, &kmap, 0, row, &k_full[ls]);
                tma_load_2d(st + kPanelBytes, &kmap, 64, row, &k_full[ls]);
            }
            // drain: every load has been consumed (and so has landed) before the CTA leaves
            for (int ls = 0; ls < p.stages && ls < total_loads; ++ls) {
                const int last = ((total_loads - 1 - ls) / p.stages) * p.stages + ls;
                mbar_wait(&k_empty[ls], (last / p.stages) & 1, p.err, kErrScoreDrain);
            }
        }
        __syncwarp();
        if (C > 1) cluster_wait();
    } else if (warp == mma_warp) {
        // ---------------------------------------------------------------- MMA warp: one thread issues tcgen05.mma
        // The issuing thread shares its SM sub-partition with consumer warps, so its instruction stream is kept
        // short: descriptors are built once and advanced by adding to the 14-bit start-address field.
        if (C > 1) cluster_arrive();
        if (lane == 0) {
            const uint32_t idescA = idesc_bf16_f32(128, 128);
            const uint32_t idescB = idesc_bf16_f32(128, static_cast<uint32_t>(NB));
            const uint32_t q_panel = static_cast<uint32_t>(p.q_rows) * 128u;  // bytes per 64-column panel
            const uint64_t qdesc = sw128_kmajor_desc(smem_u32(q_s));
            const uint64_t kdesc = sw128_kmajor_desc(smem_u32(st_s));
            // start-address steps (16-byte units) of the eight K = 16 slices of d = 128
            uint32_t koff[8], qoff[8];
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {
                koff[kk] = ((kk >> 2) * kPanelBytes + (kk & 3) * 32) >> 4;
                qoff[kk] = ((kk >> 2) * q_panel + (kk & 3) * 32) >> 4;
            }
            if (ok) ok = mbar_wait(q_full, 0, p.err, kErrScoreQ);
            int s = 0, s_phase = 0;        // K stage ring position
            int buf = 0, use = 0;          // accumulator ring position
            for (int pass = 0; pass < 2; ++pass) {
                const int n_sub = pass == 0 ? n_rbA : n_rb;
                for (int j = 0; j < n_my; ++j) {
                    if (ok) ok = mbar_wait(&k_full[s], s_phase, p.err, kErrScoreKFull);
                    const uint64_t kt = kdesc + ((static_cast<uint32_t>(s) * stage_bytes) >> 4);
                    for (int sub = 0; sub < n_sub; ++sub) {
                        if (use > 0 && ok) ok = mbar_wait(&t_empty[buf], (use - 1) & 1, p.err, kErrScoreTEmpty);
                        tc_fence_after();
                        const uint32_t d = taddr + static_cast<uint32_t>(buf * bufcols);
                        if (ok) {
                            if (pass == 0) {
                                // A = window rows of row block `sub` (128 lanes), B = the tile's tokens
                                const uint64_t qa = qdesc + ((static_cast<uint32_t>(sub) * 128u * 128u) >> 4);
#pragma unroll
                                for (int kk = 0; kk < 8; ++kk)
                                    tc_mma_bf16(d, qa + qoff[kk], kt + koff[kk], idescA, kk > 0 ? 1u : 0u);
                            } else {
                                // A = the tile's tokens (128 lanes), B = window rows of row block `sub`
                                const uint64_t qb = qdesc + ((static_cast<uint32_t>(sub) * NB * 128u) >> 4);
#pragma unroll
                                for (int kk = 0; kk < 8; ++kk)
                                    tc_mma_bf16(d, kt + koff[kk], qb + qoff[kk], idescB, kk > 0 ? 1u : 0u);
                            }
                            tc_commit(&t_full[buf]);
                            if (sub == n_sub - 1) tc_commit(&k_empty[s]);
                        } else {
                            // keep every phase moving; the data is garbage and the error word is set
                            mbar_arrive(&t_full[buf]);
                            if (sub == n_sub - 1) mbar_arrive(&k_empty[s]);
                        }
                        if (++buf == nbuf) {
                            buf = 0;
                            ++use;
                        }
                    }
                    if (++s == p.stages) {
                        s = 0;
                        s_phase ^= 1;
                    }
                }
            }
            // drain: the consumers have read every accumulator, so every MMA has completed
            const int n_items = itemsA + itemsB;
            for (int b = 0; b < nbuf; ++b) {
                const int uses = (n_items - b + nbuf - 1) / nbuf;
                if (uses > 0) mbar_wait(&t_empty[b], (uses - 1) & 1, p.err, kErrScoreDrain);
            }
        }
        __syncwarp();
        if (C > 1) cluster_wait();
    } else {
        // ---------------------------------------------------------------- consumer warpgroups
        const int grp = tid >> 7;   // 0 or 1
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
        // ------------------------------------ pass A: row statistics
        for (int j = 0; j < n_my; ++j) {
            const int tile = t_begin + j;
            const int s = j % p.stages;
            const int tok0 = tile * kTileTokens;
            for (int sub = 0; sub < n_rbA; ++sub) {
                const int item = j * n_rbA + sub;
                if ((item & 1) != grp) continue;
                const int buf = item % nbuf;
                const int use = item / nbuf;
                if (ok) ok = mbar_wait(&t_full[buf], use & 1, p.err, kErrScoreTFull);
                tc_fence_after();
                float m = pmg[sub * 128 + L];
                float l = plg[sub * 128 + L];
                // online (max, sum of exp2) over this lane's token columns, 64 (or 32) at a time
                for (int c = 0; c < cw; c += 64) {
                    float v[64];
                    const int width = cw - c >= 64 ? 64 : 32;
                    if (width == 64) {
                        tmem_ld64(taddr + lane_base + static_cast<uint32_t>(buf * bufcols + c0 + c), v);
                    } else {
                        float h[32];
                        tmem_ld32(taddr + lane_base + static_cast<uint32_t>(buf * bufcols + c0 + c), h);
#pragma unroll
                        for (int k = 0; k < 32; ++k) {
                            v[k] = h[k];
                            v[k + 32] = -INFINITY;
                        }
                    }
                    const int nvalid = min(width, p.N - (tok0 + c0 + c));
                    if (nvalid < 64) {
#pragma unroll
                        for (int k = 0; k < 64; ++k)
                            if (k >= nvalid) v[k] = -INFINITY;
                    }
                    float cm0 = v[0], cm1 = v[1], cm2 = v[2], cm3 = v[3];
#pragma unroll
                    for (int k = 4; k < 64; k += 4) {
                        cm0 = fmaxf(cm0, v[k]);
                        cm1 = fmaxf(cm1, v[k + 1]);
                        cm2 = fmaxf(cm2, v[k + 2]);
                        cm3 = fmaxf(cm3, v[k + 3]);
                    }
                    const float mn = fmaxf(m, fmaxf(fmaxf(cm0, cm1), fmaxf(cm2, cm3)) * cs);
                    if (mn != -INFINITY) {
                        float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
#pragma unroll
                        for (int k = 0; k < 64; k += 4) {
                            s0 += ex2(fmaf(v[k], cs, -mn));
                            s1 += ex2(fmaf(v[k + 1], cs, -mn));
                            s2 += ex2(fmaf(v[k + 2], cs, -mn));
                            s3 += ex2(fmaf(v[k + 3], cs, -mn));
                        }
                        l = l * ex2(m - mn) + ((s0 + s1) + (s2 + s3));
                        m = mn;
                    }
                }
                pmg[sub * 128 + L] = m;
                plg[sub * 128 + L] = l;
                tc_fence_before();
                mbar_arrive(&t_empty[buf]);
            }
            mbar_arrive(&k_empty[s]);
        }
        // ------------------------------------ merge the row statistics: groups, copies, then the cluster
        named_bar(1, kConsumers);
        for (int r = tid; r < GWp; r += kConsumers) {
            float m = -INFINITY, l = 0.f;
            for (int g = 0; g < kGroups; ++g) {
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
                xm[r] = m;
                xl[r] = l;
            }
        }
        if (C > 1) {
            cluster_arrive();
            cluster_wait();
        } else {
            named_bar(1, kConsumers);
        }
        for (int r = tid; r < GWp; r += kConsumers) {
            float m = -INFINITY, l = 0.f;
            for (int c = 0; c < C; ++c) merge_ml(m, l, xm[c * GWp + r], xl[c * GWp + r]);
            const bool real = r < p.GW;
            rowm[r] = real ? m : INFINITY;
            roww[r] = real ? p.inv_gw / l : 0.f;
        }
        named_bar(1, kConsumers);
        // ------------------------------------ pass B: per-token accumulation
        // With two row blocks (G*W > 256) each group owns one of them for every tile and writes its own
        // partial sum (attn part `grp`); the selection kernel adds the parts.
        for (int j = 0; j < n_my; ++j) {
            const int tile = t_begin + j;
            const int s = (n_my + j) % p.stages;
            const int token = tile * kTileTokens + L;
            float acc = 0.f;
            bool mine = false;
            for (int sub = 0; sub < n_rb; ++sub) {
                const int item = itemsA + j * n_rb + sub;
                if ((item & 1) != grp) continue;
                mine = true;
                const int buf = item % nbuf;
                const int use = item / nbuf;
                if (ok) ok = mbar_wait(&t_full[buf], use & 1, p.err, kErrScoreTFull);
                tc_fence_after();
                for (int c = 0; c < NB; c += 64) {
                    float v[64];
                    const int width = NB - c >= 64 ? 64 : 32;
                    if (width == 64) {
                        tmem_ld64(taddr + lane_base + static_cast<uint32_t>(buf * bufcols + c), v);
                    } else {
                        float h[32];
                        tmem_ld32(taddr + lane_base + static_cast<uint32_t>(buf * bufcols + c), h);
#pragma unroll
                        for (int k = 0; k < 32; ++k) v[k] = h[k];
                    }
                    const float4* m4 = reinterpret_cast<const float4*>(rowm + sub * NB + c);
                    const float4* w4 = reinterpret_cast<const float4*>(roww + sub * NB + c);
                    float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
#pragma unroll
                    for (int k = 0; k < 16; ++k) {
                        if (k < width / 4) {
                            const float4 mm = m4[k];
                            const float4 ww = w4[k];
                            a0 = fmaf(ex2(fmaf(v[4 * k], cs, -mm.x)), ww.x, a0);
                            a1 = fmaf(ex2(fmaf(v[4 * k + 1], cs, -mm.y)), ww.y, a1);
                            a2 = fmaf(ex2(fmaf(v[4 * k + 2], cs, -mm.z)), ww.z, a2);
                            a3 = fmaf(ex2(fmaf(v[4 * k + 3], cs, -mm.w)), ww.w, a3);
                        }
                    }
                    acc += (a0 + a1) + (a2 + a3);
                }
                tc_fence_before();
                mbar_arrive(&t_empty[buf]);
            }
            mbar_arrive(&k_empty[s]);
            if (mine && token < p.N) {
                const int part = n_rb > 1 ? grp : 0;
                attn_out[(static_cast<int64_t>(part) * p.units + unit) * p.N + token] = acc;
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == tma_warp) tmem_dealloc(taddr, static_cast<uint32_t>(p.tmem_cols));
}

}  // namespace

size_t score_attn_smem_bytes(int q_rows, int n_rbA, int GWp, int cluster, int stages) {
    return score_layout(q_rows, n_rbA, GWp, cluster, stages, kTileBytes).total + 1024;
}

cudaError_t score_attn_set_attributes(size_t smem_bytes, int cluster) {
    cudaError_t e = cudaFuncSetAttribute(score_attn_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem_bytes));
    if (e != cudaSuccess) return e;
    if (cluster > 8) e = cudaFuncSetAttribute(score_attn_kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    return e;
}

cudaError_t launch_score_attn(const CUtensorMap& kmap, const CUtensorMap& qmap, const ScoreAttnParams& p, int units,
                              size_t smem_bytes, cudaStream_t s) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(p.cluster), static_cast<unsigned>(units), static_cast<unsigned>(p.batch.n));
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = smem_bytes;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = static_cast<unsigned>(p.cluster);
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, score_attn_kernel, kmap, qmap, p);
}

}  // namespace vase
