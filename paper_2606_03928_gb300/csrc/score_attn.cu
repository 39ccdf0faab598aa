// Window attention score of VaSE-AttnV on tcgen05 tensor cores.
//
// For one unit (sequence s, KV head h) the score of cached slot i is
//     a_i = (1 / (G*W)) * sum_r softmax_i(q_r . k_i / sqrt(d))
// over the G*W cached window queries r of the unit's query heads, with the
// softmax taken over all N = K + B cached keys (Eq. (1) and Eq. (2), Sec. 2;
// non-causal cached queries per the footnote of Eq. (2)).  Pooling is done by
// the selection kernel.
//
// Decomposition: a cluster of C CTAs per unit, each owning a contiguous range
// of 128-token tiles.  A producer warp streams K tiles with TMA (128-byte
// swizzle) into a shared-memory ring and issues tcgen05.mma with the tile as
// A (M = 128 tokens) and the window queries as B (N = row block), so TMEM
// lane t holds token t's logits against every window row.  Four consumer
// warps make three passes over the logits:
//   pass 0: per-row maximum over tokens       (warp reduce-scatter, then cluster exchange)
//   pass 1: per-row sum of exp2(x - max)      (same)
//   pass 2: a_i = sum_r exp2(x_ri - max_r) / (sum_r * G*W), thread-local per token.
// Logits are recomputed per pass from K tiles re-read through L2.
#include <cfloat>

#include "kernels.cuh"
#include "ptx.cuh"

namespace vase {

namespace {

constexpr int kConsumerWarps = 4;
constexpr int kThreads = 32 * (kConsumerWarps + 1);
constexpr uint32_t kStageBytes = kTileTokens * kRowBytes;  // 32 KB: two 64-column panels of 128 rows
constexpr uint32_t kPanelBytes = kTileTokens * 128;        // 16 KB

struct ScoreSmem {
    uint32_t q_off, k_off, bar_off, slot_off, wst_off, xin_off, rowm_off, roww_off, total;
};

__host__ __device__ inline ScoreSmem score_layout(int GWp, int cluster, int stages) {
    ScoreSmem L;
    uint32_t o = 0;
    L.q_off = o;
    o += static_cast<uint32_t>(GWp) * kRowBytes;  // two panels of GWp rows x 128 B
    L.k_off = o;
    o += static_cast<uint32_t>(stages) * kStageBytes;
    L.bar_off = o;
    o += 8 * (1 + 2 * stages + 4);
    o = (o + 15u) & ~15u;
    L.slot_off = o;
    o += 16;
    L.wst_off = o;
    o += 4u * kConsumerWarps * GWp;
    L.xin_off = o;
    o += 4u * cluster * GWp;
    L.rowm_off = o;
    o += 4u * GWp;
    L.roww_off = o;
    o += 4u * GWp;
    L.total = o;
    return L;
}

struct OpMax {
    __device__ __forceinline__ float operator()(float a, float b) const { return fmaxf(a, b); }
};
struct OpSum {
    __device__ __forceinline__ float operator()(float a, float b) const { return a + b; }
};

// Reduce 32 values per lane across the warp so that lane l ends with the
// reduction of column l over all 32 lanes (31 shuffles instead of 160).
template <class Op>
__device__ __forceinline__ float warp_reduce_scatter(float (&v)[32], int lane, Op op) {
#pragma unroll
    for (int i = 0; i < 16; ++i) {
        const bool up = lane & 16;
        const float send = up ? v[i] : v[i + 16];
        const float keep = up ? v[i + 16] : v[i];
        v[i] = op(keep, __shfl_xor_sync(0xffffffffu, send, 16));
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const bool up = lane & 8;
        const float send = up ? v[i] : v[i + 8];
        const float keep = up ? v[i + 8] : v[i];
        v[i] = op(keep, __shfl_xor_sync(0xffffffffu, send, 8));
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const bool up = lane & 4;
        const float send = up ? v[i] : v[i + 4];
        const float keep = up ? v[i + 4] : v[i];
        v[i] = op(keep, __shfl_xor_sync(0xffffffffu, send, 4));
    }
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        const bool up = lane & 2;
        const float send = up ? v[i] : v[i + 2];
        const float keep = up ? v[i + 2] : v[i];
        v[i] = op(keep, __shfl_xor_sync(0xffffffffu, send, 2));
    }
    {
        const bool up = lane & 1;
        const float send = up ? v[0] : v[1];
        const float keep = up ? v[1] : v[0];
        v[0] = op(keep, __shfl_xor_sync(0xffffffffu, send, 1));
    }
    return v[0];
}

__global__ void __launch_bounds__(kThreads, 1)
    score_attn_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap qmap,
                      const ScoreAttnParams p) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const ScoreSmem L = score_layout(p.GWp, p.cluster, p.stages);

    uint8_t* q_s = smem + L.q_off;
    uint8_t* k_s = smem + L.k_off;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L.bar_off);
    uint64_t* q_full = bars;
    uint64_t* k_full = bars + 1;
    uint64_t* k_empty = bars + 1 + p.stages;
    uint64_t* t_full = bars + 1 + 2 * p.stages;
    uint64_t* t_empty = t_full + 2;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L.slot_off);
    float* wst = reinterpret_cast<float*>(smem + L.wst_off);    // [4][GWp] per-warp partials
    float* xin = reinterpret_cast<float*>(smem + L.xin_off);    // [C][GWp] cluster inbox
    float* rowm = reinterpret_cast<float*>(smem + L.rowm_off);  // [GWp] scaled row max
    float* roww = reinterpret_cast<float*>(smem + L.roww_off);  // [GWp] 1 / (row sum * G*W)

    const int tid = threadIdx.x;
    const int warp = tid >> 5;
    const int lane = tid & 31;
    const int unit = blockIdx.y;
    const int rank = blockIdx.x;
    const int C = p.cluster;
    const int GWp = p.GWp;
    const int NB = p.NB;
    const int n_rb = p.n_rb;
    const int t_begin = rank * p.tiles_per_cta;
    const int t_end = min(p.n_tiles, t_begin + p.tiles_per_cta);
    const int n_my = max(0, t_end - t_begin);
    const int64_t k_row = p.k_row0 + static_cast<int64_t>(unit) * p.N;
    const int seq = unit / p.Hkv;
    const int head = unit - seq * p.Hkv;
    const int64_t q_row = p.q_row0 + (static_cast<int64_t>(seq) * p.Hq + static_cast<int64_t>(head) * p.G) * p.W;

    if (tid == 0) {
        mbar_init(q_full, 1);
        for (int s = 0; s < p.stages; ++s) {
            mbar_init(&k_full[s], 1);
            mbar_init(&k_empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&t_full[b], 1);
            mbar_init(&t_empty[b], 32 * kConsumerWarps);
        }
        fence_mbar_init();
    }
    for (int i = tid; i < kConsumerWarps * GWp; i += kThreads) wst[i] = -INFINITY;
    if (warp == kConsumerWarps) {
        tmem_alloc(tmem_slot, static_cast<uint32_t>(p.tmem_cols));
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t taddr = *tmem_slot;
    if (C > 1) cluster_sync();  // every peer is running before any DSMEM store

    bool ok = true;
    const int total_items_per_pass = n_my * n_rb;
    (void)total_items_per_pass;

    if (warp == kConsumerWarps) {
        // ---------------------------------------------------------------- producer warp
        const uint32_t idesc = idesc_bf16_f32(128, static_cast<uint32_t>(NB));
        const uint32_t q_addr = smem_u32(q_s);
        const uint32_t k_addr = smem_u32(k_s);
        const int total_loads = 3 * n_my;
        int load_next = 0;
        if (lane == 0) {
            tma_prefetch_desc(&kmap);
            tma_prefetch_desc(&qmap);
            mbar_arrive_expect_tx(q_full, static_cast<uint32_t>(GWp) * kRowBytes);
            for (int panel = 0; panel < 2; ++panel) {
                for (int r0 = 0; r0 < GWp; r0 += 256) {
                    tma_load_2d(q_s + panel * GWp * 128 + r0 * 128, &qmap, panel * 64,
                                static_cast<int32_t>(q_row + r0), q_full);
                }
            }
        }
        for (int pass = 0; pass < 3; ++pass) {
            for (int j = 0; j < n_my; ++j) {
                const int Lidx = pass * n_my + j;
                const int s = Lidx % p.stages;
                if (lane == 0) {
                    while (load_next < total_loads && load_next < Lidx + p.stages) {
                        const int ls = load_next % p.stages;
                        const int ln = load_next / p.stages;
                        if (ln > 0 && ok) ok = mbar_wait(&k_empty[ls], (ln - 1) & 1, p.err, kErrScoreKEmpty);
                        const int tile = t_begin + (load_next % n_my);
                        const int32_t row = static_cast<int32_t>(k_row + static_cast<int64_t>(tile) * kTileTokens);
                        mbar_arrive_expect_tx(&k_full[ls], kStageBytes);
                        tma_load_2d(k_s + ls * kStageBytes, &kmap, 0, row, &k_full[ls]);
                        tma_load_2d(k_s + ls * kStageBytes + kPanelBytes, &kmap, 64, row, &k_full[ls]);
                        ++load_next;
                    }
                    if (ok) ok = mbar_wait(&k_full[s], (Lidx / p.stages) & 1, p.err, kErrScoreKFull);
                    if (Lidx == 0 && ok) ok = mbar_wait(q_full, 0, p.err, kErrScoreQ);
                }
                for (int rb = 0; rb < n_rb; ++rb) {
                    const int item = Lidx * n_rb + rb;
                    const int buf = item & 1;
                    const int use = item >> 1;
                    if (lane == 0) {
                        if (use > 0 && ok) ok = mbar_wait(&t_empty[buf], (use - 1) & 1, p.err, kErrScoreTEmpty);
                        tc_fence_after();
                        if (ok) {
                            const uint32_t a_base = k_addr + s * kStageBytes;
                            const uint32_t b_base = q_addr + rb * NB * 128;
#pragma unroll
                            for (int kk = 0; kk < 8; ++kk) {
                                const uint32_t koff = (kk >> 2) * kPanelBytes + (kk & 3) * 32;
                                const uint32_t qoff = (kk >> 2) * (GWp * 128) + (kk & 3) * 32;
                                tc_mma_bf16(taddr + buf * NB, sw128_kmajor_desc(a_base + koff),
                                            sw128_kmajor_desc(b_base + qoff), idesc, kk > 0 ? 1u : 0u);
                            }
                            tc_commit(&t_full[buf]);
                            if (rb == n_rb - 1) tc_commit(&k_empty[s]);
                        } else {
                            // keep the consumers' phases moving; their data is garbage and ignored
                            mbar_arrive(&t_full[buf]);
                            if (rb == n_rb - 1) mbar_arrive(&k_empty[s]);
                        }
                    }
                    __syncwarp();
                }
            }
            if (C > 1) {
                if (pass == 0) {
                    cluster_arrive();
                } else if (pass == 1) {
                    cluster_wait();
                    cluster_arrive();
                } else {
                    cluster_wait();
                }
            }
        }
        // Drain: every issued TMA load and MMA must land before the CTA leaves.
        if (lane == 0) {
            const int n_items = 3 * n_my * n_rb;
            for (int b = 0; b < 2; ++b) {
                const int uses = (n_items - b + 1) / 2;  // items with this buffer
                if (uses > 0) mbar_wait(&t_empty[b], (uses - 1) & 1, p.err, kErrScoreDrain);
            }
            for (int ls = 0; ls < p.stages && ls < total_loads; ++ls) {
                const int last = ((total_loads - 1 - ls) / p.stages) * p.stages + ls;  // last load using stage ls
                mbar_wait(&k_empty[ls], (last / p.stages) & 1, p.err, kErrScoreDrain);
            }
        }
        __syncwarp();
    } else {
        // ---------------------------------------------------------------- consumer warps
        const int ct = tid;  // 0..127
        const uint32_t lane_base = static_cast<uint32_t>(warp * 32) << 16;
        const float scale = p.scale_log2;
        for (int pass = 0; pass < 3; ++pass) {
            for (int j = 0; j < n_my; ++j) {
                const int Lidx = pass * n_my + j;
                const int tile = t_begin + j;
                const int token = tile * kTileTokens + warp * 32 + lane;
                const bool valid = token < p.N;
                float acc = 0.f;
                for (int rb = 0; rb < n_rb; ++rb) {
                    const int item = Lidx * n_rb + rb;
                    const int buf = item & 1;
                    const int use = item >> 1;
                    if (ok) ok = mbar_wait(&t_full[buf], use & 1, p.err, kErrScoreTFull);
                    tc_fence_after();
                    for (int c = 0; c < NB / 32; ++c) {
                        float v[32];
                        tmem_ld32(taddr + lane_base + static_cast<uint32_t>(buf * NB + c * 32), v);
                        const int row0 = rb * NB + c * 32;
                        if (pass == 0) {
#pragma unroll
                            for (int k = 0; k < 32; ++k) v[k] = valid ? v[k] : -INFINITY;
                            const float r = warp_reduce_scatter(v, lane, OpMax());
                            float* w = &wst[warp * GWp + row0 + lane];
                            *w = fmaxf(*w, r);
                        } else if (pass == 1) {
#pragma unroll
                            for (int k = 0; k < 32; ++k)
                                v[k] = valid ? exp2f(fmaf(v[k], scale, -rowm[row0 + k])) : 0.f;
                            const float r = warp_reduce_scatter(v, lane, OpSum());
                            wst[warp * GWp + row0 + lane] += r;
                        } else {
#pragma unroll
                            for (int k = 0; k < 32; ++k)
                                acc = fmaf(exp2f(fmaf(v[k], scale, -rowm[row0 + k])), roww[row0 + k], acc);
                        }
                    }
                    tc_fence_before();
                    mbar_arrive(&t_empty[buf]);
                }
                if (pass == 2 && valid) p.attn[static_cast<int64_t>(unit) * p.N + token] = acc;
            }
            if (pass < 2) {
                // combine the four warps, then the C CTAs of the cluster
                named_bar(1, 32 * kConsumerWarps);
                for (int row = ct; row < GWp; row += 32 * kConsumerWarps) {
                    float x = wst[row];
                    for (int w = 1; w < kConsumerWarps; ++w)
                        x = pass == 0 ? fmaxf(x, wst[w * GWp + row]) : x + wst[w * GWp + row];
                    for (int w = 0; w < kConsumerWarps; ++w) wst[w * GWp + row] = 0.f;
                    if (C > 1) {
                        for (int peer = 0; peer < C; ++peer)
                            st_cluster_f32(map_to_rank(&xin[rank * GWp + row], static_cast<uint32_t>(peer)), x);
                    } else {
                        xin[row] = x;
                    }
                }
                if (C > 1) {
                    cluster_arrive();
                    cluster_wait();
                } else {
                    named_bar(1, 32 * kConsumerWarps);
                }
                for (int row = ct; row < GWp; row += 32 * kConsumerWarps) {
                    float y = xin[row];
                    for (int c = 1; c < C; ++c) y = pass == 0 ? fmaxf(y, xin[c * GWp + row]) : y + xin[c * GWp + row];
                    if (pass == 0) {
                        rowm[row] = row < p.GW ? y * scale : INFINITY;
                    } else {
                        roww[row] = row < p.GW ? p.inv_gw / y : 0.f;
                    }
                }
                named_bar(1, 32 * kConsumerWarps);
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == kConsumerWarps) tmem_dealloc(taddr, static_cast<uint32_t>(p.tmem_cols));
}

}  // namespace

size_t score_attn_smem_bytes(int GWp, int cluster, int stages) {
    return score_layout(GWp, cluster, stages).total + 1024;  // + alignment slack
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
    cfg.gridDim = dim3(static_cast<unsigned>(p.cluster), static_cast<unsigned>(units), 1);
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
