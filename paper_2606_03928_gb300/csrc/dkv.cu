// VaSE-DKV leverage scores on tcgen05 tensor cores.
//
// For every candidate slot i < K of a unit:
//     s_i = ||G_t^T k_i||^2 * ||G_t^T v_i||^2                       (Eq. (4), Sec. 2)
// with G_t in R^{d x r}, entries i.i.d. N(0, 1/r), drawn afresh for every
// eviction round t (Sec. 3.2, VaSE-DKV), or once per stream for the CurDKV
// option.  G_t is generated on chip from Philox4x32-10 with Box-Muller and
// never stored in global memory.
//
// The projections K_tile (128 x d) * G_t (d x r) run as one bf16 MMA with
// fp32 accumulation: each entry of G_t is split exactly into three bf16
// terms g = g1 + g2 + g3 (|g - g1 - g2 - g3| <= 2^-24 |g|), which become
// three groups of 32 columns of the B operand (r <= 32, unused columns
// zero).  Keys and values are bf16 already, so every product is exact and
// the accumulation is plain fp32: the result matches an fp32 projection.
#include <cuda_bf16.h>

#include "kernels.cuh"
#include "ptx.cuh"

namespace vase {

namespace {

constexpr int kConsumerWarps = 4;
constexpr int kThreads = 32 * (kConsumerWarps + 1);
constexpr uint32_t kTileBytes = kTileTokens * kRowBytes;   // 32 KB per K or V tile
constexpr uint32_t kPanelBytes = kTileTokens * 128;        // 16 KB
constexpr uint32_t kStageBytes = 2 * kTileBytes;           // K tile + V tile
constexpr int kProjCols = 96;                              // 3 splits x 32 columns
constexpr uint32_t kGPanelBytes = kProjCols * 128;         // 12 KB per 64-element panel
constexpr uint32_t kTmemCols = 512;                        // 2 buffers x (96 K + 96 V) columns, rounded up

struct DkvSmem {
    uint32_t g_off, k_off, bar_off, slot_off, total;
};

__host__ __device__ inline DkvSmem dkv_layout(int stages) {
    DkvSmem L;
    uint32_t o = 0;
    L.g_off = o;
    o += 2 * kGPanelBytes;  // 24 KB, 1024-aligned panels
    L.k_off = o;
    o += static_cast<uint32_t>(stages) * kStageBytes;
    L.bar_off = o;
    o += 8 * (2 * stages + 4);
    o = (o + 15u) & ~15u;
    L.slot_off = o;
    o += 16;
    L.total = o;
    return L;
}

// Byte offset of bf16 element (row, col) of a K-major operand stored as two
// 64-column panels of `rows` 128-byte rows with the 128-byte swizzle.
__device__ __forceinline__ uint32_t sw128_offset(int row, int col, int rows) {
    const int panel = col >> 6;
    const int cb = (col & 63) * 2;      // byte within the 128-byte row
    const int chunk = (cb >> 4) ^ (row & 7);
    return static_cast<uint32_t>(panel * rows * 128 + row * 128 + chunk * 16 + (cb & 15));
}

__global__ void __launch_bounds__(kThreads, 1)
    dkv_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap,
               const DkvParams p) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const DkvSmem L = dkv_layout(p.stages);
    uint8_t* g_s = smem + L.g_off;
    uint8_t* kv_s = smem + L.k_off;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L.bar_off);
    uint64_t* k_full = bars;
    uint64_t* k_empty = bars + p.stages;
    uint64_t* t_full = bars + 2 * p.stages;
    uint64_t* t_empty = t_full + 2;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L.slot_off);

    const int tid = threadIdx.x;
    const int warp = tid >> 5;
    const int lane = tid & 31;
    const int unit = blockIdx.y;
    const int slot = blockIdx.z;
    const int layer = p.batch.layer[slot];
    const int rnd = p.fixed_g ? 0 : p.batch.rnd[slot];
    float* const out = p.out + static_cast<int64_t>(slot) * p.units * p.N;
    const int t_begin = blockIdx.x * p.tiles_per_cta;
    const int t_end = min(p.n_tiles_k, t_begin + p.tiles_per_cta);
    const int n_my = max(0, t_end - t_begin);
    const int64_t row_base = static_cast<int64_t>(layer) * p.layer_rows + static_cast<int64_t>(unit) * p.N;

    if (tid == 0) {
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
    if (warp == kConsumerWarps) {
        tmem_alloc(tmem_slot, kTmemCols);
        tmem_relinquish();
    }
    __syncthreads();
    // Start the first tile loads before generating G (they do not depend on it).

    if (warp == kConsumerWarps && lane == 0) {
        tma_prefetch_desc(&kmap);
        tma_prefetch_desc(&vmap);
        for (int ld = 0; ld < p.stages && ld < n_my; ++ld) {
            const int32_t row = static_cast<int32_t>(row_base + static_cast<int64_t>(t_begin + ld) * kTileTokens);
            uint8_t* st = kv_s + ld * kStageBytes;
            mbar_arrive_expect_tx(&k_full[ld], kStageBytes);
            tma_load_2d(st, &kmap, 0, row, &k_full[ld]);
            tma_load_2d(st + kPanelBytes, &kmap, 64, row, &k_full[ld]);
            tma_load_2d(st + kTileBytes, &vmap, 0, row, &k_full[ld]);
            tma_load_2d(st + kTileBytes + kPanelBytes, &vmap, 64, row, &k_full[ld]);
        }
    }

    // G (d x r) as three exact bf16 splits: B-operand row n = split * 32 + b, column a.
    {
        const int r = p.r;
        const float inv_sqrt_r = 1.0f / sqrtf(static_cast<float>(r));
        const uint32_t c1 = static_cast<uint32_t>(rnd);
        // shared G: one projection per round for every layer and unit (0 in the layer bits and the unit word)
        const uint32_t c2 = static_cast<uint32_t>(p.shared_g ? 0 : layer) | (kTagDkv << 24);
        const uint32_t c3 = static_cast<uint32_t>(p.shared_g ? 0 : unit);
        for (int idx = tid; idx < kHeadDim * 32; idx += kThreads) {
            const int a = idx >> 5;
            const int b = idx & 31;
            float g = 0.f;
            if (b < r) {
                const Philox4 w = philox4x32_10(Philox4{static_cast<uint32_t>(a * r + b), c1, c2, c3}, p.seed_lo,
                                                p.seed_hi);
                const float u1 = open_uniform(w.x);
                const float u2 = open_uniform(w.y);
                g = sqrtf(-2.0f * logf(u1)) * cospif(2.0f * u2) * inv_sqrt_r;
            }
            const __nv_bfloat16 g1 = __float2bfloat16_rn(g);
            const float rem1 = g - __bfloat162float(g1);
            const __nv_bfloat16 g2 = __float2bfloat16_rn(rem1);
            const float rem2 = rem1 - __bfloat162float(g2);
            const __nv_bfloat16 g3 = __float2bfloat16_rn(rem2);
            *reinterpret_cast<__nv_bfloat16*>(g_s + sw128_offset(b, a, kProjCols)) = g1;
            *reinterpret_cast<__nv_bfloat16*>(g_s + sw128_offset(32 + b, a, kProjCols)) = g2;
            *reinterpret_cast<__nv_bfloat16*>(g_s + sw128_offset(64 + b, a, kProjCols)) = g3;
        }
    }
    // generic-proxy writes of G must be visible to the tensor cores' async proxy
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t taddr = *tmem_slot;
    bool ok = true;

    if (warp == kConsumerWarps) {
        const uint32_t idesc = idesc_bf16_f32(128, kProjCols);
        const uint32_t g_addr = smem_u32(g_s);
        const uint32_t kv_addr = smem_u32(kv_s);
        for (int j = 0; j < n_my; ++j) {
            const int s = j % p.stages;
            const int buf = j & 1;
            const int use = j >> 1;
            if (lane == 0) {
                if (ok) ok = mbar_wait(&k_full[s], (j / p.stages) & 1, p.err, kErrDkvKFull);
                if (use > 0 && ok) ok = mbar_wait(&t_empty[buf], (use - 1) & 1, p.err, kErrDkvTEmpty);
                tc_fence_after();
                if (ok) {
                    const uint32_t kb = kv_addr + s * kStageBytes;
                    const uint32_t vb = kb + kTileBytes;
                    const uint32_t dk = taddr + buf * (2 * kProjCols);
                    const uint32_t dv = dk + kProjCols;
#pragma unroll
                    for (int kk = 0; kk < 8; ++kk) {
                        const uint32_t toff = (kk >> 2) * kPanelBytes + (kk & 3) * 32;
                        const uint32_t goff = (kk >> 2) * kGPanelBytes + (kk & 3) * 32;
                        const uint64_t gdesc = sw128_kmajor_desc(g_addr + goff);
                        tc_mma_bf16(dk, sw128_kmajor_desc(kb + toff), gdesc, idesc, kk > 0 ? 1u : 0u);
                        tc_mma_bf16(dv, sw128_kmajor_desc(vb + toff), gdesc, idesc, kk > 0 ? 1u : 0u);
                    }
                    tc_commit(&t_full[buf]);
                    tc_commit(&k_empty[s]);
                } else {
                    mbar_arrive(&t_full[buf]);
                    mbar_arrive(&k_empty[s]);
                }
                // refill this stage with the tile `stages` ahead once its MMAs are done
                const int nxt = j + p.stages;
                if (nxt < n_my) {
                    if (ok) ok = mbar_wait(&k_empty[s], (j / p.stages) & 1, p.err, kErrDkvKEmpty);
                    const int32_t row =
                        static_cast<int32_t>(row_base + static_cast<int64_t>(t_begin + nxt) * kTileTokens);
                    uint8_t* st = kv_s + s * kStageBytes;
                    mbar_arrive_expect_tx(&k_full[s], kStageBytes);
                    tma_load_2d(st, &kmap, 0, row, &k_full[s]);
                    tma_load_2d(st + kPanelBytes, &kmap, 64, row, &k_full[s]);
                    tma_load_2d(st + kTileBytes, &vmap, 0, row, &k_full[s]);
                    tma_load_2d(st + kTileBytes + kPanelBytes, &vmap, 64, row, &k_full[s]);
                }
            }
            __syncwarp();
        }
        if (lane == 0) {
            for (int b = 0; b < 2; ++b) {
                const int uses = (n_my - b + 1) / 2;
                if (uses > 0) mbar_wait(&t_empty[b], (uses - 1) & 1, p.err, kErrDkvDrain);
            }
            for (int s = 0; s < p.stages && s < n_my; ++s) {
                const int last = ((n_my - 1 - s) / p.stages) * p.stages + s;
                mbar_wait(&k_empty[s], (last / p.stages) & 1, p.err, kErrDkvDrain);
            }
        }
        __syncwarp();
    } else {
        const uint32_t lane_base = static_cast<uint32_t>(warp * 32) << 16;
        for (int j = 0; j < n_my; ++j) {
            const int buf = j & 1;
            const int use = j >> 1;
            if (ok) ok = mbar_wait(&t_full[buf], use & 1, p.err, kErrDkvTFull);
            tc_fence_after();
            float lsum[2];
#pragma unroll
            for (int t = 0; t < 2; ++t) {
                const uint32_t col = static_cast<uint32_t>(buf * (2 * kProjCols) + t * kProjCols);
                float a0[32], a1[32], a2[32];
                tmem_ld32(taddr + lane_base + col, a0);
                tmem_ld32(taddr + lane_base + col + 32, a1);
                tmem_ld32(taddr + lane_base + col + 64, a2);
                float acc = 0.f;
#pragma unroll
                for (int b = 0; b < 32; ++b) {
                    const float y = (a0[b] + a1[b]) + a2[b];
                    acc = fmaf(y, y, acc);
                }
                lsum[t] = acc;
            }
            tc_fence_before();
            mbar_arrive(&t_empty[buf]);
            const int tok = (t_begin + j) * kTileTokens + warp * 32 + lane;
            if (tok < p.K) out[static_cast<int64_t>(unit) * p.N + tok] = lsum[0] * lsum[1];
        }
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == kConsumerWarps) tmem_dealloc(taddr, kTmemCols);
}

}  // namespace

size_t dkv_smem_bytes(int stages) { return dkv_layout(stages).total + 1024; }

cudaError_t dkv_set_attributes(size_t smem_bytes) {
    return cudaFuncSetAttribute(dkv_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem_bytes));
}

cudaError_t launch_dkv(const CUtensorMap& kmap, const CUtensorMap& vmap, const DkvParams& p, int units,
                       size_t smem_bytes, cudaStream_t s) {
    const int ctas = (p.n_tiles_k + p.tiles_per_cta - 1) / p.tiles_per_cta;
    dkv_kernel<<<dim3(static_cast<unsigned>(ctas), static_cast<unsigned>(units), static_cast<unsigned>(p.batch.n)),
                 kThreads, smem_bytes, s>>>(kmap, vmap, p);
    return cudaGetLastError();
}

}  // namespace vase
