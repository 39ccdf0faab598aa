// Decode-step attention over the cache the eviction keeps (Eq. (1), Sec. 2):
//     o_g = sum_i alpha_gi v_i,  alpha_gi = softmax_i(q_g . k_i / sqrt(d)),
// for the G query heads g of each KV head, over the `fill` slots of the unit in
// slot order (slots 0..fill-1 of k_cache / v_cache, the layout the eviction
// leaves).
//
// Two kernels compute it.  With G >= 3 query heads per KV head both contractions
// run on the tensor cores (decode_tc_kernel, tcgen05 with accumulators in TMEM):
//   S   = K_c . Q^T     M = 64 slots of chunk c, N = 16 (query heads, zero-padded), K = d
//   O^T = V_c^T . P^T   M = d, N = 2G padded to 16 or 32, K = 64 slots
// where P holds the chunk's softmax weights exp2(s - m) split into a bf16 high
// part and a bf16 low part (two columns per head, p = hi + lo to about 2^-17), so
// the bf16 operand keeps fp32-level accuracy.  A of the second MMA is the V tile
// as TMA wrote it (slot rows of 64 dims, 128-byte swizzle): the MN-major form.
//
// One thread-block cluster per unit splits the unit's slots: CTA r takes chunks
// r, r + C, ... of 64 slots.  Warp roles: warp 0 issues the TMA loads of K and V
// (three-stage ring), warp 1 issues the MMAs, warps 2..5 (one per TMEM lane
// quadrant) read the scores (thread = slot), keep the running max per head
// (raised only when a chunk's max passes it by more than 2^8, so the weights
// stay below 2^8 and most chunks need no rescaling), write P, and fold each
// chunk's O^T columns into fp32 registers (thread = output dimension).  S and O
// are double-buffered in TMEM, so the MMAs of chunk c+1 overlap the softmax of
// chunk c.  The CTAs of a cluster fold their (max, sum, output) states through
// distributed shared memory.
//
// With G <= 2 the dot products are a small share of the work and the kernel on
// the CUDA cores (decode_simt_kernel) keeps a smaller footprint (50 KB of
// shared memory and 5 warps per CTA, 32-slot chunks, bulk copies instead of
// tensor maps), so about twice as many CTAs share an SM and the next launch's
// prologue fits beside them: each consumer warp owns 8 slots of every chunk,
// four lanes per slot split the score dot product, each lane owns 4 output
// dimensions of the weighted V sum, and the warps keep their own running
// softmax states, folded per CTA and then per cluster as above.
//
// Both are bound by reading K and V once from HBM: 2 * 256 bytes per slot.
#include <cfloat>

#include <cuda_bf16.h>

#include "kernels.cuh"
#include "ptx.cuh"

namespace vase {

namespace {

// ================================================================== CUDA-core kernel (G <= 2)
#include "decode_simt.cuh"

// ================================================================== tensor-core kernel (G >= 3)
namespace tc {

constexpr int kChunk = kDecodeTileRows;  // 64 slots: the M of the score MMA
constexpr int kStages = 3;
constexpr int kSoftWarps = 4;
constexpr int kThreads = 32 * (2 + kSoftWarps);
constexpr int kBuildWarps = 4;                             // store: the warps that write the V tiles
constexpr int kThreadsStore = kThreads + 32 * kBuildWarps;
constexpr uint32_t kBoxBytes = kChunk * 128;          // 64 rows x 64 dims bf16 (one TMA box)
constexpr uint32_t kStageBytes = 4 * kBoxBytes;       // K dims 0-63, K dims 64-127, V dims 0-63, V dims 64-127
// With the compressed value store the V tile of a stage is written by builder warps straight from the store (a
// bf16 slot's row from the ring, a coded slot's codes expanded), so a stage has the same size in both forms.
__host__ __device__ constexpr uint32_t stage_bytes_of(bool) { return kStageBytes; }
constexpr int kNS = 16;                               // score columns (query heads, padded)
constexpr float kLazyMax = 8.f;                       // log2 units

struct DecodeSmem {
    uint32_t stage_off;  // kStages x kStageBytes; after the last chunk: the CTA's fold state (res_o, res_ml)
    uint32_t q_off;      // Q as the score MMA's B operand: 2 panels x 16 rows x 128 B (K-major, 128-byte swizzle)
    uint32_t p_off;      // 2 buffers x NP rows x 128 B: P^T as the output MMA's B operand (K-major over slots)
    uint32_t red_off;    // [2][kSoftWarps][16] chunk maxima, [2][kSoftWarps] status flags (padded to 16),
                         // [kSoftWarps][16] sums, [kSoftWarps][16] bias sums (store)
    uint32_t mask_off;   // store: the unit's bf16 masks [kDecodeMaxMaskWords]
    uint32_t bar_off;
    uint32_t total;      // bytes from the 1024-aligned base
};

__host__ __device__ inline DecodeSmem decode_layout(int NP, bool store = false) {
    DecodeSmem L;
    uint32_t o = 0;
    L.stage_off = o;
    o += kStages * stage_bytes_of(store);
    L.q_off = o;
    o += 2 * kNS * 128;
    L.p_off = o;
    o += 2u * NP * 128;
    L.red_off = o;
    o += 4u * (4 * kSoftWarps * kNS + 16);
    L.mask_off = o;
    o += store ? 4u * kDecodeMaxMaskWords : 0u;
    L.bar_off = o;
    o += 8u * (3 * kStages + 9) + 16;  // full, empty, v_full (x kStages), s_full, s_empty, p_full, o_full (x2),
                                       // mma_done, TMEM slot
    L.total = (o + 15u) & ~15u;
    return L;
}

__device__ __forceinline__ float ex2(float x) {  // 2^x on the SFU (relative error about 2^-22; 2^-inf = 0)
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// MN-major operand with the 128-byte swizzle (rows of 64 consecutive M elements, one row per K index, as TMA
// writes a box of 64 dims x 64 slots): LBO = bytes between 64-element blocks along M, SBO = bytes between
// 8-row groups along K.
__device__ __forceinline__ uint64_t sw128_mnmajor_desc(uint32_t smem_addr, uint32_t lbo, uint32_t sbo) {
    uint64_t d = 0;
    d |= static_cast<uint64_t>((smem_addr & 0x3FFFFu) >> 4);
    d |= static_cast<uint64_t>(lbo >> 4) << 16;
    d |= static_cast<uint64_t>(sbo >> 4) << 32;
    d |= static_cast<uint64_t>(1u) << 46;
    d |= static_cast<uint64_t>(2u) << 61;
    return d;
}

// 32 lanes x 16 consecutive 32-bit columns, load and wait in one statement.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16]) {
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];\n\t"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr)
        : "memory");
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// The codes of dims 8q .. 8q+7 of a half row (kBits-bit fields, dim i at bit i*kBits of the little-endian words
// cw) as eight bf16 values: the integers themselves (exact in bf16: their fp32 bits' top half).
template <int kBits>
__device__ __forceinline__ uint4 expand8(const uint32_t* cw, int q) {
    uint32_t w[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const int b0 = (8 * q + 2 * e) * kBits, b1 = b0 + kBits;
        const uint32_t c0 = (cw[b0 >> 5] >> (b0 & 31)) & ((1u << kBits) - 1u);
        const uint32_t c1 = (cw[b1 >> 5] >> (b1 & 31)) & ((1u << kBits) - 1u);
        w[e] = (__float_as_uint(static_cast<float>(c0)) >> 16) | (__float_as_uint(static_cast<float>(c1)) & 0xFFFF0000u);
    }
    return make_uint4(w[0], w[1], w[2], w[3]);
}

// Byte offset of bf16 element (row, col) in a K-major panel of 128-byte rows with the 128-byte swizzle.
__device__ __forceinline__ uint32_t sw128_offset(int row, int col) {
    return static_cast<uint32_t>(row * 128 + ((((col >> 3) ^ (row & 7)) & 7) << 4) + ((col & 7) << 1));
}

// kStore: the values come from the compressed value store.  Four more warps (builders) write each stage's V
// tile from the store, in the layout TMA gives the bf16 form (rows of 64 dims, 128-byte swizzle): a bf16 slot's
// row read from the ring, a coded slot's row as its codes (integers, exact in bf16); they reuse a stage once its
// output MMA has read it (empty) and signal v_full.  A coded slot's weight in P is p s and its p z joins a
// per-head bias: o = sum p v' = sum (p s) Q + sum p z.
template <int NP, bool kStore>
__global__ void __launch_bounds__(kStore ? kThreadsStore : kThreads) decode_tc_kernel(const __grid_constant__ CUtensorMap kmap,
                                                               const __grid_constant__ CUtensorMap vmap,
                                                               const DecodeParams p) {
    constexpr int GH = NP / 2;  // query heads the instantiation handles
    constexpr uint32_t kTmemCols = NP == 16 ? 64 : 128;
    constexpr uint32_t kSB = stage_bytes_of(kStore);
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const DecodeSmem Ly = decode_layout(NP, kStore);
    uint32_t* mask_s = reinterpret_cast<uint32_t*>(smem + Ly.mask_off);
    uint8_t* stage = smem + Ly.stage_off;
    uint8_t* q_s = smem + Ly.q_off;
    uint8_t* p_s = smem + Ly.p_off;
    float* red = reinterpret_cast<float*>(smem + Ly.red_off);
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + Ly.bar_off);
    uint64_t* empty = full + kStages;
    uint64_t* v_full = empty + kStages;  // store: the builders have written the stage's V tile
    uint64_t* s_full = v_full + kStages;
    uint64_t* s_empty = s_full + 2;
    uint64_t* p_full = s_empty + 2;
    uint64_t* o_full = p_full + 2;
    uint64_t* mma_done = o_full + 2;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);

    const int tid = threadIdx.x;
    const int lane = tid & 31;
    const int warp = tid >> 5;
    const int G = p.G;
    const int C = p.cluster;
    const int rank = static_cast<int>(cluster_rank());
    const int unit = blockIdx.y;
    const int n_mine = rank < p.n_chunks ? (p.n_chunks - 1 - rank) / C + 1 : 0;  // >= 1 (C <= n_chunks)
    const int seq = unit / p.Hkv;
    const int head = unit - seq * p.Hkv;
    const int64_t unit_row = static_cast<int64_t>(unit) * p.N;

    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
            mbar_init(&v_full[s], kBuildWarps);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&s_full[b], 1);
            mbar_init(&s_empty[b], kSoftWarps);
            mbar_init(&p_full[b], kSoftWarps);
            mbar_init(&o_full[b], 1);
        }
        mbar_init(mma_done, 1);
        fence_mbar_init();
        // warm L2 with the first chunks while the preceding kernel finishes (L2 is where device memory is
        // coherent: rows it still writes are read fresh by the loads, which come after the wait below)
        for (int j = 0; j < min(kStages, n_mine); ++j) {
            const int s0 = (rank + j * C) * kChunk;
            const uint32_t bytes = static_cast<uint32_t>(min(kChunk, p.fill - s0)) * kRowBytes;
            asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p.kc + (unit_row + s0) * kVecPerRow),
                         "r"(bytes)
                         : "memory");
            if (!kStore)
                asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p.vc + (unit_row + s0) * kVecPerRow),
                             "r"(bytes)
                             : "memory");
        }
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, kTmemCols);
        tmem_relinquish();
    }
    asm volatile("griddepcontrol.wait;" ::: "memory");  // query and cache rows of preceding kernels are visible
    // store: the unit's bf16 masks and the ring row of its first bf16 value
    int ring_head = 0;
    if (kStore) {
        for (int w = tid; w < p.mask_words; w += kThreadsStore) mask_s[w] = p.rmask[static_cast<int64_t>(unit) * p.mask_words + w];
        ring_head = p.ring_state[4 * unit];
        if (ring_head < 0 || ring_head >= p.hp_cap) {  // not a state the store kernels wrote
            if (tid == 0) record_error(p.err, kErrDecodeMask);
            ring_head = 0;
        }
        __syncthreads();
    }
    // bf16 mask of a chunk's slots (store), limited to its filled rows
    auto chunk_bf16 = [&](int c, int rows) -> uint64_t {
        const uint32_t w0 = 2 * c < p.mask_words ? mask_s[2 * c] : 0u;
        const uint32_t w1 = 2 * c + 1 < p.mask_words ? mask_s[2 * c + 1] : 0u;
        const uint64_t m = static_cast<uint64_t>(w0) | static_cast<uint64_t>(w1) << 32;
        return rows >= 64 ? m : m & ((1ull << rows) - 1ull);
    };
    // chunk j of this CTA into stage j % kStages
    auto load_chunk = [&](int j) {
        const int s = j % kStages;
        const int c = rank + j * C;
        const int32_t y = p.row_base + static_cast<int32_t>(unit_row) + c * kChunk;
        uint8_t* st = stage + s * kSB;
        if (!kStore) {
            mbar_arrive_expect_tx(&full[s], kStageBytes);
            tma_load_2d(st, &kmap, 0, y, &full[s]);
            tma_load_2d(st + kBoxBytes, &kmap, 64, y, &full[s]);
            tma_load_2d(st + 2 * kBoxBytes, &vmap, 0, y, &full[s]);
            tma_load_2d(st + 3 * kBoxBytes, &vmap, 64, y, &full[s]);
            return;
        }
        mbar_arrive_expect_tx(&full[s], 2 * kBoxBytes);  // K only: the builders write the V tile
        tma_load_2d(st, &kmap, 0, y, &full[s]);
        tma_load_2d(st + kBoxBytes, &kmap, 64, y, &full[s]);
    };
    if (tid == 0)
        for (int j = 0; j < min(kStages, n_mine); ++j) load_chunk(j);  // the ring's first fill, before anything else
    // Q rows of this KV head (query heads head*G .. head*G+G-1 of sequence seq) as the B operand; rows >= G zero
    {
        const uint4* qrow =
            p.q + (static_cast<int64_t>(seq) * p.Hkv * G + static_cast<int64_t>(head) * G) * kVecPerRow;
        for (int i = tid; i < kNS * kVecPerRow; i += (kStore ? kThreadsStore : kThreads)) {
            const int n = i / kVecPerRow;
            const int c = i - n * kVecPerRow;  // 16-byte piece: dims 8c .. 8c+7
            const uint4 v = n < G ? qrow[n * kVecPerRow + c] : make_uint4(0, 0, 0, 0);
            *reinterpret_cast<uint4*>(q_s + (c >> 3) * (kNS * 128) + sw128_offset(n, (c & 7) * 8)) = v;
        }
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // Q writes -> tensor-core reads
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    const uint32_t t_s = tmem;         // S buffers: columns [0, 16) and [16, 32)
    const uint32_t t_o = tmem + 32;    // O buffers: columns [32, 32 + NP) and [32 + NP, 32 + 2 NP)

    bool ok = true;
    if (warp == 0) {
        // ---- TMA producer: the rest of the chunks as the MMAs free their stages
        if (lane == 0) {
            int issued = min(kStages, n_mine);
            for (int j = kStages; j < n_mine; ++j) {
                if (!mbar_wait(&empty[j % kStages], ((j / kStages) - 1) & 1, p.err, kErrDecodeEmpty)) break;
                load_chunk(j);
                issued = j + 1;
            }
            for (int j = max(0, issued - kStages); j < issued; ++j)  // every load landed before the CTA exits
                mbar_wait(&full[j % kStages], (j / kStages) & 1, p.err, kErrDecodeDrain);
        }
    } else if (warp == 1) {
        // ---- MMA issuer: S(j), then O(j-1), so the softmax of chunk j overlaps the output MMA of chunk j-1
        if (lane == 0) {
            constexpr uint32_t idesc_s = idesc_bf16_f32(64, kNS);
            constexpr uint32_t idesc_o = idesc_bf16_f32(128, NP) | (1u << 15);  // A (V^T) MN-major
            const uint32_t q_addr = smem_u32(q_s);
            auto issue_o = [&](int jj) -> bool {
                const int b = jj & 1;
                if (!mbar_wait(&p_full[b], (jj >> 1) & 1, p.err, kErrDecodeFull)) return false;
                if (kStore && !mbar_wait(&v_full[jj % kStages], (jj / kStages) & 1, p.err, kErrDecodeFull)) return false;
                tc_fence_after();
                const uint32_t v_addr = smem_u32(stage + (jj % kStages) * kSB + 2 * kBoxBytes);
                const uint32_t p_addr = smem_u32(p_s + b * NP * 128);
#pragma unroll
                for (int kk = 0; kk < kChunk / 16; ++kk)
                    tc_mma_bf16(t_o + b * NP, sw128_mnmajor_desc(v_addr + kk * 2048, kBoxBytes, 1024),
                                sw128_kmajor_desc(p_addr + kk * 32), idesc_o, kk > 0 ? 1u : 0u);
                tc_commit(&o_full[b]);
                tc_commit(&empty[jj % kStages]);  // K and V of the stage are consumed
                return true;
            };
            for (int j = 0; j < n_mine && ok; ++j) {
                const int s = j % kStages;
                const int b = j & 1;
                if (!mbar_wait(&full[s], (j / kStages) & 1, p.err, kErrDecodeFull) ||
                    (j >= 2 && !mbar_wait(&s_empty[b], ((j >> 1) - 1) & 1, p.err, kErrDecodeFull))) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t k_addr = smem_u32(stage + s * kSB);
#pragma unroll
                for (int kk = 0; kk < 8; ++kk)
                    tc_mma_bf16(t_s + b * kNS, sw128_kmajor_desc(k_addr + (kk >> 2) * kBoxBytes + (kk & 3) * 32),
                                sw128_kmajor_desc(q_addr + (kk >> 2) * (kNS * 128) + (kk & 3) * 32), idesc_s,
                                kk > 0 ? 1u : 0u);
                tc_commit(&s_full[b]);
                if (j >= 1 && !issue_o(j - 1)) ok = false;
            }
            if (ok) issue_o(n_mine - 1);
            // every MMA issued has finished before TMEM is freed (also on an error path)
            tc_commit(mma_done);
            mbar_wait(mma_done, 0, p.err, kErrDecodeDrain);
        }
    }

    // ---- softmax and output warps: quadrant qd of the TMEM lanes
    const int qd = warp & 3;
    const int sw = warp - 2;  // 0..3 among the softmax warps
    float acc[GH];            // thread = output dimension 32 qd + lane
    float m_run[GH];
    float l_part[GH];         // this thread's slot share of the sum (threads with lane < 16 own a slot)
    float b_part[GH];         // store: this thread's slot share of sum p z over coded slots
#pragma unroll
    for (int g = 0; g < GH; ++g) {
        acc[g] = 0.f;
        m_run[g] = -INFINITY;
        l_part[g] = 0.f;
        b_part[g] = 0.f;
    }
    if (warp >= 2 && warp < 2 + kSoftWarps) {
        const uint32_t lane_base = static_cast<uint32_t>(32 * qd) << 16;
        float alpha_prev[GH];
#pragma unroll
        for (int g = 0; g < GH; ++g) alpha_prev[g] = 1.f;
        auto fold_o = [&](int jj, const float (&alpha)[GH]) -> bool {
            const int b = jj & 1;
            if (!mbar_wait(&o_full[b], (jj >> 1) & 1, p.err, kErrDecodeFull)) return false;
            tc_fence_after();
            float o[16];
#pragma unroll
            for (int h = 0; h < NP / 16; ++h) {
                tmem_ld16(t_o + lane_base + b * NP + 16 * h, o);
#pragma unroll
                for (int e = 0; e < 16; e += 2) {
                    const int g = 8 * h + e / 2;
                    acc[g] = fmaf(acc[g], alpha[g], o[e] + o[e + 1]);
                }
            }
            return true;
        };
        const int slot_l = 16 * qd + lane;  // the chunk slot of this thread (M = 64: lanes 0-15 of each quadrant)
        // A wait that runs out in one warp must not leave the others at the named barrier: each warp posts its
        // status before the barrier and all four leave the loop together.
        int* flags = reinterpret_cast<int*>(red + 2 * kSoftWarps * kNS);  // [2][kSoftWarps], beside red_l
        for (int j = 0; j < n_mine; ++j) {
            const int b = j & 1;
            const int s0 = (rank + j * C) * kChunk;
            const int rows = min(kChunk, p.fill - s0);
            // store: this slot's (s, z), requested before the wait for the scores so that its latency hides there
            // (a bf16 slot's pair is read and ignored)
            float2 szv = make_float2(1.f, 0.f);
            if (kStore && lane < 16 && slot_l < rows)
                szv = reinterpret_cast<const float2*>(p.qparams)[static_cast<int64_t>(unit) * p.Kp + s0 + slot_l];
            float sv[16];
            const bool got = ok && mbar_wait(&s_full[b], (j >> 1) & 1, p.err, kErrDecodeFull);
            if (got) {
                tc_fence_after();
                tmem_ld16(t_s + lane_base + b * kNS, sv);
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&s_empty[b]);
            }
            const bool valid = got && lane < 16 && slot_l < rows;
            float sc[GH];
#pragma unroll
            for (int g = 0; g < GH; ++g) sc[g] = (valid && g < G) ? sv[g] * p.scale_log2 : -INFINITY;
            // chunk maxima: lanes 0-15 of each warp, then the four warps through shared memory
            float* red_j = red + b * kSoftWarps * kNS;
#pragma unroll
            for (int g = 0; g < GH; ++g) {
                float mx = sc[g];
                mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
                mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
                mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 4));
                mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 8));
                if (lane == 0) red_j[sw * kNS + g] = mx;
            }
            if (lane == 0) flags[b * kSoftWarps + sw] = got ? 1 : 0;
            named_bar(1, 32 * kSoftWarps);
            if (!(flags[b * kSoftWarps] & flags[b * kSoftWarps + 1] & flags[b * kSoftWarps + 2] &
                  flags[b * kSoftWarps + 3])) {
                ok = false;
                break;
            }
            float alpha[GH];
#pragma unroll
            for (int g = 0; g < GH; ++g) {
                float mc = red_j[g];
#pragma unroll
                for (int w = 1; w < kSoftWarps; ++w) mc = fmaxf(mc, red_j[w * kNS + g]);
                const bool raise = mc > m_run[g] + kLazyMax;  // the same decision in every thread
                alpha[g] = raise ? ex2(m_run[g] - mc) : 1.f;  // 0 on the first chunk (m_run = -inf)
                if (raise) m_run[g] = mc;
            }
            // the rows past the unit's fill in a ragged chunk hold stale bytes: zero their V rows (P is 0 there)
            uint8_t* vt = stage + (j % kStages) * kSB + 2 * kBoxBytes;
            if (!kStore && rows < kChunk) {  // (the store's builders write those rows themselves)
                for (int i = tid - 64; i < (kChunk - rows) * 16; i += 32 * kSoftWarps) {
                    const int r = rows + (i >> 4);
                    const int c = i & 15;
                    *reinterpret_cast<uint4*>(vt + (c >> 3) * kBoxBytes + r * 128 + (c & 7) * 16) =
                        make_uint4(0, 0, 0, 0);
                }
            }
            float sz_s = 1.f, sz_z = 0.f;  // store: (s, z) of this thread's slot if it is coded
            if (kStore && lane < 16 && slot_l < rows && !((chunk_bf16(rank + j * C, rows) >> slot_l) & 1ull)) {
                sz_s = szv.x;
                sz_z = szv.y;
            }
            // weights exp2(s - m) <= 2^8 as hi + lo bf16 pairs: P^T rows 2g and 2g + 1, column = slot; a coded
            // slot's column holds p s and its p z joins the head's bias
            if (lane < 16) {
                uint8_t* pb = p_s + b * NP * 128;
#pragma unroll
                for (int g = 0; g < GH; ++g) {
                    const float w0 = g < G ? ex2(sc[g] - m_run[g]) : 0.f;
                    l_part[g] = fmaf(l_part[g], alpha[g], w0);
                    if (kStore) b_part[g] = fmaf(b_part[g], alpha[g], w0 * sz_z);
                    const float w = kStore ? w0 * sz_s : w0;
                    const __nv_bfloat16 hi = __float2bfloat16_rn(w);
                    const __nv_bfloat16 lo = __float2bfloat16_rn(w - __bfloat162float(hi));
                    *reinterpret_cast<__nv_bfloat16*>(pb + sw128_offset(2 * g, slot_l)) = hi;
                    *reinterpret_cast<__nv_bfloat16*>(pb + sw128_offset(2 * g + 1, slot_l)) = lo;
                }
            }
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // P and zeroed V rows -> tensor core
            __syncwarp();
            if (lane == 0) mbar_arrive(&p_full[b]);
            if (j >= 1 && !fold_o(j - 1, alpha_prev)) ok = false;  // seen by all four at the next barrier
#pragma unroll
            for (int g = 0; g < GH; ++g) alpha_prev[g] = alpha[g];
        }
        if (ok && !fold_o(n_mine - 1, alpha_prev)) ok = false;
        tc_fence_before();
    } else if (kStore && warp >= 2 + kSoftWarps) {
        // ---- builders (store): the V tile of every chunk of this CTA.  Thread (row r, half) writes dims
        // 64 half .. 64 half + 63 of slot row r, 16 bytes (8 dims) at a time into the 128-byte swizzled row: a bf16
        // slot's from its ring row (the k-th bf16 slot of the chunk is ring entry pre + k behind the head), a coded
        // slot's as its codes, rows past the fill as zeros (P is 0 there)
        const int t = tid - 32 * (2 + kSoftWarps);
        const int r = t >> 1, half = t & 1;
        int pre_val = 0, pre_upto = 0;  // bf16 values of the unit before mask word pre_upto
        for (int j = 0; j < n_mine; ++j) {
            const int s = j % kStages;
            const int c = rank + j * C;
            const int s0 = c * kChunk;
            const int rows = min(kChunk, p.fill - s0);
            // the stage's previous tile has been read by its output MMA
            if (j >= kStages && !mbar_wait(&empty[s], ((j / kStages) - 1) & 1, p.err, kErrDecodeEmpty)) break;
            const uint64_t m = chunk_bf16(c, rows);
            while (pre_upto < 2 * c) {
                if (pre_upto < p.mask_words) pre_val += __popc(mask_s[pre_upto]);
                ++pre_upto;
            }
            uint4 v[8];
#pragma unroll
            for (int q = 0; q < 8; ++q) v[q] = make_uint4(0, 0, 0, 0);
            if (r < rows && ((m >> r) & 1ull)) {
                const int k = pre_val + __popcll(m & ((1ull << r) - 1ull));
                if (k < p.hp_cap) {
                    int at = ring_head + k;
                    at -= at >= p.hp_cap ? p.hp_cap : 0;
                    const uint4* src = p.hp_rows + (static_cast<int64_t>(unit) * p.hp_cap + at) * kVecPerRow + half * 8;
#pragma unroll
                    for (int q = 0; q < 8; ++q) v[q] = src[q];
                } else {  // masks that do not match the ring: a zero row
                    record_error(p.err, kErrDecodeMask);
                }
            } else if (r < rows) {
                const int bits = p.bits;
                const uint4* cr = reinterpret_cast<const uint4*>(
                    p.codes + (static_cast<int64_t>(unit) * p.Kq + s0 + r) * p.code_row + half * 8 * bits);
                uint32_t cw[16];
                if (bits == 8) {
#pragma unroll
                    for (int i = 0; i < 4; ++i) *reinterpret_cast<uint4*>(cw + 4 * i) = cr[i];
#pragma unroll
                    for (int q = 0; q < 8; ++q) v[q] = expand8<8>(cw, q);
                } else if (bits == 4) {
#pragma unroll
                    for (int i = 0; i < 2; ++i) *reinterpret_cast<uint4*>(cw + 4 * i) = cr[i];
#pragma unroll
                    for (int q = 0; q < 8; ++q) v[q] = expand8<4>(cw, q);
                } else {
                    *reinterpret_cast<uint4*>(cw) = cr[0];
#pragma unroll
                    for (int q = 0; q < 8; ++q) v[q] = expand8<2>(cw, q);
                }
            }

            uint8_t* dst = stage + s * kSB + 2 * kBoxBytes + half * kBoxBytes + r * 128;
#pragma unroll
            for (int q = 0; q < 8; ++q) *reinterpret_cast<uint4*>(dst + (((q ^ (r & 7)) & 7) << 4)) = v[q];
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // tile writes -> tensor-core reads
            __syncwarp();
            if (lane == 0) mbar_arrive(&v_full[s]);
        }
    }
    __syncthreads();  // every MMA read and TMEM load is done; the stage area is free
    if (warp == 1) tmem_dealloc(tmem, kTmemCols);

    // ---- the CTA's state: per head the running max, the sum over its slots and the output row
    float* res_o = reinterpret_cast<float*>(stage);                       // [GH][d]
    float* res_ml = reinterpret_cast<float*>(stage + GH * kHeadDim * 4);  // [GH][2]
    float* red_l = red + 2 * kSoftWarps * kNS + 16;                       // [kSoftWarps][16] (after the flags)
    float* red_b = red_l + kSoftWarps * kNS;                              // [kSoftWarps][16] bias sums (store)
    if (warp >= 2 && warp < 2 + kSoftWarps) {
#pragma unroll
        for (int g = 0; g < GH; ++g) {
            float sum = l_part[g];
            sum += __shfl_xor_sync(0xffffffffu, sum, 1);
            sum += __shfl_xor_sync(0xffffffffu, sum, 2);
            sum += __shfl_xor_sync(0xffffffffu, sum, 4);
            sum += __shfl_xor_sync(0xffffffffu, sum, 8);
            sum += __shfl_xor_sync(0xffffffffu, sum, 16);
            if (lane == 0) red_l[sw * kNS + g] = sum;
            if (kStore) {
                float bs = b_part[g];
                bs += __shfl_xor_sync(0xffffffffu, bs, 1);
                bs += __shfl_xor_sync(0xffffffffu, bs, 2);
                bs += __shfl_xor_sync(0xffffffffu, bs, 4);
                bs += __shfl_xor_sync(0xffffffffu, bs, 8);
                bs += __shfl_xor_sync(0xffffffffu, bs, 16);
                if (lane == 0) red_b[sw * kNS + g] = bs;
            } else if (g < G) {
                res_o[g * kHeadDim + 32 * qd + lane] = acc[g];
            }
        }
        named_bar(1, 32 * kSoftWarps);
        if (kStore) {  // the output rows with the heads' bias: sum p z over every coded slot, added to each dim
#pragma unroll
            for (int g = 0; g < GH; ++g)
                if (g < G)
                    res_o[g * kHeadDim + 32 * qd + lane] =
                        acc[g] + ((red_b[g] + red_b[kNS + g]) + (red_b[2 * kNS + g] + red_b[3 * kNS + g]));
        }
        if (tid - 64 < G) {
            const int g = tid - 64;
            res_ml[2 * g] = m_run[0];
#pragma unroll
            for (int h = 1; h < GH; ++h)
                if (h == g) res_ml[2 * g] = m_run[h];
            res_ml[2 * g + 1] = red_l[g] + red_l[kNS + g] + red_l[2 * kNS + g] + red_l[3 * kNS + g];
        }
    }
    cluster_sync();  // every CTA's state is in its shared memory
    {
        // ---- fold the cluster: CTA r writes outputs [r * per, (r + 1) * per) of the unit's G x d
        const int total = G * kHeadDim;
        const int per = (total + C - 1) / C;
        const int end = min(total, (rank + 1) * per);
        for (int i = rank * per + tid; i < end; i += (kStore ? kThreadsStore : kThreads)) {
            const int g = i / kHeadDim;
            const int d = i - g * kHeadDim;
            float2 ml[kDecodeMaxCluster];
            float o[kDecodeMaxCluster];
            float M = -INFINITY;
#pragma unroll
            for (int r = 0; r < kDecodeMaxCluster; ++r) {
                if (r < C) {
                    ml[r] = ld_cluster_f32x2(map_to_rank(res_ml + g * 2, r));
                    o[r] = ld_cluster_f32(map_to_rank(res_o + g * kHeadDim + d, r));
                    M = fmaxf(M, ml[r].x);
                }
            }
            float L = 0.f, O = 0.f;
#pragma unroll
            for (int r = 0; r < kDecodeMaxCluster; ++r) {
                if (r < C) {
                    const float f = ex2(ml[r].x - M);
                    L = fmaf(ml[r].y, f, L);
                    O = fmaf(o[r], f, O);
                }
            }
            p.out[(static_cast<int64_t>(seq) * p.Hkv * G + static_cast<int64_t>(head) * G + g) * kHeadDim + d] =
                O / L;
        }
    }
    cluster_sync();  // every CTA has read what it needs from the others' shared memory
}

template <int NP, bool kStore>
cudaError_t launch_np(const CUtensorMap& kmap, const CUtensorMap& vmap, const DecodeParams& p, size_t smem_bytes,
                      cudaStream_t s) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(p.cluster), static_cast<unsigned>(p.units));
    cfg.blockDim = dim3(kStore ? kThreadsStore : kThreads);
    cfg.dynamicSmemBytes = smem_bytes;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = static_cast<unsigned>(p.cluster);
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // see griddepcontrol in the kernel
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, decode_tc_kernel<NP, kStore>, kmap, vmap, p);
}

}  // namespace tc

// The tensor cores from G = 3 on (below, the dot products are a small share of the work); the compressed value
// store always, since its V tiles are written by the builder warps off the softmax path.
bool use_tc(int G, bool store) { return store || G >= 3; }
int tc_np(int G) { return G <= 8 ? 16 : 32; }
// CTAs per unit: enough clusters to fill the GPU `per_sm` CTAs deep (the kernel's residency), at most
// kDecodeMaxCluster and at most one CTA per chunk.
int cluster_for(int units, int n_chunks, int num_sms, int per_sm) {
    int c = (per_sm * num_sms) / (units > 0 ? units : 1);
    c = c < 1 ? 1 : c > kDecodeMaxCluster ? kDecodeMaxCluster : c;
    return c < n_chunks ? c : (n_chunks > 0 ? n_chunks : 1);
}

}  // namespace

size_t decode_smem_bytes(int G, bool store) {
    return use_tc(G, store) ? tc::decode_layout(tc_np(G), store).total + 1024 : simt::decode_layout(2).total;
}

cudaError_t decode_set_attributes(int G, size_t smem_bytes, bool store) {
    const int bytes = static_cast<int>(smem_bytes);
    if (!use_tc(G, store))
        return cudaFuncSetAttribute(simt::decode_simt_kernel<2, 0>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (store)
        return tc_np(G) == 16
                   ? cudaFuncSetAttribute(tc::decode_tc_kernel<16, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes)
                   : cudaFuncSetAttribute(tc::decode_tc_kernel<32, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    return tc_np(G) == 16
               ? cudaFuncSetAttribute(tc::decode_tc_kernel<16, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes)
               : cudaFuncSetAttribute(tc::decode_tc_kernel<32, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
}

cudaError_t launch_decode(const CUtensorMap& kmap, const CUtensorMap& vmap, DecodeParams p, size_t smem_bytes,
                          int num_sms, cudaStream_t s) {
    if (!use_tc(p.G, p.ring_state != nullptr)) {
        p.n_chunks = (p.fill + simt::kChunk - 1) / simt::kChunk;
        p.cluster = cluster_for(p.units, p.n_chunks, num_sms, 4);
        return simt::launch_gp<2, 0>(p, smem_bytes, s);
    }
    p.n_chunks = (p.fill + tc::kChunk - 1) / tc::kChunk;
    p.cluster = cluster_for(p.units, p.n_chunks, num_sms, 2);  // two CTAs per SM
    if (p.ring_state)  // the compressed value store
        return tc_np(p.G) == 16 ? tc::launch_np<16, true>(kmap, vmap, p, smem_bytes, s)
                                : tc::launch_np<32, true>(kmap, vmap, p, smem_bytes, s);
    return tc_np(p.G) == 16 ? tc::launch_np<16, false>(kmap, vmap, p, smem_bytes, s)
                            : tc::launch_np<32, false>(kmap, vmap, p, smem_bytes, s);
}

}  // namespace vase
