// The CUDA-core decode-attention kernel (one query head pair per paired FMA), shared by decode.cu (bf16 values)
// and decode_mixed.cu (values of unreserved slots read from b-bit codes).  Included inside an unnamed namespace
// by each of them.
#pragma once

namespace simt {

constexpr int kChunk = 32;    // slots per stage: 8 per consumer warp
constexpr int kStages = 3;
constexpr int kConsumerWarps = kChunk / 8;      // 8 slots per consumer warp
constexpr int kThreads = 32 * (kConsumerWarps + 1);   // + one producer warp
constexpr uint32_t kChunkBytes = kChunk * kRowBytes;
// Query rows in shared memory, fp32 and pre-scaled by log2(e)/sqrt(d): per head, 16 pieces of 8 dimensions,
// each padded to 12 floats so that the eight lanes of a quarter-warp reading eight different pieces hit
// distinct banks.
constexpr int kQPieceFloats = 12;
// The running max of a warp is raised only when a score exceeds it by more than this (log2 units).
constexpr float kLazyMax = 8.f;

// Stage of one chunk: K rows, V rows (bf16; with b-bit values the chunk's reserved rows compacted at the front
// and the rows of slots past the quantized ones at their own rows), then with b-bit values the chunk's code
// rows and (s, z).
__host__ __device__ constexpr uint32_t stage_bytes(int bits) {
    return 2 * kChunkBytes + (bits > 0 ? kChunk * 16u * bits + kChunk * 8u : 0u);
}

struct DecodeSmem {
    uint32_t stage_off;  // kStages stages; after the last chunk: the fold areas below
    uint32_t fold_o;     // [warps][Gp][d] per-warp output sums (in the stage area)
    uint32_t res_o;      // [Gp][d] the CTA's output sum (in the stage area)
    uint32_t res_ml;     // [Gp][2] the CTA's (max, sum) (in the stage area)
    uint32_t q_off;      // [Gp][16][12] fp32
    uint32_t pw_off;     // [warps][8][Gp][2] softmax weights of the warp's slots, each twice
    uint32_t wml_off;    // [warps][Gp][2] per-warp (max, sum)
    uint32_t mask_off;   // b-bit values: [mask_words] the unit's reserved-slot masks
    uint32_t bar_off;    // full[kStages], empty[kStages]
    uint32_t total;
};

__host__ __device__ inline DecodeSmem decode_layout(int Gp, int bits = 0, int mask_words = 0) {
    DecodeSmem L;
    uint32_t o = 0;
    L.stage_off = o;
    L.fold_o = o;
    L.res_o = L.fold_o + 4u * kConsumerWarps * Gp * kHeadDim;
    L.res_ml = L.res_o + 4u * Gp * kHeadDim;
    o += kStages * stage_bytes(bits);
    L.q_off = o;
    o += 4u * Gp * 16 * kQPieceFloats;
    L.pw_off = o;
    o += 8u * kConsumerWarps * 8 * Gp;
    L.wml_off = o;
    o += 4u * kConsumerWarps * Gp * 2;
    L.mask_off = o;
    if (bits > 0) o += 4u * ((mask_words + 3) & ~3);
    o = (o + 15u) & ~15u;
    L.bar_off = o;
    o += 8u * 2 * kStages;
    L.total = (o + 15u) & ~15u;
    return L;
}

__host__ __device__ constexpr uint32_t low_mask(int n) { return n >= 32 ? 0xFFFFFFFFu : (n <= 0 ? 0u : (1u << n) - 1u); }

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

// 2^x on the SFU (ex2.approx.ftz: relative error about 2^-22; 2^-inf = 0).
__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ float2 bf16x2_to_f32x2(uint32_t w) { return make_float2(bf16_lo(w), bf16_hi(w)); }

__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
    asm volatile("cp.async.bulk.shared::cta.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                     smem_u32(dst)),
                 "l"(src), "r"(bytes), "r"(smem_u32(bar))
                 : "memory");
}

// kBits = 0: bf16 values.  kBits = 2, 4, 8: slots below Kq that the chunk's reserved mask leaves out read their
// values from b-bit codes, v' = Q s + z.
template <int Gp, int kBits>
__global__ void __launch_bounds__(kThreads) decode_simt_kernel(const DecodeParams p) {
    extern __shared__ __align__(16) uint8_t smem_raw[];
    constexpr uint32_t kStageBytes = stage_bytes(kBits);
    constexpr uint32_t kCodeRow = 16u * kBits;  // bytes of one code row (d * bits / 8)
    const DecodeSmem Ly = decode_layout(Gp, kBits, kBits > 0 ? p.mask_words : 0);
    uint32_t* mask_s = reinterpret_cast<uint32_t*>(smem_raw + Ly.mask_off);
    uint8_t* stage = smem_raw + Ly.stage_off;
    float* q_s = reinterpret_cast<float*>(smem_raw + Ly.q_off);
    float* wml = reinterpret_cast<float*>(smem_raw + Ly.wml_off);
    uint64_t* full = reinterpret_cast<uint64_t*>(smem_raw + Ly.bar_off);
    uint64_t* empty = full + kStages;
    const int tid = threadIdx.x;
    const int lane = tid & 31;
    const int warp = tid >> 5;
    const int G = p.G;
    const int C = p.cluster;
    const int rank = static_cast<int>(cluster_rank());
    const int unit = blockIdx.y;
    const int n_mine = rank < p.n_chunks ? (p.n_chunks - 1 - rank) / C + 1 : 0;
    const int64_t unit_row = static_cast<int64_t>(unit) * p.N;
    const int seq = unit / p.Hkv;
    const int head = unit - seq * p.Hkv;

    const int producer = 32 * kConsumerWarps;  // lane 0 of the last warp
    // chunk j of this CTA (slots (rank + j*C) * chunk ...) into stage j % kStages: the bulk part (K rows; with
    // b-bit values also the code rows and (s, z) of the slots below Kq), then (issue_bf16) the bf16 V rows
    auto issue = [&](int j) {
        const int s = j % kStages;
        const int s0 = (rank + j * C) * kChunk;
        const int rows = min(kChunk, p.fill - s0);
        const uint32_t bytes = static_cast<uint32_t>(rows) * kRowBytes;
        uint8_t* kdst = stage + s * kStageBytes;
        if (kBits == 0) {
            mbar_arrive_expect_tx(&full[s], 2 * bytes);
            bulk_load(kdst, p.kc + (unit_row + s0) * kVecPerRow, bytes, &full[s]);
            bulk_load(kdst + kChunkBytes, p.vc + (unit_row + s0) * kVecPerRow, bytes, &full[s]);
            return;
        }
        const int rq = max(0, min(rows, p.Kq - s0));
        const uint32_t qp_bytes = (static_cast<uint32_t>(rq) * 8u + 15u) & ~15u;
        mbar_arrive_expect_tx(&full[s], bytes + static_cast<uint32_t>(rq) * kCodeRow + qp_bytes);
        bulk_load(kdst, p.kc + (unit_row + s0) * kVecPerRow, bytes, &full[s]);
        if (rq > 0) {
            const int64_t qrow = static_cast<int64_t>(unit) * p.Kq + s0;
            bulk_load(kdst + 2 * kChunkBytes, p.codes + qrow * kCodeRow, static_cast<uint32_t>(rq) * kCodeRow, &full[s]);
            bulk_load(kdst + 2 * kChunkBytes + kChunk * kCodeRow, p.qparams + (static_cast<int64_t>(unit) * p.Kp + s0) * 2,
                      qp_bytes, &full[s]);
        }
    };
    // b-bit values: the chunk's reserved slots below Kq (mask bits) read their bf16 rows from the reserved cache
    // (contiguous there: slot order), copied to the first rows of the stage's V area; slots appended since the
    // quantization (rows >= rq) read the cache rows, at their own rows of the V area.
    auto chunk_mask = [&](int j) -> uint32_t {
        const int c = rank + j * C;
        const int s0 = c * kChunk;
        const int rq = max(0, min(min(kChunk, p.fill - s0), p.Kq - s0));
        return c < p.mask_words ? mask_s[c] & low_mask(rq) : 0u;
    };
    int pre_val = 0, pre_upto = 0;  // producer: reserved rows of the unit before chunk pre_upto
    int ring_head = 0;              // producer: compressed value store, the ring row of the unit's first bf16 value
    auto issue_bf16 = [&](int j) {
        const int s = j % kStages;
        const int c = rank + j * C;
        const int s0 = c * kChunk;
        const int rows = min(kChunk, p.fill - s0);
        const int rq = max(0, min(rows, p.Kq - s0));
        while (pre_upto < c && pre_upto < p.mask_words) pre_val += __popc(mask_s[pre_upto++]);
        int n_res = __popc(chunk_mask(j));
        if (pre_val + n_res > p.hp_cap) {  // masks that do not match the reserved cache: copy nothing past it
            record_error(p.err, kErrDecodeMask);
            n_res = max(0, p.hp_cap - pre_val);
        }
        uint8_t* vdst = stage + s * kStageBytes + kChunkBytes;
        mbar_arrive_expect_tx(&full[s], static_cast<uint32_t>(n_res + rows - rq) * kRowBytes);
        if (n_res > 0) {
            // the chunk's bf16 rows follow each other in the reserved cache; in the store's ring they may wrap
            int at = pre_val + ring_head;
            if (at >= p.hp_cap) at -= p.hp_cap;
            const int first = min(n_res, p.hp_cap - at);
            const int64_t row0 = static_cast<int64_t>(unit) * p.hp_cap;
            bulk_load(vdst, p.hp_rows + (row0 + at) * kVecPerRow, static_cast<uint32_t>(first) * kRowBytes, &full[s]);
            if (n_res > first)
                bulk_load(vdst + first * kRowBytes, p.hp_rows + row0 * kVecPerRow,
                          static_cast<uint32_t>(n_res - first) * kRowBytes, &full[s]);
        }
        if (rows > rq)
            bulk_load(vdst + rq * kRowBytes, p.vc + (unit_row + s0 + rq) * kVecPerRow,
                      static_cast<uint32_t>(rows - rq) * kRowBytes, &full[s]);
    };
    // Programmatic dependent launch: the next kernel of the stream may start its own prologue once every CTA of
    // this grid runs; it reads nothing this grid writes before its griddepcontrol.wait.
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    if (tid == producer) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&full[s], kBits > 0 ? 2 : 1);  // b-bit values: the bulk part and the bf16 rows arrive apart
            mbar_init(&empty[s], kConsumerWarps);
        }
        fence_mbar_init();
        // Warm L2 with the ring's first chunks while the preceding kernel finishes (a prefetch into L2 is only
        // a hint: L2 is where device memory is coherent, so rows the preceding kernel still writes are read
        // fresh by the copies below, which come after the wait).
        for (int j = 0; j < min(kStages, n_mine); ++j) {
            const int s0 = (rank + j * C) * kChunk;
            const uint32_t bytes = static_cast<uint32_t>(min(kChunk, p.fill - s0)) * kRowBytes;
            asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p.kc + (unit_row + s0) * kVecPerRow),
                         "r"(bytes)
                         : "memory");
            if (kBits == 0) {
                asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p.vc + (unit_row + s0) * kVecPerRow),
                             "r"(bytes)
                             : "memory");
            } else if (s0 < p.Kq) {  // b-bit values: the code rows (bf16 rows are a minority)
                const uint32_t cbytes = static_cast<uint32_t>(min(kChunk, p.Kq - s0)) * kCodeRow;
                asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(
                                 p.codes + (static_cast<int64_t>(unit) * p.Kq + s0) * kCodeRow),
                             "r"(cbytes)
                             : "memory");
            }
        }
    }
    // everything the preceding kernels of the stream wrote (query rows, cache rows) is visible after this
    asm volatile("griddepcontrol.wait;" ::: "memory");
    if (tid == producer)
        for (int j = 0; j < min(kStages, n_mine); ++j) issue(j);  // the ring's first fill
    if (kBits > 0)  // the unit's reserved-slot masks
        for (int w = tid; w < p.mask_words; w += kThreads) mask_s[w] = p.rmask[static_cast<int64_t>(unit) * p.mask_words + w];
    // the query rows of this KV head (query heads head*G .. head*G+G-1 of sequence seq) in fp32, scaled by
    // log2(e)/sqrt(d); a padding head reads zeros
    const uint32_t* qrow = reinterpret_cast<const uint32_t*>(
        p.q + (static_cast<int64_t>(seq) * p.Hkv * G + static_cast<int64_t>(head) * G) * kVecPerRow);
    for (int i = tid; i < Gp * (kHeadDim / 2); i += kThreads) {
        const int g = i / (kHeadDim / 2);
        const int dp = i - g * (kHeadDim / 2);  // dimension pair
        const uint32_t w = g < G ? qrow[g * (kHeadDim / 2) + dp] : 0u;
        float* dst = q_s + (g * 16 + (dp >> 2)) * kQPieceFloats + 2 * (dp & 3);
        dst[0] = bf16_lo(w) * p.scale_log2;
        dst[1] = bf16_hi(w) * p.scale_log2;
    }
    // running softmax state of a consumer warp: max per query head (uniform over the warp), this lane's share
    // of the sum (each slot counted by its four lanes), and the output sum over dims 4*lane .. 4*lane+3
    // With b-bit values a coded row contributes p (Q s + z) = (p s) Q + p z: its weight is stored as p s and
    // bias collects this lane's share of sum p z, added to every output dimension at the end.
    float m[Gp], l[Gp], bias[Gp];
    float2 acc[Gp][2];
#pragma unroll
    for (int g = 0; g < Gp; ++g) {
        m[g] = -INFINITY;
        l[g] = 0.f;
        bias[g] = 0.f;
        acc[g][0] = acc[g][1] = make_float2(0.f, 0.f);
    }
    __syncthreads();

    if (warp == kConsumerWarps) {
        // ---- producer: the rest of the ring's chunks as the consumers free their stages
        if (lane == 0) {
            if (kBits > 0 && p.ring_state) {
                ring_head = p.ring_state[4 * unit];
                if (ring_head < 0 || ring_head >= p.hp_cap) {  // not a state the store kernels wrote
                    record_error(p.err, kErrDecodeMask);
                    ring_head = 0;
                }
            }
            if (kBits > 0)
                for (int j = 0; j < min(kStages, n_mine); ++j) issue_bf16(j);
            int issued = min(kStages, n_mine);
            for (int j = kStages; j < n_mine; ++j) {
                if (!mbar_wait(&empty[j % kStages], ((j / kStages) - 1) & 1, p.err, kErrDecodeEmpty)) break;
                issue(j);
                if (kBits > 0) issue_bf16(j);
                issued = j + 1;
            }
            // every copy issued has landed before the stage area is reused (or the CTA exits)
            for (int j = max(0, issued - kStages); j < issued; ++j)
                mbar_wait(&full[j % kStages], (j / kStages) & 1, p.err, kErrDecodeDrain);
        }
    } else {
        // ---- consumers: warp w owns slots w*8 .. w*8+7 of every chunk; lane = 4 * slot + part
        const int sl = lane >> 2;    // slot of the warp's 8
        const int part = lane & 3;   // quarter of the dot product: pieces part + 4c (16-byte pieces of 8 dims)
        const int rot = sl & 1;      // neighbouring slots start at different pieces (bank spread)
        for (int j = 0; j < n_mine; ++j) {
            const int s = j % kStages;
            if (!mbar_wait(&full[s], (j / kStages) & 1, p.err, kErrDecodeFull)) break;
            const int s0 = (rank + j * C) * kChunk;
            const int nr = min(8, min(kChunk, p.fill - s0) - warp * 8);  // valid slots of the warp
            if (nr > 0) {
                const uint8_t* k_s = stage + s * kStageBytes + warp * 8 * kRowBytes;
                // b-bit values: the chunk's reserved rows below Kq, and where the quantized slots end
                const uint32_t res_mask = kBits > 0 ? chunk_mask(j) : 0u;
                const int rq = kBits > 0 ? max(0, min(kChunk, p.Kq - s0)) : kChunk;
                const uint8_t* code_s = stage + s * kStageBytes + 2 * kChunkBytes + warp * 8 * kCodeRow;
                const float2* sz_s = reinterpret_cast<const float2*>(stage + s * kStageBytes + 2 * kChunkBytes +
                                                                     kChunk * kCodeRow) + warp * 8;
                // partial dot products over this lane's 32 dimensions, even and odd dimensions apart
                constexpr int kChains = Gp >= 4 ? 1 : 2;
                float2 dot[Gp][kChains];
#pragma unroll
                for (int g = 0; g < Gp; ++g)
#pragma unroll
                    for (int h = 0; h < kChains; ++h) dot[g][h] = make_float2(0.f, 0.f);
                const uint4* krow = reinterpret_cast<const uint4*>(k_s + sl * kRowBytes);
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    const int piece = part + 4 * ((c + rot) & 3);
                    const uint4 u = krow[piece];
                    const float2 k0 = bf16x2_to_f32x2(u.x), k1 = bf16x2_to_f32x2(u.y);
                    const float2 k2 = bf16x2_to_f32x2(u.z), k3 = bf16x2_to_f32x2(u.w);
#pragma unroll
                    for (int g = 0; g < Gp; ++g) {
                        const float4* qp = reinterpret_cast<const float4*>(q_s + (g * 16 + piece) * kQPieceFloats);
                        const float4 qa = qp[0], qb = qp[1];
                        float2& d = dot[g][c % kChains];
                        d = __ffma2_rn(k0, make_float2(qa.x, qa.y), d);
                        d = __ffma2_rn(k1, make_float2(qa.z, qa.w), d);
                        d = __ffma2_rn(k2, make_float2(qb.x, qb.y), d);
                        d = __ffma2_rn(k3, make_float2(qb.z, qb.w), d);
                    }
                }
                const bool valid = sl < nr;
                float sc[Gp];
                bool raise = false;
#pragma unroll
                for (int g = 0; g < Gp; ++g) {
                    float v = dot[g][0].x + dot[g][0].y;
                    if (kChains > 1) v += dot[g][kChains - 1].x + dot[g][kChains - 1].y;
                    v += __shfl_xor_sync(0xffffffffu, v, 1);
                    v += __shfl_xor_sync(0xffffffffu, v, 2);
                    sc[g] = valid ? v : -INFINITY;
                    raise |= sc[g] > m[g] + kLazyMax;
                }
                if (__any_sync(0xffffffffu, raise)) {
                    // a score passed the running max by more than 2^8: move the max to the chunk's and rescale
#pragma unroll
                    for (int g = 0; g < Gp; ++g) {
                        float mx = sc[g];
                        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 4));
                        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 8));
                        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
                        const float m_new = fmaxf(m[g], mx);  // finite: slot 0 of the warp is valid
                        const float alpha = ex2(m[g] - m_new);  // 0 on the first chunk (m = -inf)
                        m[g] = m_new;
                        l[g] *= alpha;
                        if (kBits > 0) bias[g] *= alpha;
                        acc[g][0] = __fmul2_rn(acc[g][0], make_float2(alpha, alpha));
                        acc[g][1] = __fmul2_rn(acc[g][1], make_float2(alpha, alpha));
                    }
                }
                // weights exp2(s - m) <= 2^8 (0 for a slot past the chunk), each stored twice for the paired FMAs
                float2* pw_w = reinterpret_cast<float2*>(smem_raw + Ly.pw_off) + warp * 8 * Gp;
                float2 sz_t = make_float2(1.f, 0.f);  // a coded slot's (s, z); bf16 slots keep (1, 0)
                if (kBits > 0) {
                    const int t = warp * 8 + sl;
                    if (valid && t < rq && !((res_mask >> t) & 1u)) sz_t = sz_s[sl];
                }
#pragma unroll
                for (int g = 0; g < Gp; g += 2) {
                    const float w0 = ex2(sc[g] - m[g]);
                    const float w1 = ex2(sc[g + 1] - m[g + 1]);
                    l[g] += w0;
                    l[g + 1] += w1;
                    if (kBits > 0) {
                        bias[g] = fmaf(w0, sz_t.y, bias[g]);
                        bias[g + 1] = fmaf(w1, sz_t.y, bias[g + 1]);
                    }
                    const float u0 = kBits > 0 ? w0 * sz_t.x : w0, u1 = kBits > 0 ? w1 * sz_t.x : w1;
                    if (part == 0) *reinterpret_cast<float4*>(pw_w + sl * Gp + g) = make_float4(u0, u0, u1, u1);
                }
                __syncwarp();
                // weighted V rows: lane takes dims 4*lane .. 4*lane+3 of each valid row
                auto add_row = [&](int r, float2 v0, float2 v1) {
#pragma unroll
                    for (int g = 0; g < Gp; g += 2) {
                        const float4 w = *reinterpret_cast<const float4*>(pw_w + r * Gp + g);
                        acc[g][0] = __ffma2_rn(make_float2(w.x, w.y), v0, acc[g][0]);
                        acc[g][1] = __ffma2_rn(make_float2(w.x, w.y), v1, acc[g][1]);
                        acc[g + 1][0] = __ffma2_rn(make_float2(w.z, w.w), v0, acc[g + 1][0]);
                        acc[g + 1][1] = __ffma2_rn(make_float2(w.z, w.w), v1, acc[g + 1][1]);
                    }
                };
                const uint8_t* v_area = stage + s * kStageBytes + kChunkBytes;
                if (kBits == 0) {
#pragma unroll 2
                    for (int r = 0; r < nr; ++r) {
                        const uint2 vv = reinterpret_cast<const uint2*>(v_area + (warp * 8 + r) * kRowBytes)[lane];
                        add_row(r, bf16x2_to_f32x2(vv.x), bf16x2_to_f32x2(vv.y));
                    }
                } else {
                    // the warp's coded rows first, then its bf16 rows: two branch-free loops over row masks
                    const uint32_t rows_w = low_mask(nr);
                    uint32_t cm = ~(res_mask >> (warp * 8)) & low_mask(rq - warp * 8) & rows_w;
                    uint32_t bm = rows_w & ~cm;
                    constexpr uint32_t kLevels = (1u << (kBits > 0 ? kBits : 1)) - 1u;
                    while (cm) {  // the codes as floats; s and z are in the row's weight and the bias
                        const int r = __ffs(cm) - 1;
                        cm &= cm - 1u;
                        const uint8_t* cp = code_s + r * kCodeRow + lane * (kBits / 2);
                        uint32_t packed;
                        if (kBits == 8) packed = *reinterpret_cast<const uint32_t*>(cp);
                        else if (kBits == 4) packed = *reinterpret_cast<const uint16_t*>(cp);
                        else packed = *cp;
                        // a code c < 2^23 as a float: the bits of 2^23 + c, minus 2^23 (exact)
                        auto cf = [&](int e) {
                            return __uint_as_float(0x4B000000u | ((packed >> (e * kBits)) & kLevels)) - 8388608.f;
                        };
                        add_row(r, make_float2(cf(0), cf(1)), make_float2(cf(2), cf(3)));
                    }
                    while (bm) {  // reserved rows below rq sit compacted at the front of the V area
                        const int r = __ffs(bm) - 1;
                        bm &= bm - 1u;
                        const int t = warp * 8 + r;
                        const int vrow = t < rq ? __popc(res_mask & low_mask(t)) : t;
                        const uint2 vv = reinterpret_cast<const uint2*>(v_area + vrow * kRowBytes)[lane];
                        add_row(r, bf16x2_to_f32x2(vv.x), bf16x2_to_f32x2(vv.y));
                    }
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty[s]);
        }
    }
    __syncthreads();  // every chunk consumed and every copy landed: the stage area holds the fold areas now
    if (warp < kConsumerWarps) {
        float* fold_o = reinterpret_cast<float*>(smem_raw + Ly.fold_o);
#pragma unroll
        for (int g = 0; g < Gp; ++g) {
            float b = 0.f;  // sum p z over the warp's coded slots (each counted by its four lanes)
            if (kBits > 0) {
                b = bias[g];
#pragma unroll
                for (int o = 16; o >= 1; o >>= 1) b += __shfl_xor_sync(0xffffffffu, b, o);
                b *= 0.25f;
            }
            *reinterpret_cast<float4*>(fold_o + (warp * Gp + g) * kHeadDim + 4 * lane) =
                make_float4(acc[g][0].x + b, acc[g][0].y + b, acc[g][1].x + b, acc[g][1].y + b);
            float lsum = l[g];
#pragma unroll
            for (int o = 16; o >= 1; o >>= 1) lsum += __shfl_xor_sync(0xffffffffu, lsum, o);
            if (lane == 0) {
                wml[(warp * Gp + g) * 2] = m[g];
                wml[(warp * Gp + g) * 2 + 1] = 0.25f * lsum;  // every slot was counted by its four lanes
            }
        }
    }
    __syncthreads();
    // ---- fold the warps: CTA state (M, L, O) per query head
    {
        const float* fold_o = reinterpret_cast<const float*>(smem_raw + Ly.fold_o);
        float* res_o = reinterpret_cast<float*>(smem_raw + Ly.res_o);
        float* res_ml = reinterpret_cast<float*>(smem_raw + Ly.res_ml);
        for (int i = tid; i < G * kHeadDim; i += kThreads) {
            const int g = i / kHeadDim;
            const int d = i - g * kHeadDim;
            float M = -INFINITY;
#pragma unroll
            for (int w = 0; w < kConsumerWarps; ++w) M = fmaxf(M, wml[(w * Gp + g) * 2]);
            float L = 0.f, O = 0.f;
#pragma unroll
            for (int w = 0; w < kConsumerWarps; ++w) {
                const float f = ex2(wml[(w * Gp + g) * 2] - M);  // a warp with no slot: m = -inf, f = 0
                L = fmaf(wml[(w * Gp + g) * 2 + 1], f, L);
                O = fmaf(fold_o[(w * Gp + g) * kHeadDim + d], f, O);
            }
            res_o[g * kHeadDim + d] = O;
            if (d == 0) {
                res_ml[g * 2] = M;
                res_ml[g * 2 + 1] = L;
            }
        }
    }
    cluster_sync();  // every CTA's state is in its shared memory
    {
        // ---- fold the cluster: CTA r writes outputs [r * per, (r + 1) * per) of the unit's G x d
        const float* res_o = reinterpret_cast<const float*>(smem_raw + Ly.res_o);
        const float* res_ml = reinterpret_cast<const float*>(smem_raw + Ly.res_ml);
        const int total = G * kHeadDim;
        const int per = (total + C - 1) / C;
        const int end = min(total, (rank + 1) * per);
        for (int i = rank * per + tid; i < end; i += kThreads) {
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

template <int Gp, int kBits>
cudaError_t launch_gp(const DecodeParams& p, size_t smem_bytes, cudaStream_t s) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(p.cluster), static_cast<unsigned>(p.units));
    cfg.blockDim = dim3(kThreads);
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
    return cudaLaunchKernelEx(&cfg, decode_simt_kernel<Gp, kBits>, p);
}

}  // namespace simt
