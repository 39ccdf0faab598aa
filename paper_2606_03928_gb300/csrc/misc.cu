// Bandwidth kernels of the eviction step: window/cache append, value
// magnitude, selection (reservation + stochastic top-k) and the stable
// in-place compaction of the kept rows.
#include <cfloat>
#include <cuda_bf16.h>

#include "kernels.cuh"
#include "ptx.cuh"
#include "quant.cuh"

namespace vase {

namespace {

// ------------------------------------------------------------------ append
// One decode step appends one (k, v) pair per KV head and one query per query
// head (Sec. 2, periodic eviction; the last W queries are cached for Eq. (2)).
// The value magnitude of a token (Range, L2 or Var of its value row, Eq. (5) and App. A)
// never changes once it is cached, so it is taken here, where the row is written, and
// kept per slot beside the positions; the eviction step then never reads V to score.
__device__ __forceinline__ void bf16x8_to_f32(const uint4 u, float (&f)[8]) {
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        f[2 * i] = __uint_as_float(w[i] << 16);
        f[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
    }
}

// Value magnitude of a 128-element row spread over the 16 lanes of a half warp (8 elements
// each); every lane of the warp must call it.  The result is valid in all 16 lanes.
__device__ __forceinline__ float half_warp_value_magnitude(const uint4 u, int kind) {
    float f[8];
    bf16x8_to_f32(u, f);
    if (kind == 0) {
        float mx = f[0], mn = f[0];
#pragma unroll
        for (int i = 1; i < 8; ++i) {
            mx = fmaxf(mx, f[i]);
            mn = fminf(mn, f[i]);
        }
#pragma unroll
        for (int o = 8; o >= 1; o >>= 1) {
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
            mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, o));
        }
        return mx - mn;
    }
    if (kind == 1) {
        float ss = 0.f;
#pragma unroll
        for (int i = 0; i < 8; ++i) ss = fmaf(f[i], f[i], ss);
#pragma unroll
        for (int o = 8; o >= 1; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
        return sqrtf(ss);
    }
    float sm = 0.f;
#pragma unroll
    for (int i = 0; i < 8; ++i) sm += f[i];
#pragma unroll
    for (int o = 8; o >= 1; o >>= 1) sm += __shfl_xor_sync(0xffffffffu, sm, o);
    const float mu = sm * (1.0f / kHeadDim);
    float ss = 0.f;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const float dl = f[i] - mu;
        ss = fmaf(dl, dl, ss);
    }
#pragma unroll
    for (int o = 8; o >= 1; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
    return ss * (1.0f / kHeadDim);
}

// One block per (sequence, layer slot, chunk of kAppendSteps decode steps).  A half warp moves one 256-byte
// row: the Hkv key rows and Hkv value rows of every step, and the Hq query rows of the steps that stay in
// the window ring (the last W); value rows also get their magnitude.
constexpr int kAppendSteps = 4;

__global__ void __launch_bounds__(256) append_kernel(const AppendParams p) {
    const int z = blockIdx.y;  // layer slot
    const int layer = p.layer[z];
    const int s = static_cast<int>(blockIdx.x) % p.b;  // sequence
    const int t0 = (static_cast<int>(blockIdx.x) / p.b) * p.steps_per_block;
    const int t1 = min(p.n, t0 + p.steps_per_block);
    const int Hq = p.Hq, Hkv = p.Hkv, N = p.N, W = p.W;
    const int fill = p.fill[z];
    const int64_t units = static_cast<int64_t>(p.b) * Hkv;
    const int64_t unit0 = static_cast<int64_t>(layer) * units + static_cast<int64_t>(s) * Hkv;  // unit of head 0
    uint4* const kc = p.kc + unit0 * N * kVecPerRow;
    uint4* const vc = p.vc ? p.vc + unit0 * N * kVecPerRow : nullptr;  // null: the values go to the compressed store
    int32_t* const pos = p.pos + unit0 * N;
    float* const vmag = p.vmag + unit0 * N;
    uint4* const qwin = p.qwin + (static_cast<int64_t>(layer) * p.b + s) * Hq * W * kVecPerRow;
    const uint4* const qin = p.q + static_cast<int64_t>(z) * p.q_stride;
    const uint4* const kin = p.k + static_cast<int64_t>(z) * p.kv_stride;
    const uint4* const vin = p.v + static_cast<int64_t>(z) * p.kv_stride;
    for (int t = t0; t < t1; ++t) {
        const bool q_lives = t >= p.n - W;
        const int per = (2 * Hkv + (q_lives ? Hq : 0)) * 16;  // 16-byte vectors of this step
        const int64_t row_in = static_cast<int64_t>(t) * p.b + s;
        const int slot = q_lives ? (p.q_ring[z] + t) % W : 0;
        // the trip count is the same for every thread of the block, so the half-warp shuffles see full warps
        for (int e0 = 0; e0 < per; e0 += blockDim.x) {
            const int e = e0 + static_cast<int>(threadIdx.x);
            const int r = e >> 4;
            const int seg = e & 15;
            uint4 val = make_uint4(0, 0, 0, 0);
            bool is_v = false;
            if (e < per) {
                if (r < Hkv) {
                    kc[(static_cast<int64_t>(r) * N + fill + t) * kVecPerRow + seg] =
                        kin[(row_in * Hkv + r) * kVecPerRow + seg];
                } else if (r < 2 * Hkv) {
                    is_v = true;
                    val = vin[(row_in * Hkv + (r - Hkv)) * kVecPerRow + seg];
                    if (vc) vc[(static_cast<int64_t>(r - Hkv) * N + fill + t) * kVecPerRow + seg] = val;
                } else {
                    const int hq = r - 2 * Hkv;
                    qwin[(static_cast<int64_t>(hq) * W + slot) * kVecPerRow + seg] =
                        qin[(row_in * Hq + hq) * kVecPerRow + seg];
                }
            }
            if (__any_sync(0xffffffffu, is_v)) {
                const float mag = half_warp_value_magnitude(val, p.kind);
                if (is_v && seg == 0) vmag[static_cast<int64_t>(r - Hkv) * N + fill + t] = mag;
            }
        }
        for (int h = threadIdx.x; h < Hkv; h += blockDim.x)
            pos[static_cast<int64_t>(h) * N + fill + t] = static_cast<int32_t>(p.next_pos[z] + t);
    }
}

// ------------------------------------------------------------------ value magnitude refresh
// Recomputes the per-slot value magnitudes of slots 0..rows-1 of every unit of one layer
// from the V cache (for callers that write cache rows directly).  A half warp per row.
__global__ void value_score_kernel(const ValueParams p) {
    const int warp = threadIdx.x >> 5;
    const int hsel = (threadIdx.x >> 4) & 1;
    const int l = threadIdx.x & 15;
    const int halves = blockDim.x >> 4;
    const int64_t rows = static_cast<int64_t>(p.units) * p.rows;
    for (int64_t r0 = static_cast<int64_t>(blockIdx.x) * halves + 2 * warp; r0 < rows;
         r0 += static_cast<int64_t>(gridDim.x) * halves) {
        const int64_t r = r0 + hsel;
        const bool valid = r < rows;
        const int unit = valid ? static_cast<int>(r / p.rows) : 0;
        const int slot = valid ? static_cast<int>(r - static_cast<int64_t>(unit) * p.rows) : 0;
        const int64_t row = static_cast<int64_t>(unit) * p.N + slot;
        const float out =
            half_warp_value_magnitude(valid ? __ldg(&p.vc[row * kVecPerRow + l]) : make_uint4(0, 0, 0, 0), p.kind);
        if (valid && l == 0) p.out[row] = out;
    }
}

// ------------------------------------------------------------------ selection
constexpr int kSelThreads = 256;
constexpr int kSelWarps = kSelThreads / 32;
constexpr uint8_t kFlagValue = 1;
constexpr uint8_t kFlagSampled = 2;

constexpr int kSelBins = 256;

struct SelShared {
    uint32_t hist[kSelBins];
    int warp_tot[32];  // one per warp of the block (up to 1024 threads)
    uint32_t bcast[4];
    int first_evicted;  // lowest evicted slot (slots below it keep their place)
    uint32_t small_x[64];  // radix_top_k: the keys of a boundary digit with at most 64 members ...
    int small_i[64];       // ... and their slots
    int n_small;
};

// Exclusive prefix over threads of `v` in thread order; returns the offset and
// writes the block total to *total.  Every thread of the kT-thread block must call it.
template <int kT = kSelThreads>
__device__ __forceinline__ int block_exclusive_scan(int v, SelShared& sh, int* total) {
    constexpr int kW = kT / 32;
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) sh.warp_tot[warp] = x;
    __syncthreads();
    if (warp == 0) {
        int w = lane < kW ? sh.warp_tot[lane] : 0;
        int inc = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, inc, o);
            if (lane >= o) inc += y;
        }
        if (lane < kW) sh.warp_tot[lane] = inc - w;  // exclusive warp offsets
        if (lane == kW - 1) sh.bcast[3] = static_cast<uint32_t>(inc);
    }
    __syncthreads();
    const int off = sh.warp_tot[warp] + x - v;
    *total = static_cast<int>(sh.bcast[3]);
    __syncthreads();
    return off;
}

// Marks with `flag` the k largest values of ord[0..n) (ties to the lower
// index), by an MSB-first radix select on four 8-bit digits (lanes with the
// same digit are merged with __match_any_sync before the shared-memory atomic)
// followed by a slot-ordered rank of the elements equal to the threshold.
// Each thread of the kT-thread block owns the contiguous slots [seg_lo, seg_hi).
template <int kT = kSelThreads>
__device__ void radix_top_k(const uint32_t* ord, int n, int k, uint8_t* flags, uint8_t flag, int seg_lo,
                            int seg_hi, SelShared& sh) {
    static_assert(kT >= kSelBins, "a thread per histogram bin");
    if (k <= 0) return;
    const int tid = threadIdx.x;
    const int lane = tid & 31;
    uint32_t prefix = 0, mask = 0;
    int remain = k;
    for (int shift = 24; shift >= 0; shift -= 8) {
        if (tid < kSelBins) sh.hist[tid] = 0;
        __syncthreads();
        const int n_round = (n + 31) & ~31;
        for (int i = tid; i < n_round; i += kT) {
            const uint32_t x = i < n ? ord[i] : 0u;
            const bool in = i < n && (x & mask) == prefix;
            const uint32_t bin = in ? ((x >> shift) & 0xFFu) : 0xFFFFFFFFu;
            const uint32_t peers = __match_any_sync(0xffffffffu, bin);
            if (in && lane == __ffs(peers) - 1) atomicAdd(&sh.hist[bin], static_cast<uint32_t>(__popc(peers)));
        }
        __syncthreads();
        if (tid < 32) {
            // lane owns bins 8*lane .. 8*lane+7; suffix sums find the digit holding the remain-th largest
            uint32_t c[8];
            uint32_t tot = 0;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                c[j] = sh.hist[8 * lane + ((j + lane) & 7)];  // bank-rotated read
                tot += c[j];
            }
            uint32_t suf = tot;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const uint32_t y = __shfl_down_sync(0xffffffffu, suf, o);
                if (lane + o < 32) suf += y;
            }
            uint32_t above = suf - tot;
            if (above < static_cast<uint32_t>(remain) && suf >= static_cast<uint32_t>(remain)) {
#pragma unroll
                for (int j = 7; j >= 0; --j) {
                    const uint32_t cj = sh.hist[8 * lane + j];
                    if (above < static_cast<uint32_t>(remain) && above + cj >= static_cast<uint32_t>(remain)) {
                        sh.bcast[0] = static_cast<uint32_t>(8 * lane + j);
                        sh.bcast[1] = above;
                        sh.bcast[2] = cj;
                    }
                    above += cj;
                }
            }
            if (lane == 0) sh.n_small = 0;
        }
        __syncthreads();
        remain -= static_cast<int>(sh.bcast[1]);
        prefix |= sh.bcast[0] << shift;
        mask |= 0xFFu << shift;
        if (shift > 0 && sh.bcast[2] <= 64u) {
            // At most 64 keys share the digits so far: every key above them is taken, and they are ranked among
            // themselves by two warps (larger key, or equal key at a lower slot) instead of the remaining passes.
            for (int i = tid; i < n; i += kT) {
                const uint32_t x = ord[i];
                if ((x & mask) == prefix) {
                    const int j = atomicAdd(&sh.n_small, 1);
                    sh.small_x[j] = x;
                    sh.small_i[j] = i;
                } else if ((x & mask) > prefix) {
                    flags[i] |= flag;
                }
            }
            __syncthreads();
            const int ns = sh.n_small;
            if (tid < ns) {
                const uint32_t x = sh.small_x[tid];
                const int xi = sh.small_i[tid];
                int rank = 0;
                for (int j = 0; j < ns; ++j) {
                    const uint32_t y = sh.small_x[j];
                    rank += (y > x) || (y == x && sh.small_i[j] < xi);
                }
                if (rank < remain) flags[xi] |= flag;
            }
            __syncthreads();
            return;
        }
    }
    const uint32_t thr = prefix;
    int eq = 0;
    for (int i = seg_lo; i < seg_hi; ++i) eq += ord[i] == thr;
    int total;
    int rank = block_exclusive_scan<kT>(eq, sh, &total);
    for (int i = seg_lo; i < seg_hi; ++i) {
        const uint32_t x = ord[i];
        bool take = x > thr;
        if (x == thr) {
            take = rank < remain;
            ++rank;
        }
        if (take) flags[i] |= flag;
    }
    __syncthreads();
}

// The same selection as radix_top_k for n candidates, by rank, by a team of nt >= n threads (t = 0 .. nt - 1,
// whole warps): slot i is taken when fewer than k slots outrank it (a larger key, or an equal key at a lower slot).
// Each candidate's count is split over P = 1, 2 or 4 neighbouring threads (as many as nt / n allows): part p
// compares against the groups of four keys g with g % P == p, read as broadcasts (the parts of a warp read
// neighbouring 16-byte groups, so different banks), and the parts' counts are summed by shuffles.  Groups wholly
// below i count keys >= x, groups wholly above it keys > x (one comparison per key); only i's own group tests
// the slot order.  No histogram passes and no barrier (rank_top_k: the whole block, then a barrier).
__device__ __forceinline__ void rank_top_k_team(const uint32_t* ord, int n, int k, uint8_t* flags, uint8_t flag,
                                                int t, int nt) {
    const int P = 4 * n <= nt ? 4 : (2 * n <= nt ? 2 : 1);
    const int i = t / P, part = t - i * P;
    int rank = 0;
    uint32_t x = 0;
    const bool live = k > 0 && i < n;
    if (live) {
        x = ord[i];
        const uint4* ord4 = reinterpret_cast<const uint4*>(ord);
        const int g4 = n >> 2, gi = i >> 2;  // groups of four keys; gi holds candidate i itself
        int g = part;
        for (; g < gi && g < g4; g += P) {  // every slot below i: an equal key outranks it too
            const uint4 y = ord4[g];
            rank += (y.x >= x) + (y.y >= x) + (y.z >= x) + (y.w >= x);
        }
        if (g == gi && g < g4) {  // the group of i: ties count for the slots below it only
            const uint4 y = ord4[g];
            const int j = 4 * g;
            rank += (y.x > x) + (y.y > x) + (y.z > x) + (y.w > x);
            rank += (y.x == x && j < i) + (y.y == x && j + 1 < i) + (y.z == x && j + 2 < i);
            g += P;
        }
        for (; g < g4; g += P) {  // every slot above i: only a larger key outranks it
            const uint4 y = ord4[g];
            rank += (y.x > x) + (y.y > x) + (y.z > x) + (y.w > x);
        }
        if (part == 0)
            for (int j = 4 * g4; j < n; ++j) rank += (ord[j] > x) + (ord[j] == x && j < i);
    }
    // the parts of a candidate are P neighbouring lanes of one warp (P divides 32); all lanes take part
    for (int o = 1; o < P; o <<= 1) rank += __shfl_xor_sync(0xffffffffu, rank, o);
    if (live && part == 0 && rank < k) flags[i] |= flag;
}

template <int kT>
__device__ void rank_top_k(const uint32_t* ord, int n, int k, uint8_t* flags, uint8_t flag) {
    rank_top_k_team(ord, n, k, flags, flag, threadIdx.x, kT);
    __syncthreads();
}

template <int kT>
__device__ __forceinline__ void top_k_select(const uint32_t* ord, int n, int k, uint8_t* flags, uint8_t flag,
                                             int seg_lo, int seg_hi, SelShared& sh) {
    if (n <= kT) rank_top_k<kT>(ord, n, k, flags, flag);
    else radix_top_k<kT>(ord, n, k, flags, flag, seg_lo, seg_hi, sh);
}

// One CTA per unit.  AttnV (Sec. 3.2): R_B = slots >= K; R_V = N_v largest
// value magnitudes among slots < K; the m = K - N_v - B remaining slots are
// the m largest keys pooled_i / E_i over C = [K] \ R_V, E_i = -ln u_i, which is
// weighted sampling without replacement proportional to the pooled score
// (exponential race); with stochastic = 0 the key is the pooled score itself
// (Sec. 4.1).  DKV: the K - B largest leverage products.  Writes the ascending
// list of kept slots.
// Asynchronous copy of `count` 32-bit words from global to shared memory by the whole block (or by the team of
// threads t = 0 .. nt - 1), in 16-byte pieces when both ends allow it; completion by cp_async_wait_all().
__device__ __forceinline__ void cp_async_words(void* smem_dst, const void* gsrc, int count, int t = -1, int nt = 0) {
    if (t < 0) {  // the whole block
        t = threadIdx.x;
        nt = blockDim.x;
    }
    const bool vec = ((reinterpret_cast<uintptr_t>(gsrc) | smem_u32(smem_dst)) & 15u) == 0;
    if (vec) {
        const int n4 = count >> 2;
        for (int i = t; i < n4; i += nt)
            asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(smem_dst) + 16u * i),
                         "l"(static_cast<const uint8_t*>(gsrc) + 16 * i)
                         : "memory");
        for (int i = 4 * n4 + t; i < count; i += nt)
            asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_u32(smem_dst) + 4u * i),
                         "l"(static_cast<const uint8_t*>(gsrc) + 4 * i)
                         : "memory");
    } else {
        for (int i = t; i < count; i += nt)
            asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_u32(smem_dst) + 4u * i),
                         "l"(static_cast<const uint8_t*>(gsrc) + 4 * i)
                         : "memory");
    }
}

__device__ __forceinline__ void cp_async_wait_all() {
    asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
}

// Gather of the kept rows: one warp per tensor (K, V), a ring of kGatherStages chunks of kGatherRows
// destination rows each.
constexpr int kGatherRows = 24;
constexpr int kGatherStages = 3;       // ring depth when the selection's buffers leave no more room
constexpr int kGatherMaxStages = 16;   // ring depth where they do (units of many slots)
constexpr uint32_t kGatherChunkBytes = kGatherRows * kRowBytes;
constexpr uint32_t kGatherRingBytes = kGatherStages * kGatherChunkBytes;  // per tensor, at the base depth

// Shared-memory layout of the selection: window scores (one array per part) or leverage products, then
// (staged) value magnitudes and positions, then the orderable keys and the flags.  The gather rings
// overlay all of these once the selection is done; the kept list and the rings' barriers follow.
struct SelLayout {
    uint32_t a_off, vm_off, pos_off, ord_off, flag_off, src_off, bar_off, total;
    int gather_stages;  // ring depth per tensor: as many chunks as the selection's buffers hold, 3 at least
};

__host__ __device__ inline SelLayout sel_layout(int N, int K, int n_parts, bool staged) {
    SelLayout L;
    uint32_t o = 0;
    L.a_off = o;
    o += 4u * (staged ? n_parts : 1) * N;
    L.vm_off = o;
    if (staged) o += 4u * N;
    L.pos_off = o;
    if (staged) o += 4u * N;
    o = (o + 15u) & ~15u;  // the keys are read four at a time (rank_top_k)
    L.ord_off = o;
    o += 4u * K;
    L.flag_off = o;
    o += N;
    if (o < 2 * kGatherRingBytes) o = 2 * kGatherRingBytes;
    L.gather_stages = static_cast<int>(o / (2 * kGatherChunkBytes));
    if (L.gather_stages > kGatherMaxStages) L.gather_stages = kGatherMaxStages;
    o = (o + 15u) & ~15u;
    L.src_off = o;
    o += 4u * K;
    o = (o + 7u) & ~7u;
    L.bar_off = o;
    o += 8u * 2 * kGatherMaxStages;
    L.total = o;
    return L;
}

__device__ __forceinline__ void bulk_load(void* smem_dst, const void* gsrc, uint32_t bytes, uint64_t* bar) {
    asm volatile("cp.async.bulk.shared::cta.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                     smem_u32(smem_dst)),
                 "l"(gsrc), "r"(bytes), "r"(smem_u32(bar))
                 : "memory");
}
__device__ __forceinline__ void bulk_store(void* gdst, const void* smem_src, uint32_t bytes) {
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(gdst), "r"(smem_u32(smem_src)),
                 "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read0() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read1() { asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// Stable in-place gather of one tensor's kept rows (K or V of one unit) by one warp: new row j takes old
// row src[j] >= j for j >= j_first (the rows below the lowest evicted slot stay).  Destination chunks of
// kGatherRows rows go in ascending order: the kept rows of a chunk form runs of consecutive source rows,
// each fetched by one bulk copy into a ring stage, and the chunk goes back with one bulk store.  The
// sources of a chunk lie at or above its first row and its store ends below the next chunk's first row,
// so loads issued ahead never read a row that an earlier chunk's store overwrites; a chunk is stored only
// after its own loads have landed.
__device__ void gather_rows(uint8_t* base, const int32_t* src, int j_first, int K, uint8_t* ring, uint64_t* full,
                            int stages, uint32_t* err) {
    const int lane = threadIdx.x & 31;
    if (lane == 0) {
        for (int s = 0; s < stages; ++s) mbar_init(&full[s], 1);
        fence_mbar_init();
    }
    __syncwarp();
    const int n_chunks = (K - j_first + kGatherRows - 1) / kGatherRows;
    auto load = [&](int c) {
        const int stage = c % stages;
        uint8_t* dst = ring + stage * kGatherChunkBytes;
        const int j0 = j_first + c * kGatherRows;
        const int rows = min(kGatherRows, K - j0);
        if (lane == 0) mbar_arrive_expect_tx(&full[stage], static_cast<uint32_t>(rows) * kRowBytes);
        __syncwarp();
        // a run of consecutive sources starts where src[j] != src[j-1] + 1 (or at the chunk start)
        const bool in = lane < rows;
        const int sv = in ? src[j0 + lane] : 0;
        const bool st = in && (lane == 0 || src[j0 + lane - 1] + 1 != sv);
        const uint32_t starts = __ballot_sync(0xffffffffu, st);
        if (st) {
            const uint32_t later = lane < 31 ? (starts >> (lane + 1)) << (lane + 1) : 0u;
            const int next = later ? __ffs(later) - 1 : rows;
            bulk_load(dst + lane * kRowBytes, base + static_cast<int64_t>(sv) * kRowBytes,
                      static_cast<uint32_t>(next - lane) * kRowBytes, &full[stage]);
        }
    };
    // Loads run `ahead` chunks in front of the stores.  With the base depth the stage reloaded next was read by
    // the store just issued, so every store must have read its bytes first (wait_group.read 0); with a deeper
    // ring the reloaded stage's last store is at least two back, so the newest store may still be reading
    // (wait_group.read 1).
    const int ahead = stages > kGatherStages ? stages - 2 : stages - 1;
    bool ok = true;
    for (int c = 0; c < ahead && c < n_chunks; ++c) load(c);
    for (int c = 0; c < n_chunks; ++c) {
        const int nxt = c + ahead;
        if (nxt < n_chunks) {
            if (lane == 0) {
                if (stages > kGatherStages) bulk_wait_read1();
                else bulk_wait_read0();
            }
            __syncwarp();
            load(nxt);
        }
        const int stage = c % stages;
        if (ok) ok = mbar_wait(&full[stage], (c / stages) & 1, err, kErrCompactFull);
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        if (lane == 0) {
            const int j0 = j_first + c * kGatherRows;
            const int rows = min(kGatherRows, K - j0);
            bulk_store(base + static_cast<int64_t>(j0) * kRowBytes, ring + stage * kGatherChunkBytes,
                       static_cast<uint32_t>(rows) * kRowBytes);
            bulk_commit();
        }
        __syncwarp();
    }
    if (lane == 0) bulk_wait_all();
    __syncwarp();
}

// kT threads per CTA: 256 where four CTAs share an SM; 512 or 1024 where the unit's arrays leave room for two
// or one, so that the selection phase, which no other CTA's gather hides there, runs on as many warps.
//
// The staged value magnitudes and positions of one unit, requested into the selection's shared-memory layout
// (completion by cp_async_wait_all, which select_unit runs): the fused small-unit eviction issues them before
// its window score, so that their memory latency passes under the score.
__device__ __forceinline__ void select_stage_rows(const SelectParams& p, int unit, int z, uint8_t* smem_raw,
                                                  int t = -1, int nt = 0) {
    const int N = p.N;
    const SelLayout Ly = sel_layout(N, p.K, p.n_parts, true);
    const int layer = p.batch.layer[z];
    const int64_t base = static_cast<int64_t>(layer) * p.units * N + static_cast<int64_t>(unit) * N;
    cp_async_words(smem_raw + Ly.vm_off, p.vmag + base, N, t, nt);
    cp_async_words(smem_raw + Ly.pos_off, p.pos + base, N, t, nt);
}

// The reservation key of slot i (orderable; the N_v largest are R_V): its value magnitude vm (Eq. (5), Sec. 3.1),
// or with random reservation a Philox uniform keyed by the slot's position, the round and the unit.
__device__ __forceinline__ uint32_t reserve_ord(const SelectParams& p, int layer, int rnd, int unit, float vm,
                                                int32_t pi) {
    if (p.reserve_random) {  // the N_v largest reservation uniforms: a uniformly random N_v-subset
        const uint32_t c2_res = static_cast<uint32_t>(layer) | (kTagReserve << 24);
        const Philox4 w = philox4x32_10(
            Philox4{static_cast<uint32_t>(pi), static_cast<uint32_t>(rnd), c2_res, static_cast<uint32_t>(unit)},
            p.seed_lo, p.seed_hi);
        return (w.x >> 9) + 1u;
    }
    return __float_as_uint(vm) + 1u;
}

// R_V of one AttnV unit (the N_v largest reservation keys among the slots below K, ties to the lower slot) by a
// team of threads t = 0 .. nt - 1 (whole warps, K <= nt, using named barrier bar_id) while the rest of the block
// does other work, on inputs the team itself staged (select_stage_rows with the same team): the flags cleared,
// the keys, then the rank count.  select_unit(..., rv_ready = true) then skips these steps; the caller orders
// the two with a block barrier.
__device__ void select_reserve_team(const SelectParams& p, int unit, int z, uint8_t* smem_raw, int t, int nt,
                                    uint32_t bar_id) {
    const int N = p.N, K = p.K;
    const SelLayout Ly = sel_layout(N, K, p.n_parts, true);
    const float* vm_s = reinterpret_cast<const float*>(smem_raw + Ly.vm_off);
    const int32_t* pos_s = reinterpret_cast<const int32_t*>(smem_raw + Ly.pos_off);
    uint32_t* ord = reinterpret_cast<uint32_t*>(smem_raw + Ly.ord_off);
    uint8_t* flags = smem_raw + Ly.flag_off;
    const int layer = p.batch.layer[z], rnd = p.batch.rnd[z];
    float* const vscore_dbg =
        p.vscore_dbg ? p.vscore_dbg + (static_cast<int64_t>(z) * p.units + unit) * N : nullptr;
    cp_async_wait_all();
    named_bar(bar_id, static_cast<uint32_t>(nt));
    for (int i = t; i < N; i += nt) flags[i] = 0;
    for (int i = t; i < K; i += nt) {
        const float vm = vm_s[i];
        ord[i] = reserve_ord(p, layer, rnd, unit, vm, p.reserve_random ? pos_s[i] : 0);
        if (vscore_dbg) vscore_dbg[i] = vm;
    }
    named_bar(bar_id, static_cast<uint32_t>(nt));
    rank_top_k_team(ord, K, p.n_v, flags, kFlagValue, t, nt);
}

// The body is select_unit, which the fused small-unit eviction (evict_small_kernel) runs too, on window scores it
// has already written to shared memory (a_ready: the staging skips them; one part).
template <int kT>
__device__ __forceinline__ void select_unit(const SelectParams& p, int unit, int z, uint8_t* smem_raw, SelShared& sh,
                                            bool a_ready, uint4* gbuf = nullptr, int gbuf_rows = 0,
                                            bool rv_ready = false) {
    const int N = p.N, K = p.K;
    const bool staged = p.staged != 0;
    const SelLayout Ly = sel_layout(N, K, p.n_parts, staged);
    float* a_s = reinterpret_cast<float*>(smem_raw + Ly.a_off);         // [N] window score (AttnV)
    uint32_t* ord = reinterpret_cast<uint32_t*>(smem_raw + Ly.ord_off);  // [K] orderable keys
    uint8_t* flags = smem_raw + Ly.flag_off;                            // [N]
    const int layer = p.batch.layer[z];
    const int rnd = p.batch.rnd[z];
    const int tid = threadIdx.x;
    const int64_t base = static_cast<int64_t>(unit) * N;                     // within one layer / slot
    const int64_t zs = static_cast<int64_t>(z) * p.units * N;               // slot offset of [units][N] arrays
    const float* const attn = p.attn + zs * p.n_parts;
    const float* const dkv = p.dkv + zs;
    int32_t* const pos = p.pos + static_cast<int64_t>(layer) * p.units * N;
    float* const vmag = p.vmag + static_cast<int64_t>(layer) * p.units * N;
    float* const vscore_dbg = p.vscore_dbg ? p.vscore_dbg + zs : nullptr;
    int32_t* const src_out = p.src + static_cast<int64_t>(z) * p.units * K;
    uint8_t* const resv_out = p.resv ? p.resv + static_cast<int64_t>(z) * p.units * store_resv_stride(K) : nullptr;
    float* const pooled_dbg = p.pooled_dbg ? p.pooled_dbg + zs : nullptr;
    float* const key_dbg = p.key_dbg ? p.key_dbg + zs : nullptr;
    uint8_t* const keep_dbg = p.keep_dbg ? p.keep_dbg + zs : nullptr;
    const int seg = (N + kT - 1) / kT;
    const int seg_lo = min(N, tid * seg);
    const int seg_hi = min(N, seg_lo + seg);
    const int kseg_lo = min(K, seg_lo);
    const int kseg_hi = min(K, seg_hi);

    // The unit's inputs: with `staged`, every array is requested at once (one memory latency for all),
    // and the positions and value magnitudes are compacted from the staged copies at the end.  With a_ready the
    // caller has written the window scores and requested the value magnitudes and positions itself
    // (select_stage_rows) before its own work.
    float* vm_s = staged ? reinterpret_cast<float*>(smem_raw + Ly.vm_off) : nullptr;
    int32_t* pos_s = staged ? reinterpret_cast<int32_t*>(smem_raw + Ly.pos_off) : nullptr;
    if (staged && !a_ready) {
        if (p.variant == 0) {
            for (int part = 0; part < p.n_parts; ++part)
                cp_async_words(a_s + part * N, attn + (static_cast<int64_t>(part) * p.units + unit) * N, N);
        } else {
            cp_async_words(a_s, dkv + base, K);
        }
        cp_async_words(vm_s, vmag + base, N);
        cp_async_words(pos_s, pos + base, N);
    } else if (!staged) {
        // unstaged: the first score part into a_s, the value magnitudes (as raw words) into ord and the candidates'
        // positions into the kept list's region (free until the kept list), all requested at once; ord turns into
        // the reservation keys in place below
        if (p.variant == 0 && !a_ready) cp_async_words(a_s, attn + base, N);
        if (p.variant == 0 && !rv_ready) cp_async_words(ord, vmag + base, K);
        if (p.variant == 0 && (p.stochastic || p.reserve_random)) cp_async_words(smem_raw + Ly.src_off, pos + base, K);
    }
    const int32_t* const pos_k = staged ? pos_s : reinterpret_cast<const int32_t*>(smem_raw + Ly.src_off);
    if (!rv_ready)
        for (int i = tid; i < N; i += kT) flags[i] = 0;
    if (tid == 0) sh.first_evicted = K;
    cp_async_wait_all();
    __syncthreads();
    if (p.variant == 0) {
        if (staged) {
            if (p.n_parts > 1) {
                for (int i = tid; i < N; i += kT) {
                    float a = a_s[i];
                    for (int part = 1; part < p.n_parts; ++part)
                        a = p.gqa_max ? fmaxf(a, a_s[part * N + i]) : a + a_s[part * N + i];
                    a_s[i] = a;
                }
            }
        } else if (!a_ready && p.n_parts > 1) {
            for (int i = tid; i < N; i += kT) {
                float b[3];  // the other parts (at most four in all), loaded before any is used
#pragma unroll
                for (int part = 1; part < 4; ++part)
                    b[part - 1] = part < p.n_parts ? attn[(static_cast<int64_t>(part) * p.units + unit) * N + i] : 0.f;
                float a = a_s[i];
#pragma unroll
                for (int part = 1; part < 4; ++part)
                    if (part < p.n_parts) a = p.gqa_max ? fmaxf(a, b[part - 1]) : a + b[part - 1];
                a_s[i] = a;
            }
        }
        if (p.n_parts > 1 && pooled_dbg) {
            __syncthreads();
            for (int i = tid; i < N; i += kT) const_cast<float*>(attn)[base + i] = a_s[i];
        }
        if (!rv_ready) {  // (otherwise select_reserve_team has set the R_V flags)
            for (int i = tid; i < K; i += kT) {
                const float vm = staged ? vm_s[i] : __uint_as_float(ord[i]);
                const int32_t pi = p.reserve_random ? pos_k[i] : 0;
                ord[i] = reserve_ord(p, layer, rnd, unit, vm, pi);
                if (vscore_dbg) vscore_dbg[base + i] = vm;
            }
            __syncthreads();
            top_k_select<kT>(ord, K, p.n_v, flags, kFlagValue, kseg_lo, kseg_hi, sh);
        }
        // keys over the candidates C
        const int h = p.pool / 2;
        const float inv_pool = 1.0f / static_cast<float>(p.pool);
        const uint32_t c2 = static_cast<uint32_t>(layer) | (kTagSelect << 24);
        for (int i = tid; i < N; i += kT) {
            float sum = 0.f;
            const int lo = max(0, i - h), hi = min(N - 1, i + h);
            for (int j = lo; j <= hi; ++j) sum += a_s[j];
            const float pooled = sum * inv_pool;
            if (pooled_dbg) pooled_dbg[base + i] = pooled;
            if (i >= K) continue;
            float key = -1.f;
            if (flags[i] & kFlagValue) {
                ord[i] = 0u;
            } else {
                key = pooled;
                if (p.stochastic) {
                    const int32_t pi = pos_k[i];
                    const Philox4 w = philox4x32_10(
                        Philox4{static_cast<uint32_t>(pi), static_cast<uint32_t>(rnd), c2,
                                static_cast<uint32_t>(unit)},
                        p.seed_lo, p.seed_hi);
                    key = pooled / (-logf(open_uniform(w.x)));
                }
                ord[i] = __float_as_uint(key) + 1u;
            }
            if (key_dbg) key_dbg[base + i] = key;
        }
        __syncthreads();
        top_k_select<kT>(ord, K, p.m, flags, kFlagSampled, kseg_lo, kseg_hi, sh);
    } else {
        for (int i = tid; i < K; i += kT) {
            const float s = staged ? a_s[i] : dkv[base + i];
            ord[i] = __float_as_uint(s) + 1u;
            if (key_dbg) key_dbg[base + i] = s;
        }
        __syncthreads();
        top_k_select<kT>(ord, K, p.m, flags, kFlagSampled, kseg_lo, kseg_hi, sh);
    }
    // positions move with the kept rows (unstaged: copy the old ones into shared memory, a_s is free now)
    if (!staged) {
        pos_s = reinterpret_cast<int32_t*>(a_s);
        __syncthreads();  // every read of the scores in a_s is done
        cp_async_words(pos_s, pos + base, N);
        cp_async_wait_all();  // (block_exclusive_scan below is the barrier)
    }
    // keep = R_B u R_V u sampled; ascending list of kept slots (also kept in shared memory for the gather)
    int32_t* src_s = reinterpret_cast<int32_t*>(smem_raw + Ly.src_off);
    int cnt = 0;
    for (int i = seg_lo; i < seg_hi; ++i) cnt += (i >= K) || flags[i];
    int total;
    const int dst0 = block_exclusive_scan<kT>(cnt, sh, &total);  // also a barrier after the staging above
    int dst = dst0;
    int first_ev = K;
    for (int i = seg_lo; i < seg_hi; ++i) {
        const bool keep = (i >= K) || flags[i];
        if (keep) {
            if (dst < K) src_s[dst] = i;
            ++dst;
        } else if (i < first_ev) {
            first_ev = i;
        }
        if (keep_dbg) keep_dbg[base + i] = keep ? 1 : 0;
        if (key_dbg && i >= K) key_dbg[base + i] = -1.f;
    }
    if (first_ev < K) atomicMin(&sh.first_evicted, first_ev);
    if (total != K) {  // cannot happen for a consistent state; the rows stay where they are
        if (tid == 0) record_error(p.err, kErrSelectCount);
        return;
    }
    __syncthreads();  // the kept list is complete
    // The kept list, positions and value magnitudes of the new slots, written slot by slot (coalesced) from the
    // old slots' copies in shared memory; the compressed value store also gets each new slot's reserved flag.
    int32_t* const src_u = src_out + static_cast<int64_t>(unit) * K;
    for (int j = tid; j < K; j += kT) {
        const int i = src_s[j];
        src_u[j] = i;
        pos[base + j] = pos_s[i];
        if (staged) vmag[base + j] = vm_s[i];
        // compressed value store: new slot j keeps a reserved (bf16) value if it is in R_B or R_V
        if (resv_out)
            resv_out[static_cast<int64_t>(unit) * store_resv_stride(K) + j] = (i >= K || (flags[i] & kFlagValue)) ? 1 : 0;
    }
    for (int i = K + tid; i < N; i += kT) pos[base + i] = -1;
    if (!staged) {  // value magnitudes through the same shared-memory array as the positions
        __syncthreads();
        vm_s = a_s;
        cp_async_words(vm_s, vmag + base, N);
        cp_async_wait_all();
        __syncthreads();
        for (int j = tid; j < K; j += kT) vmag[base + j] = vm_s[src_s[j]];
    }
    __syncthreads();  // the kept list and the lowest evicted slot are complete; the selection data is dead

    // ---- stable in-place gather of the kept K and V rows into slots 0..K-1 (the cache is restored to K
    // pairs, Sec. 2): warp 0 moves the K rows, warp 1 the V rows, through rings over the selection's
    // shared memory (written by generic stores until now: order them before the bulk copies).
    if (gbuf) {
        // Gather by every thread (the fused small-unit kernel): the moving rows go in blocks of gbuf_rows destination
        // rows; all the block's K and V source rows are read into shared memory, then (after a barrier) written to
        // their new slots.  In place this is safe: a block's sources lie at or above its first destination row, so
        // no earlier block's stores touch them, and within a block every read precedes every write.
        const int64_t unit_row = (static_cast<int64_t>(layer) * p.units + unit) * N;
        uint4* const kc = p.kc + unit_row * kVecPerRow;
        uint4* const vc = p.vc + unit_row * kVecPerRow;
        const int jf = sh.first_evicted;
        constexpr int kBatch = 8;  // loads in flight per thread before their shared-memory stores
        for (int j0 = jf; j0 < K; j0 += gbuf_rows) {
            const int n_vec = min(gbuf_rows, K - j0) * 2 * kVecPerRow;
            for (int e0 = 0; e0 < n_vec; e0 += kBatch * kT) {
                uint4 val[kBatch];
#pragma unroll
                for (int b = 0; b < kBatch; ++b) {
                    const int e = e0 + b * kT + tid;
                    if (e < n_vec) {
                        const int r = e >> 5, part = e & 31;
                        const int64_t row = src_s[j0 + r];
                        val[b] = part < kVecPerRow ? kc[row * kVecPerRow + part] : vc[row * kVecPerRow + part - kVecPerRow];
                    }
                }
#pragma unroll
                for (int b = 0; b < kBatch; ++b) {
                    const int e = e0 + b * kT + tid;
                    if (e < n_vec) gbuf[e] = val[b];
                }
            }
            __syncthreads();
            for (int e = tid; e < n_vec; e += kT) {
                const int r = e >> 5, part = e & 31;
                const int64_t row = j0 + r;
                if (part < kVecPerRow) kc[row * kVecPerRow + part] = gbuf[e];
                else vc[row * kVecPerRow + part - kVecPerRow] = gbuf[e];
            }
            __syncthreads();
        }
        return;
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    const int warp = tid >> 5;
    if (warp == 0 || (warp == 1 && p.vc)) {  // no V rows here with the compressed value store
        const int64_t unit_row = (static_cast<int64_t>(layer) * p.units + unit) * N;
        uint8_t* const rows = reinterpret_cast<uint8_t*>((warp == 0 ? p.kc : p.vc) + unit_row * kVecPerRow);
        gather_rows(rows, src_s, sh.first_evicted, K, smem_raw + warp * Ly.gather_stages * kGatherChunkBytes,
                    reinterpret_cast<uint64_t*>(smem_raw + Ly.bar_off) + warp * kGatherMaxStages, Ly.gather_stages,
                    p.err);
    }
}

template <int kT>
__global__ void __launch_bounds__(kT, 1024 / kT) select_kernel(const SelectParams p) {
    extern __shared__ __align__(16) uint8_t smem_raw[];
    __shared__ SelShared sh;
    select_unit<kT>(p, blockIdx.x, blockIdx.y, smem_raw, sh, false);
}

// ------------------------------------------------------------------ fused eviction of small units
// For launch-bound configurations (every unit of the launch fits in one wave, one CTA per unit) the window score,
// the selection and the gather run in one launch.  The unit's score matrix is small enough to stay in TMEM whole:
// S = K Q^T (M = 128 tokens per tile, N = the G*W window rows) for every 128-token tile, one tcgen05 product per
// (row, token) pair, no second transposed product and no second read of K.  With tokens in TMEM lanes, the
// softmax statistics of a window row are reductions across lanes (warp shuffles, then shared memory across the
// warps), and the per-token sum of Eq. (2) is a reduction along a lane's own columns.
struct SmallLayout {
    uint32_t sel_total, q_off, k_off, bar_off, part_off, row_off, slot_off, total;
};

__host__ __device__ inline SmallLayout small_layout(int N, int K, int GWp, int q_rows, int n_tiles, int stages) {
    SmallLayout L;
    uint32_t o = sel_layout(N, K, 1, true).total;
    L.sel_total = o;
    o = (o + 1023u) & ~1023u;
    L.q_off = o;
    o += static_cast<uint32_t>(q_rows) * kRowBytes;  // two 64-column panels of q_rows rows (the TMA box height)
    o = (o + 1023u) & ~1023u;
    L.k_off = o;
    o += static_cast<uint32_t>(stages) * kTileTokens * kRowBytes;
    L.bar_off = o;
    o += 8u * (2 + 2 * 8);
    L.part_off = o;
    o += 4u * static_cast<uint32_t>(n_tiles) * 4u * GWp;  // partial row statistics: [tile][lane quadrant][row]
    L.row_off = o;
    o += 4u * 2u * GWp;  // row offsets m_r, then -m'_r
    L.slot_off = o;
    o += 16;  // TMEM address, then the CTA-wide "waits completed" flag
    // the shared-memory gather of the selection overlays the score's buffers once they are dead: room for the K
    // rows of K and V
    const uint32_t gather = L.q_off + 2u * static_cast<uint32_t>(K) * kRowBytes;
    L.total = o > gather ? o : gather;
    return L;
}

// Reduce-scatter of a 32 x 32 block across a warp: lane l holds v[c] = its value of column c; afterwards lane l
// returns the reduction (max or sum) over the 32 lanes of column l.  Five halving steps: at offset o a lane keeps
// the half of its remaining columns whose bit o matches its own and receives the partner's partials of that half
// (16 + 8 + 4 + 2 + 1 = 31 shuffles in all, against 5 per column for 32 separate all-reduces).
template <bool kMax>
__device__ __forceinline__ float warp_reduce_scatter32(float (&v)[32]) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const bool hi = (lane & o) != 0;
#pragma unroll
        for (int i = 0; i < o; ++i) {
            const float keep = hi ? v[i + o] : v[i];
            const float send = hi ? v[i] : v[i + o];
            const float got = __shfl_xor_sync(0xffffffffu, send, o);
            v[i] = kMax ? fmaxf(keep, got) : keep + got;
        }
    }
    return v[0];
}

__device__ __forceinline__ float ex2_approx(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// The append of one unit (sequence s, KV head h) of layer slot z, the unit's share of what append_kernel does for
// a whole sequence: the key and value rows of the n new decode steps into slots fill .. fill + n - 1, with their
// positions and value magnitudes, and the query rows of its G heads for the steps that stay in the window ring
// (the last W).  A half warp moves one 256-byte row; every thread of the block calls it.
__device__ void append_unit(const AppendParams& p, int z, int s, int h) {
    const int layer = p.layer[z], fill = p.fill[z], n = p.n, W = p.W, N = p.N;
    const int G = p.Hq / p.Hkv;
    const int64_t unit = (static_cast<int64_t>(layer) * p.b + s) * p.Hkv + h;
    uint4* const kc = p.kc + unit * N * kVecPerRow;
    uint4* const vc = p.vc ? p.vc + unit * N * kVecPerRow : nullptr;
    int32_t* const pos = p.pos + unit * N;
    float* const vmag = p.vmag + unit * N;
    uint4* const qwin =
        p.qwin + ((static_cast<int64_t>(layer) * p.b + s) * p.Hq + static_cast<int64_t>(h) * G) * W * kVecPerRow;
    const uint4* const qin = p.q + static_cast<int64_t>(z) * p.q_stride;
    const uint4* const kin = p.k + static_cast<int64_t>(z) * p.kv_stride;
    const uint4* const vin = p.v + static_cast<int64_t>(z) * p.kv_stride;
    const int nq = min(n, W);          // steps n - nq .. n - 1 keep their queries
    const int rows = 2 * n + nq * G;   // key and value rows of every step (alternating), then the query rows
    // the trip count is the same for every thread of the block, so the half-warp shuffles see full warps
    for (int e0 = 0; e0 < rows * 16; e0 += blockDim.x) {
        const int e = e0 + static_cast<int>(threadIdx.x);
        const int r = e >> 4, seg = e & 15;
        uint4 val = make_uint4(0, 0, 0, 0);
        bool is_v = false;
        int t = 0;
        if (r < 2 * n) {
            t = r >> 1;
            const int64_t row_in = (static_cast<int64_t>(t) * p.b + s) * p.Hkv + h;
            if ((r & 1) == 0) {
                kc[static_cast<int64_t>(fill + t) * kVecPerRow + seg] = kin[row_in * kVecPerRow + seg];
            } else {
                is_v = true;
                val = vin[row_in * kVecPerRow + seg];
                if (vc) vc[static_cast<int64_t>(fill + t) * kVecPerRow + seg] = val;
            }
        } else if (r < rows) {
            const int qi = r - 2 * n;
            const int g = qi % G;
            t = n - nq + qi / G;
            const int slot = (p.q_ring[z] + t) % W;
            qwin[(static_cast<int64_t>(g) * W + slot) * kVecPerRow + seg] =
                qin[((static_cast<int64_t>(t) * p.b + s) * p.Hq + static_cast<int64_t>(h) * G + g) * kVecPerRow + seg];
        }
        if (__any_sync(0xffffffffu, is_v)) {
            const float mag = half_warp_value_magnitude(val, p.kind);
            if (is_v && seg == 0) vmag[fill + t] = mag;
        }
    }
    for (int t = threadIdx.x; t < n; t += blockDim.x) pos[fill + t] = static_cast<int32_t>(p.next_pos[z] + t);
}

__global__ void __launch_bounds__(kSmallThreads, 1)
    evict_small_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap qmap,
                       const SmallEvictParams p) {
    extern __shared__ __align__(1024) uint8_t smem_base[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_base) + 1023) & ~uintptr_t(1023));
    __shared__ SelShared sh;
    const SelectParams& sp = p.sel;
    const int N = sp.N, GWp = p.GWp, T = p.n_tiles, S = p.stages;
    const SmallLayout Ly = small_layout(N, sp.K, GWp, p.q_rows, T, S);
    uint8_t* q_s = smem + Ly.q_off;
    uint8_t* k_s = smem + Ly.k_off;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + Ly.bar_off);
    uint64_t* q_full = bars;           // [1]
    uint64_t* all_done = bars + 1;     // [1]
    uint64_t* k_full = bars + 2;       // [S]
    uint64_t* k_free = bars + 2 + 8;   // [S]
    float* part = reinterpret_cast<float*>(smem + Ly.part_off);  // [T][4][GWp]
    float* row_m = reinterpret_cast<float*>(smem + Ly.row_off);  // [GWp] row offset (exp2 domain)
    float* rown = row_m + GWp;                                   // [GWp] -m'_r
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + Ly.slot_off);
    volatile uint32_t* loads_ok = tmem_slot + 1;  // thread 0's waits all completed
    const int unit = blockIdx.x, z = blockIdx.y;
    const int layer = sp.batch.layer[z];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int seq = unit / sp.Hkv, head = unit - (unit / sp.Hkv) * sp.Hkv;
    const int64_t k_row = static_cast<int64_t>(layer) * p.layer_rows + static_cast<int64_t>(unit) * N;
    const int64_t q_row = static_cast<int64_t>(layer) * p.q_layer_rows +
                          (static_cast<int64_t>(seq) * p.Hq + static_cast<int64_t>(head) * p.G) * p.W;

    if (tid == 0) {
        *loads_ok = 1u;
        mbar_init(q_full, 1);
        mbar_init(all_done, 1);
        for (int s = 0; s < S; ++s) {
            mbar_init(&k_full[s], 1);
            mbar_init(&k_free[s], 1);
        }
        fence_mbar_init();
    }
    if (warp == 0) {
        tmem_alloc(tmem_slot, static_cast<uint32_t>(p.tmem_cols));
        tmem_relinquish();
    }
    if (p.append) {  // the step's append of this unit, then every row it wrote is visible to the loads below
        append_unit(p.ap, z, seq, head);
        asm volatile("fence.proxy.async.global;" ::: "memory");  // generic writes -> the TMA loads of K and Q
        __syncthreads();
    }
    // The selection's staged inputs land under the score (their region is free until then).  Where K fits the
    // rank count of warps 1.., those warps also rank R_V (it needs only the value magnitudes) while thread 0
    // issues the loads and products.
    constexpr int kTeam = kSmallThreads - 32;
    const bool rv_early = sp.staged && sp.variant == 0 && sp.K <= kTeam;
    if (sp.staged) {
        if (!rv_early) select_stage_rows(sp, unit, z, smem);
        else if (warp > 0) select_stage_rows(sp, unit, z, smem, tid - 32, kTeam);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t taddr = *tmem_slot;
    bool ok = true;

    // ---- loads and products, one thread: S_t = K_t Q^T for every tile t into TMEM columns [t*GWp, (t+1)*GWp)
    if (tid == 0) {
        tma_prefetch_desc(&kmap);
        tma_prefetch_desc(&qmap);
        const uint32_t q_panel = static_cast<uint32_t>(p.q_rows) * 128u;
        mbar_arrive_expect_tx(q_full, 2u * q_panel);
        for (int panel = 0; panel < 2; ++panel)
            tma_load_2d(q_s + panel * q_panel, &qmap, panel * 64, static_cast<int32_t>(q_row), q_full);
        auto load_tile = [&](int t) {
            const int st = t % S;
            uint8_t* dst = k_s + st * (kTileTokens * kRowBytes);
            const int32_t row = static_cast<int32_t>(k_row + static_cast<int64_t>(t) * kTileTokens);
            mbar_arrive_expect_tx(&k_full[st], kTileTokens * kRowBytes);
            tma_load_2d(dst, &kmap, 0, row, &k_full[st]);
            tma_load_2d(dst + kTileTokens * 128, &kmap, 64, row, &k_full[st]);
        };
        int issued = 0, landed = 0;  // tiles whose loads were issued / were seen to land
        for (int t = 0; t < S && t < T; ++t, ++issued) load_tile(t);
        const uint32_t idesc = idesc_bf16_f32(128, static_cast<uint32_t>(GWp));
        const uint64_t qdesc = sw128_kmajor_desc(smem_u32(q_s));
        const uint64_t kdesc = sw128_kmajor_desc(smem_u32(k_s));
        const bool q_ok = mbar_wait(q_full, 0, sp.err, kErrSmallQ);
        ok = q_ok;
        for (int t = 0; t < T; ++t) {
            const int st = t % S;
            if (ok && t < issued) {
                ok = mbar_wait(&k_full[st], (t / S) & 1, sp.err, kErrSmallKFull);
                if (ok) landed = t + 1;
            }
            tc_fence_after();
            if (ok) {
                const uint64_t kt = kdesc + ((static_cast<uint32_t>(st) * kTileTokens * kRowBytes) >> 4);
#pragma unroll
                for (int kk = 0; kk < 8; ++kk) {
                    const uint32_t koff = ((kk >> 2) * (kTileTokens * 128) + (kk & 3) * 32) >> 4;
                    const uint32_t qoff = ((kk >> 2) * q_panel + (kk & 3) * 32) >> 4;
                    tc_mma_bf16(taddr + static_cast<uint32_t>(t * GWp), kt + koff, qdesc + qoff, idesc,
                                kk > 0 ? 1u : 0u);
                }
            }
            tc_commit(&k_free[st]);  // the stage is free once these products have read it
            if (t + S < T && ok) {
                ok = mbar_wait(&k_free[st], (t / S) & 1, sp.err, kErrSmallKFree);
                if (ok) {
                    load_tile(t + S);
                    ++issued;
                }
            }
        }
        tc_commit(all_done);
        // after a wait ran out: every load that was issued lands before the CTA goes on (bounded waits)
        if (!q_ok) mbar_wait(q_full, 0, sp.err, kErrSmallQ);
        for (int t = landed; t < issued && !ok; ++t) mbar_wait(&k_full[t % S], (t / S) & 1, sp.err, kErrSmallKFull);
        if (!ok) *loads_ok = 0u;
    } else if (rv_early && warp > 0) {
        select_reserve_team(sp, unit, z, smem, tid - 32, kTeam, 1);
    }
    __syncwarp();
    if (!mbar_wait(all_done, 0, sp.err, kErrSmallDone)) atomicAnd(const_cast<uint32_t*>(loads_ok), 0u);
    tc_fence_after();

    // ---- softmax statistics of the window rows: warp w reads the lanes of quadrant w % 4 (32 tokens) of the
    // tiles t = w / 4, w / 4 + kSmallWarps / 4, ...; every column c is a window row
    const int quad = warp & 3;
    const uint32_t lane_base = static_cast<uint32_t>(quad * 32) << 16;
    const float cs = p.scale_log2;
    const int nch = GWp / 32;
    for (int t = warp >> 2; t < T; t += kSmallWarps / 4) {
        const bool valid = t * kTileTokens + quad * 32 + lane < N;
        for (int ch = 0; ch < nch; ++ch) {
            float v[32];
            tmem_ld32(taddr + lane_base + static_cast<uint32_t>(t * GWp + ch * 32), v);
            if (!valid) {
#pragma unroll
                for (int c = 0; c < 32; ++c) v[c] = -INFINITY;
            }
            part[(t * 4 + quad) * GWp + ch * 32 + lane] = warp_reduce_scatter32<true>(v);
        }
    }
    __syncthreads();
    for (int r = tid; r < GWp; r += kSmallThreads) {
        float m = -INFINITY;
        for (int j = 0; j < T * 4; ++j) m = fmaxf(m, part[j * GWp + r]);
        row_m[r] = m * cs;
    }
    __syncthreads();
    for (int t = warp >> 2; t < T; t += kSmallWarps / 4) {
        const bool valid = t * kTileTokens + quad * 32 + lane < N;
        for (int ch = 0; ch < nch; ++ch) {
            float v[32];
            tmem_ld32(taddr + lane_base + static_cast<uint32_t>(t * GWp + ch * 32), v);
#pragma unroll
            for (int c = 0; c < 32; ++c) v[c] = valid ? ex2_approx(fmaf(v[c], cs, -row_m[ch * 32 + c])) : 0.f;
            part[(t * 4 + quad) * GWp + ch * 32 + lane] = warp_reduce_scatter32<false>(v);
        }
    }
    __syncthreads();
    for (int r = tid; r < GWp; r += kSmallThreads) {
        float l = 0.f;
        for (int j = 0; j < T * 4; ++j) l += part[j * GWp + r];
        rown[r] = r < p.GW ? -(row_m[r] + log2f(l * static_cast<float>(p.fold_rows))) : -INFINITY;
    }
    __syncthreads();

    // ---- per-token score (Eq. (2)): sum over the window rows of the normalised weights, 1/(G*W) folded into rown
    // (GQA max: each head's sum over its W rows, the largest kept); into the selection's score array
    const SelLayout SL = sel_layout(N, sp.K, 1, true);
    float* a_s = reinterpret_cast<float*>(smem + SL.a_off);
    float* attn_out = p.attn ? p.attn + (static_cast<int64_t>(z) * sp.units + unit) * N : nullptr;
    for (int t = warp >> 2; t < T; t += kSmallWarps / 4) {
        const int token = t * kTileTokens + quad * 32 + lane;
        float acc = 0.f, head_sum = 0.f;
        int head_end = p.head_rows;
        for (int ch = 0; ch < nch; ++ch) {
            float v[32];
            tmem_ld32(taddr + lane_base + static_cast<uint32_t>(t * GWp + ch * 32), v);
            if (p.head_rows == 0) {
                float a0 = 0.f, a1 = 0.f;
#pragma unroll
                for (int c = 0; c < 32; c += 2) {
                    a0 += ex2_approx(fmaf(v[c], cs, rown[ch * 32 + c]));
                    a1 += ex2_approx(fmaf(v[c + 1], cs, rown[ch * 32 + c + 1]));
                }
                acc += a0 + a1;
            } else {
                for (int c = 0; c < 32; ++c) {
                    const int r = ch * 32 + c;
                    if (r >= p.GW) break;
                    if (r == head_end) {
                        acc = fmaxf(acc, head_sum);
                        head_sum = 0.f;
                        head_end += p.head_rows;
                    }
                    head_sum += ex2_approx(fmaf(v[c], cs, rown[r]));
                }
            }
        }
        if (p.head_rows != 0) acc = fmaxf(acc, head_sum);
        if (token < N) {
            a_s[token] = acc;
            if (attn_out) attn_out[token] = acc;
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(taddr, static_cast<uint32_t>(p.tmem_cols));
    if (tid == 0) {  // the barriers' memory is reused by the gather below
        mbar_inval(q_full);
        mbar_inval(all_done);
        for (int st = 0; st < S; ++st) {
            mbar_inval(&k_full[st]);
            mbar_inval(&k_free[st]);
        }
    }
    if (*loads_ok == 0u) {
        // a wait ran out (the same flag for every thread): the scores are not all there; leave the cache as it is
        // (the error word is set)
        return;
    }
    // ---- selection and gather on the scores just written (the selection's buffers sit below the score's)
    select_unit<kSmallThreads>(sp, unit, z, smem, sh, true, reinterpret_cast<uint4*>(smem + Ly.q_off), sp.K,
                               rv_early);
}



// Mixed-precision values (the quantizer of Sec. 4.4, the reserved cache of Sec. 6), one CTA per unit, right
// after an eviction (fill == K): the reserved (bf16) values are R_B, the last B slots, and R_V, the N_v largest
// value magnitudes among the first K - B slots (ties to the lower slot, the selection's own rule); every other
// kept value row gets b-bit codes Q = round((v - z) / s), z = min v, s = Range(v) / (2^b - 1), decided in fp32.
// Lane l of a warp holds dims 4l .. 4l+3 of a row and packs their four codes into 4b bits at byte 4l * b / 8.
__global__ void __launch_bounds__(kSelThreads) quantize_kernel(const QuantParams p) {
    extern __shared__ __align__(16) uint8_t smem_raw[];
    __shared__ SelShared sh;
    const int K = p.K;
    const int C = p.K - p.B;  // candidates of R_V
    uint32_t* ord = reinterpret_cast<uint32_t*>(smem_raw);
    const int ord_bytes = max(4 * ((C + 3) & ~3), 8 * p.mask_words);
    uint8_t* flags = smem_raw + ord_bytes;
    const int unit = blockIdx.x;
    const int tid = threadIdx.x;
    const int lane = tid & 31;
    const int warp = tid >> 5;
    const int64_t base = static_cast<int64_t>(unit) * p.N;
    for (int i = tid; i < K; i += kSelThreads) flags[i] = 0;
    for (int i = tid; i < C; i += kSelThreads) ord[i] = __float_as_uint(p.vmag[base + i]) + 1u;
    __syncthreads();
    const int seg = (C + kSelThreads - 1) / kSelThreads;
    const int seg_lo = min(C, tid * seg);
    const int seg_hi = min(C, seg_lo + seg);
    radix_top_k(ord, C, p.n_v, flags, kFlagValue, seg_lo, seg_hi, sh);  // ends with a barrier
    // reserved masks (shared memory over the dead selection keys, and global), then their prefix counts
    uint32_t* mask_s = ord;  // [mask_words], ord is no longer read
    uint32_t* pre_s = ord + p.mask_words;
    __syncthreads();
    for (int w = warp; w < p.mask_words; w += kSelWarps) {
        const int slot = 32 * w + lane;
        const bool res = slot < K && (slot >= C || flags[slot]);
        const uint32_t m = __ballot_sync(0xffffffffu, res);
        if (lane == 0) {
            p.rmask[static_cast<int64_t>(unit) * p.mask_words + w] = m;
            mask_s[w] = m;
        }
    }
    __syncthreads();
    if (tid == 0) {
        int run = 0;
        for (int w = 0; w < p.mask_words; ++w) {
            pre_s[w] = static_cast<uint32_t>(run);
            run += __popc(mask_s[w]);
        }
    }
    __syncthreads();
    // the reserved rows, copied in slot order to the unit's reserved cache (n_v + B rows)
    for (int j = warp; j < K; j += kSelWarps) {
        const uint32_t m = mask_s[j >> 5];
        if (!((m >> (j & 31)) & 1u)) continue;
        const int idx = static_cast<int>(pre_s[j >> 5]) + __popc(m & ((1u << (j & 31)) - 1u));
        const uint2 row = reinterpret_cast<const uint2*>(p.vc + (base + j) * kVecPerRow)[lane];
        reinterpret_cast<uint2*>(p.hp_rows + (static_cast<int64_t>(unit) * p.hp_cap + idx) * kVecPerRow)[lane] = row;
    }
    for (int j = warp; j < C; j += kSelWarps) {
        if (flags[j]) continue;  // R_V keeps its bf16 row (uniform over the warp)
        const uint2 raw = reinterpret_cast<const uint2*>(p.vc + (base + j) * kVecPerRow)[lane];
        quantize_row_warp(raw, p.bits, lane, p.codes + (static_cast<int64_t>(unit) * K + j) * p.row_bytes,
                          p.qparams + (static_cast<int64_t>(unit) * p.Kp + j) * 2);
    }
}

}  // namespace

cudaError_t launch_append(const AppendParams& p, int n_layers, cudaStream_t s) {
    // four steps per block, or one where four would leave fewer blocks than the GPU's 152 SMs (small,
    // latency-bound appends)
    AppendParams q = p;
    q.steps_per_block = static_cast<int64_t>((p.n + kAppendSteps - 1) / kAppendSteps) * p.b * n_layers < 152
                            ? 1 : kAppendSteps;
    const int chunks = (p.n + q.steps_per_block - 1) / q.steps_per_block;
    append_kernel<<<dim3(static_cast<unsigned>(chunks * p.b), static_cast<unsigned>(n_layers)), 256, 0, s>>>(q);
    return cudaGetLastError();
}

cudaError_t launch_value_score(const ValueParams& p, int num_sms, cudaStream_t s) {
    const int threads = 256;
    const int64_t rows = static_cast<int64_t>(p.units) * p.rows;
    int64_t blocks = (rows + (threads / 16) - 1) / (threads / 16);
    const int64_t cap = static_cast<int64_t>(num_sms) * 8;
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    value_score_kernel<<<static_cast<unsigned>(blocks), threads, 0, s>>>(p);
    return cudaGetLastError();
}

size_t select_smem_bytes(int N, int K, int n_parts, bool staged) { return sel_layout(N, K, n_parts, staged).total; }
size_t select_static_smem_bytes() { return sizeof(SelShared); }

cudaError_t select_set_attributes(size_t smem_bytes) {
    for (auto fn : {select_kernel<256>, select_kernel<512>, select_kernel<1024>}) {
        const cudaError_t e =
            cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem_bytes));
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

size_t quantize_smem_bytes(int K, int B) {
    const size_t words = 4u * ((K - B + 3) & ~3);
    const size_t masks = 8u * ((K + 31) / 32);  // masks and their prefix counts, over the selection keys
    return (words > masks ? words : masks) + K;
}

cudaError_t quantize_set_attributes(size_t smem_bytes) {
    return cudaFuncSetAttribute(quantize_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                static_cast<int>(smem_bytes));
}

cudaError_t launch_quantize(const QuantParams& p, int units, size_t smem_bytes, cudaStream_t s) {
    quantize_kernel<<<static_cast<unsigned>(units), kSelThreads, smem_bytes, s>>>(p);
    return cudaGetLastError();
}

size_t evict_small_smem_bytes(int N, int K, int GWp, int q_rows, int n_tiles, int stages) {
    return small_layout(N, K, GWp, q_rows, n_tiles, stages).total + 1024;
}

cudaError_t evict_small_set_attributes(size_t smem_bytes) {
    return cudaFuncSetAttribute(evict_small_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                static_cast<int>(smem_bytes));
}

cudaError_t launch_evict_small(const CUtensorMap& kmap, const CUtensorMap& qmap, const SmallEvictParams& p, int units,
                               size_t smem_bytes, cudaStream_t s) {
    evict_small_kernel<<<dim3(static_cast<unsigned>(units), static_cast<unsigned>(p.sel.batch.n)), kSmallThreads,
                         smem_bytes, s>>>(kmap, qmap, p);
    return cudaGetLastError();
}

cudaError_t launch_select(const SelectParams& p, int units, size_t smem_bytes, int threads, cudaStream_t s) {
    const dim3 grid(static_cast<unsigned>(units), static_cast<unsigned>(p.batch.n));
    if (threads == 1024) select_kernel<1024><<<grid, 1024, smem_bytes, s>>>(p);
    else if (threads == 512) select_kernel<512><<<grid, 512, smem_bytes, s>>>(p);
    else select_kernel<256><<<grid, 256, smem_bytes, s>>>(p);
    return cudaGetLastError();
}

}  // namespace vase
