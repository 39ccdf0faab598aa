// Compressed value store: the mixed-precision value cache Sec. 6 proposes, with the per-token b-bit quantizer of
// Sec. 4.4.  Keys stay in the bf16 K cache; a value is held either as a bf16 row in the unit's reserved cache or
// as its codes and (s, z).  Per layer and unit:
//   codes [N][16 b] bytes, (s, z) [Np][2] fp32, mask [mask_stride] words (bit j: slot j's value is bf16),
//   ring [H][256 bytes] (the bf16 values in slot order, entry i at row (head + i) mod H), state (head, count).
// H = N_v + 2B: R_V and R_B after an eviction (at most N_v + B values) plus the B values appended before the next.
//   * An append puts each new value in the ring.  If the ring is full, its earliest value is quantized into the
//     codes (the rule Sec. 6 states); that can only happen before the first eviction.
//   * An eviction (after the selection, which leaves the kept list src and the R_V u R_B flags) moves the codes
//     of kept coded values to their new slots, closes up the ring over the kept values of R_V u R_B, and quantizes
//     the kept bf16 values that are in neither (they no longer hold a reserved slot).  A quantized value never
//     becomes bf16 again: R_V is drawn from the earlier R_V and the new values only, since R_V is kept whole.
#include "kernels.cuh"
#include "ptx.cuh"
#include "quant.cuh"

namespace vase {

namespace {

constexpr int kStoreThreads = 256;
constexpr int kStoreWarps = kStoreThreads / 32;
constexpr int kStoreRowsPerWarp = 16;  // rows a warp has in flight per phase of the eviction sweep
constexpr int kRowWords2 = 32;         // uint2 per 256-byte row
constexpr int kEvictPhase = 64;        // new slots per phase of the eviction sweep
constexpr int kEvictBufs = 2;          // phases of the sweep in flight

struct StoreUnit {
    uint8_t* codes;
    float* sz;
    uint32_t* mask;
    uint2* ring;
    int32_t* state;
};

__device__ __forceinline__ StoreUnit store_unit(const StoreParams& p, int layer, int unit) {
    uint8_t* base = p.base + static_cast<int64_t>(layer) * p.layer_bytes;
    StoreUnit u;
    u.codes = base + p.codes_off + static_cast<int64_t>(unit) * p.N * p.code_row;
    u.sz = reinterpret_cast<float*>(base + p.qp_off) + static_cast<int64_t>(unit) * p.Np * 2;
    u.mask = reinterpret_cast<uint32_t*>(base + p.mask_off) + static_cast<int64_t>(unit) * p.mask_stride;
    u.ring = reinterpret_cast<uint2*>(base + p.ring_off) + static_cast<int64_t>(unit) * p.H * kRowWords2;
    u.state = reinterpret_cast<int32_t*>(base + p.state_off) + unit * 4;
    return u;
}

__device__ __forceinline__ int wrap(int x, int H) { return x >= H ? x - H : x; }  // 0 <= x < 2H

// Asynchronous global -> shared copies of 4, 8 or 16 bytes (both addresses aligned to the size); completion by
// cp_async_all().
template <int kBytes>
__device__ __forceinline__ void cp_async(void* smem_dst, const void* gsrc) {
    if (kBytes == 16)
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(smem_dst)), "l"(gsrc) : "memory");
    else
        asm volatile("cp.async.ca.shared.global [%0], [%1], %2;" ::"r"(smem_u32(smem_dst)), "l"(gsrc), "n"(kBytes)
                     : "memory");
}
__device__ __forceinline__ void cp_async_all() {
    asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
}
// The copies issued since the last commit form a group; cp_async_wait_prior<n>() waits for every group but the
// latest n.
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int kPending>
__device__ __forceinline__ void cp_async_wait_prior() {
    asm volatile("cp.async.wait_group %0;" ::"n"(kPending) : "memory");
}

// Exclusive scan of one value per thread over the block; *total gets the sum.  Starts and ends with a barrier
// (so consecutive scans may share warp_sums).
__device__ __forceinline__ int block_scan(int v, int* warp_sums, int* total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    __syncthreads();
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) warp_sums[warp] = x;
    __syncthreads();
    if (threadIdx.x == 0) {
        int run = 0;
        for (int w = 0; w < kStoreWarps; ++w) {
            const int t = warp_sums[w];
            warp_sums[w] = run;
            run += t;
        }
        warp_sums[kStoreWarps] = run;
    }
    __syncthreads();
    *total = warp_sums[kStoreWarps];
    return warp_sums[warp] + x - v;
}

// ------------------------------------------------------------------ append
// Shared memory of the append: the unit's masks and the scan sums; with an overflow (big) also the entry list,
// the candidates' magnitudes, a histogram and the row stage.
struct StoreAppendSmem {
    uint32_t mask_off, scan_off, ent_off, vm_off, hist_off, stage_off, total;
};

__host__ __device__ inline StoreAppendSmem store_append_layout(int mask_stride, int entries, int cands) {
    StoreAppendSmem L;
    uint32_t o = 0;
    L.mask_off = o;
    o += 4u * mask_stride;
    L.scan_off = o;
    o += 4u * (kStoreWarps + 4);
    L.ent_off = o;
    o += 4u * entries;
    L.vm_off = o;
    o += 4u * cands;
    L.hist_off = o;
    o += entries > 0 ? 4u * 256 : 0u;
    o = (o + 15u) & ~15u;
    L.stage_off = o;
    o += entries > 0 ? kStoreWarps * kStoreRowsPerWarp * 256u : 0u;
    L.total = (o + 15u) & ~15u;
    return L;
}

// One CTA per (layer slot, unit).  The n new values of slots fill .. fill + n - 1 join the ring behind its count
// entries.  If that is more than H (only before the first eviction), the earliest values of the combined list
// that are not large-Range leave for the codes, as many as it is over, and the rest close up in slot order
// behind the unchanged head.  Large-Range: the N_v largest value magnitudes among the slots below
// min(fill + n, K), the set R_V would be now (ties to the lower slot).
__global__ void __launch_bounds__(kStoreThreads) store_append_kernel(const StoreParams p) {
    extern __shared__ __align__(16) uint8_t smem[];
    const int z = blockIdx.y;
    const int unit = blockIdx.x;
    const int layer = p.layer[z];
    const int fill = p.fill[z];
    const int n = p.n;
    const int H = p.H;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const StoreAppendSmem Ly = store_append_layout(p.mask_stride, p.big ? H + n : 0, p.big ? p.K : 0);
    uint32_t* mask_s = reinterpret_cast<uint32_t*>(smem + Ly.mask_off);
    int* scan_s = reinterpret_cast<int*>(smem + Ly.scan_off);
    const StoreUnit u = store_unit(p, layer, unit);
    const bool fresh = fill == 0;  // the layer's first append: the store holds nothing yet
    const int head = fresh ? 0 : u.state[0];
    const int count = fresh ? 0 : u.state[1];
    if (head < 0 || head >= H || count < 0 || count > H || count > fill) {  // not a state this kernel wrote
        if (tid == 0) record_error(p.err, kErrStoreState);
        return;
    }
    const int ov = max(0, count + n - H);  // values leaving the ring
    if (ov > 0 && (p.round[z] > 0 || !p.big)) {
        // After an eviction the ring holds at most N_v + B values and at most B are appended before the next one,
        // so it cannot overflow; if it would, the caller's state is inconsistent.  Nothing is written.
        if (tid == 0) record_error(p.err, kErrStoreOverflow);
        return;
    }
    for (int w = tid; w < p.mask_words; w += kStoreThreads) mask_s[w] = fresh ? 0u : u.mask[w];
    const int s_seq = unit / p.Hkv;
    const int h = unit - s_seq * p.Hkv;
    const uint2* vin = reinterpret_cast<const uint2*>(p.v + static_cast<int64_t>(z) * p.kv_stride);
    auto in_row = [&](int t) { return vin + ((static_cast<int64_t>(t) * p.b + s_seq) * p.Hkv + h) * kRowWords2; };
    __syncthreads();
    if (ov == 0) {
        // every new value joins the ring behind its entries
        for (int t = warp; t < n; t += kStoreWarps) {
            const int f = fill + t;
            u.ring[((head + count + t) % H) * kRowWords2 + lane] = in_row(t)[lane];
            if (lane == 0) atomicOr(&mask_s[f >> 5], 1u << (f & 31));
        }
        __syncthreads();
        for (int w = tid; w < p.mask_words; w += kStoreThreads) u.mask[w] = mask_s[w];
        if (tid == 0) {
            u.state[0] = head;
            u.state[1] = count + n;
        }
        return;
    }

    // ---- the ring overflows.  Entries e: the old ones (e < count: the bf16 slots in slot order) and the new
    // ones (e = count + t: slot fill + t).
    uint32_t* ent_s = reinterpret_cast<uint32_t*>(smem + Ly.ent_off);  // slot | r << 15 | spilled << 31
    const int E = count + n;
    {   // (a) the old entries' slots from the mask
        const int per = (p.mask_words + kStoreThreads - 1) / kStoreThreads;
        const int w0 = min(p.mask_words, tid * per), w1 = min(p.mask_words, w0 + per);
        int c = 0;
        for (int w = w0; w < w1; ++w) c += __popc(mask_s[w]);
        int total;
        int at = block_scan(c, scan_s, &total);
        if (total != count) {  // masks that disagree with the ring state: nothing is written
            if (tid == 0) record_error(p.err, kErrStoreState);
            return;
        }
        for (int w = w0; w < w1; ++w)
            for (uint32_t m = mask_s[w]; m; m &= m - 1) ent_s[at++] = 32u * w + __ffs(m) - 1;
        for (int e = count + tid; e < E; e += kStoreThreads) ent_s[e] = static_cast<uint32_t>(fill + e - count);
    }
    // (b) the large-Range set: keys (magnitude bits; magnitudes are >= 0, so the bits order like the values)
    // above thr, and those equal to thr up to slot tie_slot
    const int C = min(fill + n, p.K);
    uint32_t thr = 0u;
    int tie_slot = -1;
    const bool all_large = p.n_v >= C;
    float* vm_s = reinterpret_cast<float*>(smem + Ly.vm_off);
    if (!all_large && p.n_v > 0) {
        const float* vmag = p.vmag + (static_cast<int64_t>(layer) * p.units + unit) * p.N;
        for (int s = tid; s < C; s += kStoreThreads) cp_async<4>(vm_s + s, vmag + s);
        cp_async_all();
        int* hist = reinterpret_cast<int*>(smem + Ly.hist_off);
        uint32_t prefix = 0u, pmask = 0u;
        int k = p.n_v;  // rank still to find among the keys that match the prefix
        for (int pass = 0; pass < 4; ++pass) {
            const int shift = 24 - 8 * pass;
            __syncthreads();
            for (int b = tid; b < 256; b += kStoreThreads) hist[b] = 0;
            __syncthreads();
            for (int s = tid; s < C; s += kStoreThreads) {
                const uint32_t key = __float_as_uint(vm_s[s]);
                if ((key & pmask) == prefix) atomicAdd(&hist[(key >> shift) & 255u], 1);
            }
            __syncthreads();
            if (tid == 0) {
                int acc = 0, sel = 0;
                for (int b = 255; b >= 0; --b) {
                    if (acc + hist[b] >= k) {
                        sel = b;
                        break;
                    }
                    acc += hist[b];
                }
                scan_s[kStoreWarps + 1] = sel;
                scan_s[kStoreWarps + 2] = k - acc;
            }
            __syncthreads();
            prefix |= static_cast<uint32_t>(scan_s[kStoreWarps + 1]) << shift;
            pmask |= 0xFFu << shift;
            k = scan_s[kStoreWarps + 2];
        }
        thr = prefix;
        // the k-th lowest slot whose key equals thr
        const int per = (C + kStoreThreads - 1) / kStoreThreads;
        const int s0 = min(C, tid * per), s1 = min(C, s0 + per);
        int c = 0;
        for (int s = s0; s < s1; ++s) c += __float_as_uint(vm_s[s]) == thr;
        int total;
        const int before = block_scan(c, scan_s, &total);
        if (before < k && k <= before + c) {
            int seen = before;
            for (int s = s0; s < s1; ++s)
                if (__float_as_uint(vm_s[s]) == thr && ++seen == k) scan_s[kStoreWarps + 3] = s;
        }
        __syncthreads();
        tie_slot = scan_s[kStoreWarps + 3];
    }
    auto large = [&](int s) {
        if (s >= C || p.n_v == 0) return false;
        if (all_large) return true;
        const uint32_t key = __float_as_uint(vm_s[s]);
        return key > thr || (key == thr && s <= tie_slot);
    };
    // (c) the earliest ov entries that are not large-Range leave; the others get their new index r
    {
        const int per = (E + kStoreThreads - 1) / kStoreThreads;
        const int e0 = min(E, tid * per), e1 = min(E, e0 + per);
        int c = 0;
        for (int e = e0; e < e1; ++e) c += !large(static_cast<int>(ent_s[e] & 0x7FFFu));
        int total;
        int before = block_scan(c, scan_s, &total);  // unprotected entries before e0
        int gone = before < ov ? before : ov;         // spilled entries before e0
        for (int e = e0; e < e1; ++e) {
            const uint32_t slot = ent_s[e] & 0x7FFFu;
            const bool spill = !large(static_cast<int>(slot)) && before++ < ov;
            ent_s[e] = spill ? (slot | 1u << 31) : (slot | static_cast<uint32_t>(e - gone) << 15);
            gone += spill;
        }
    }
    __syncthreads();
    // (d) the moves, in ascending phases (every read of a phase before any of its writes; a phase reads ring
    // entries e and writes entries r <= e, so no later phase reads what an earlier one wrote)
    uint2* stage = reinterpret_cast<uint2*>(smem + Ly.stage_off) + warp * kStoreRowsPerWarp * kRowWords2;
    constexpr int kPhase = kStoreWarps * kStoreRowsPerWarp;
    for (int base = 0; base < E; base += kPhase) {
#pragma unroll
        for (int i = 0; i < kStoreRowsPerWarp; ++i) {
            const int e = base + warp * kStoreRowsPerWarp + i;
            if (e < E) {
                const uint32_t info = ent_s[e];
                const bool spill = info >> 31;
                const int r = static_cast<int>((info >> 15) & 0x7FFFu);
                if (e >= count) cp_async<8>(stage + i * kRowWords2 + lane, in_row(e - count) + lane);
                else if (spill || r != e) cp_async<8>(stage + i * kRowWords2 + lane, u.ring + wrap(head + e, H) * kRowWords2 + lane);
            }
        }
        cp_async_all();
        __syncthreads();
#pragma unroll
        for (int i = 0; i < kStoreRowsPerWarp; ++i) {
            const int e = base + warp * kStoreRowsPerWarp + i;
            if (e < E) {
                const uint32_t info = ent_s[e];
                const int slot = static_cast<int>(info & 0x7FFFu);
                const bool spill = info >> 31;
                const int r = static_cast<int>((info >> 15) & 0x7FFFu);
                if (spill) {
                    quantize_row_warp(stage[i * kRowWords2 + lane], p.bits, lane,
                                      u.codes + static_cast<int64_t>(slot) * p.code_row, u.sz + 2 * slot);
                    if (lane == 0) atomicAnd(&mask_s[slot >> 5], ~(1u << (slot & 31)));
                } else {
                    if (e >= count || r != e) u.ring[wrap(head + r, H) * kRowWords2 + lane] = stage[i * kRowWords2 + lane];
                    if (lane == 0) atomicOr(&mask_s[slot >> 5], 1u << (slot & 31));
                }
            }
        }
        __syncwarp();
    }
    __syncthreads();
    for (int w = tid; w < p.mask_words; w += kStoreThreads) u.mask[w] = mask_s[w];
    if (tid == 0) {
        u.state[0] = head;
        u.state[1] = E - ov;
    }
}

// ------------------------------------------------------------------ eviction
constexpr uint32_t kKindCoded = 0, kKindRing = 1, kKindSpill = 2;

struct StoreEvictSmem {
    uint32_t src_off, info_off, resv_off, mask_off, pre_off, stage_off, sz_off, scan_off, total;
};

__host__ __device__ inline StoreEvictSmem store_evict_layout(int K, int mask_stride) {
    StoreEvictSmem L;
    uint32_t o = 0;
    L.src_off = o;
    o += 4u * K;
    L.info_off = o;
    o += 4u * K;
    o = (o + 15u) & ~15u;
    L.resv_off = o;
    o += static_cast<uint32_t>(store_resv_stride(K));
    L.mask_off = o;
    o += 4u * mask_stride;
    L.pre_off = o;
    o += 4u * mask_stride;
    o = (o + 15u) & ~15u;
    L.stage_off = o;
    o += static_cast<uint32_t>(kEvictBufs * kEvictPhase) * 256u;
    L.sz_off = o;
    o += static_cast<uint32_t>(kEvictBufs * kEvictPhase) * 8u;
    L.scan_off = o;
    o += 4u * (kStoreWarps + 1);
    L.total = (o + 15u) & ~15u;
    return L;
}

// One CTA per (layer slot, unit), after the selection.  New slot j holds old slot src[j]:
//   old value coded              -> its codes and (s, z) move from src[j] to j;
//   old value bf16, j in R_V u R_B -> its ring entry moves from old index o (its rank among the old bf16 slots)
//                                   to r (its rank among the kept ones), r <= o, under the same head;
//   old value bf16, otherwise    -> quantized from its ring row into slot j's codes.
// In place, in ascending phases of new slots; within a phase every read precedes every write (a barrier).  Across
// phases nothing conflicts: a phase reads codes at src[j] >= j and ring entries o, both above what any earlier
// phase wrote (src is increasing and r <= o), and it writes only after its own reads.
__global__ void __launch_bounds__(kStoreThreads) store_evict_kernel(const StoreParams p) {
    extern __shared__ __align__(16) uint8_t smem[];
    const int K = p.K;
    const StoreEvictSmem Ly = store_evict_layout(K, p.mask_stride);
    // the kept list src[j], and slot j's info word: kind << 30 | s for a coded value (s = src[j]), kind << 30 |
    // o << 15 | r for a bf16 one (o its old ring rank, r its new one where it stays in the ring).  (One array could
    // hold both and let a fifth CTA onto an SM; at the Qwen3-1.7B geometry that measured slower.)
    int32_t* src_s = reinterpret_cast<int32_t*>(smem + Ly.src_off);
    uint32_t* info_s = reinterpret_cast<uint32_t*>(smem + Ly.info_off);
    uint8_t* resv_s = smem + Ly.resv_off;
    uint32_t* mask_s = reinterpret_cast<uint32_t*>(smem + Ly.mask_off);
    uint32_t* pre_s = reinterpret_cast<uint32_t*>(smem + Ly.pre_off);
    int* scan_s = reinterpret_cast<int*>(smem + Ly.scan_off);
    const int z = blockIdx.y;
    const int unit = blockIdx.x;
    const int layer = p.layer[z];
    const int H = p.H;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const StoreUnit u = store_unit(p, layer, unit);
    const int32_t* src = p.src + (static_cast<int64_t>(z) * p.units + unit) * K;
    const int Kr = store_resv_stride(K);
    const uint8_t* resv = p.resv + (static_cast<int64_t>(z) * p.units + unit) * Kr;
    const int head = u.state[0];

    // the kept list, its R_V u R_B flags and the old bf16 mask, copied to shared memory all at once
    for (int j = tid; j < K; j += kStoreThreads) cp_async<4>(src_s + j, src + j);
    for (int c = tid; c < Kr / 16; c += kStoreThreads) cp_async<16>(resv_s + 16 * c, resv + 16 * c);
    for (int w = tid; w < p.mask_words; w += kStoreThreads) cp_async<4>(mask_s + w, u.mask + w);
    cp_async_all();
    __syncthreads();
    // exclusive prefix counts of the old mask words
    {
        const int per = (p.mask_words + kStoreThreads - 1) / kStoreThreads;
        const int w0 = min(p.mask_words, tid * per), w1 = min(p.mask_words, w0 + per);
        int c = 0;
        for (int w = w0; w < w1; ++w) c += __popc(mask_s[w]);
        int total;
        int run = block_scan(c, scan_s, &total);
        for (int w = w0; w < w1; ++w) {
            pre_s[w] = static_cast<uint32_t>(run);
            run += __popc(mask_s[w]);
        }
        if (head < 0 || head >= H || total > H) {  // not a state this library wrote: touch nothing
            if (tid == 0) record_error(p.err, kErrStoreState);
            return;
        }
    }
    // each new slot's kind, old ring index o and (kept bf16 of R_V u R_B) new ring index r
    const int seg = (K + kStoreThreads - 1) / kStoreThreads;
    const int j0 = min(K, tid * seg), j1 = min(K, j0 + seg);
    __syncthreads();
    int n_ring = 0;
    for (int j = j0; j < j1; ++j) {
        const int s = src_s[j];
        const uint32_t w = mask_s[s >> 5];
        const bool bf = (w >> (s & 31)) & 1u;
        const uint32_t o = pre_s[s >> 5] + __popc(w & ((1u << (s & 31)) - 1u));
        const uint32_t kind = !bf ? kKindCoded : (resv_s[j] ? kKindRing : kKindSpill);
        n_ring += kind == kKindRing;
        info_s[j] = kind == kKindCoded ? static_cast<uint32_t>(s) : kind << 30 | (o & 0x7FFFu) << 15;
    }
    int total_ring;
    int r = block_scan(n_ring, scan_s, &total_ring);
    for (int j = j0; j < j1; ++j)
        if ((info_s[j] >> 30) == kKindRing) info_s[j] |= static_cast<uint32_t>(r++);
    __syncthreads();
    // the new mask (slots K .. N - 1 are empty after the eviction)
    for (int w = warp; w < p.mask_words; w += kStoreWarps) {
        const int j = 32 * w + lane;
        const uint32_t m = __ballot_sync(0xffffffffu, j < K && (info_s[j] >> 30) == kKindRing);
        if (lane == 0) u.mask[w] = m;
    }
    if (tid == 0) u.state[1] = total_ring;

    // The moves, in phases of kEvictPhase new slots, kEvictBufs phases in flight: the reads of phase i + 1 ..
    // i + kEvictBufs - 1 are issued before the writes of phase i.  That is safe because no phase reads what an earlier phase writes: codes and
    // (s, z) are read at src[j] >= j and written at j, and a ring entry is read at its old rank o, which is at
    // least every new rank r of the slots before it, where the earlier phases write.  Within a phase every read
    // precedes every write (a barrier), and a buffer is refilled only after the phase that used it is done.
    // Thread t < kEvictPhase owns slot base + t and moves its whole row with 16-byte copies (a code row and its
    // (s, z), or a 256-byte ring row); the rows to quantize are staged the same way and then quantized by the
    // warps (one warp per row: the quantizer reduces over the row's lanes).  Row t's 16-byte piece c sits at
    // piece c ^ (t % 16) of its 256 bytes, so that the threads of a warp, each on its own row, touch different
    // banks.
    uint4* const stage4 = reinterpret_cast<uint4*>(smem + Ly.stage_off);   // [kEvictBufs][kEvictPhase][16]
    float2* const stage_sz = reinterpret_cast<float2*>(smem + Ly.sz_off);  // [kEvictBufs][kEvictPhase]
    const int code_vecs = p.code_row / 16;  // 16-byte pieces of a code row (2, 4 or 8)
    uint8_t* const codes = u.codes;
    const uint4* const ring4 = reinterpret_cast<const uint4*>(u.ring);
    const int sw = tid & 15;
    // this thread's slot of the phase at `base`: its reads into buffer `buf`
    auto issue_reads = [&](int base, int buf) {
        const int j = base + tid;
        if (tid >= kEvictPhase || j >= K) return;
        const uint32_t info = info_s[j];
        const uint32_t kind = info >> 30;
        const int o = static_cast<int>((info >> 15) & 0x7FFFu);
        const int rr = static_cast<int>(info & 0x7FFFu);
        uint4* dst = stage4 + (buf * kEvictPhase + tid) * 16;
        if (kind == kKindCoded) {
            const int s = static_cast<int>(info & 0x3FFFFFFFu);
            if (s != j) {  // in place already otherwise
                const uint4* src = reinterpret_cast<const uint4*>(codes + static_cast<int64_t>(s) * p.code_row);
                for (int c = 0; c < code_vecs; ++c) cp_async<16>(dst + (c ^ sw), src + c);
                cp_async<8>(stage_sz + buf * kEvictPhase + tid, u.sz + 2 * s);
            }
        } else if (kind == kKindSpill || o != rr) {
            const uint4* src = ring4 + static_cast<int64_t>(wrap(head + o, H)) * 16;
#pragma unroll
            for (int c = 0; c < 16; ++c) cp_async<16>(dst + (c ^ sw), src + c);
        }
    };
    const int n_phase = (K + kEvictPhase - 1) / kEvictPhase;
    for (int ph = 0; ph < kEvictBufs - 1; ++ph) {
        if (ph < n_phase) issue_reads(ph * kEvictPhase, ph);
        cp_async_commit();
    }
    for (int ph = 0; ph < n_phase; ++ph) {
        const int base = ph * kEvictPhase, buf = ph % kEvictBufs;
        const int ahead = ph + kEvictBufs - 1;
        if (ahead < n_phase) issue_reads(ahead * kEvictPhase, ahead % kEvictBufs);
        cp_async_commit();
        cp_async_wait_prior<kEvictBufs - 1>();  // this thread's reads of phase ph have landed
        __syncthreads();        // every read of phase ph precedes every write
        const int j = base + tid;
        if (tid < kEvictPhase && j < K) {
            const uint32_t info = info_s[j];
            const uint32_t kind = info >> 30;
            const int o = static_cast<int>((info >> 15) & 0x7FFFu);
            const int rr = static_cast<int>(info & 0x7FFFu);
            const uint4* srow = stage4 + (buf * kEvictPhase + tid) * 16;
            if (kind == kKindCoded) {
                if (static_cast<int>(info & 0x3FFFFFFFu) != j) {
                    uint4* d = reinterpret_cast<uint4*>(codes + static_cast<int64_t>(j) * p.code_row);
                    for (int c = 0; c < code_vecs; ++c) d[c] = srow[c ^ sw];
                    *reinterpret_cast<float2*>(u.sz + 2 * j) = stage_sz[buf * kEvictPhase + tid];
                }
            } else if (kind == kKindRing && o != rr) {
                uint4* d = reinterpret_cast<uint4*>(u.ring) + static_cast<int64_t>(wrap(head + rr, H)) * 16;
#pragma unroll
                for (int c = 0; c < 16; ++c) d[c] = srow[c ^ sw];
            }
        }
        // the rows to quantize: warp w takes the phase's slots w, w + kStoreWarps, ... (the test is uniform)
        for (int t = warp; t < kEvictPhase; t += kStoreWarps) {
            const int jj = base + t;
            if (jj >= K || (info_s[jj] >> 30) != kKindSpill) continue;
            const uint4* srow = stage4 + (buf * kEvictPhase + t) * 16;
            const uint2 raw = reinterpret_cast<const uint2*>(srow + ((lane >> 1) ^ (t & 15)))[lane & 1];
            quantize_row_warp(raw, p.bits, lane, codes + static_cast<int64_t>(jj) * p.code_row, u.sz + 2 * jj);
        }
        __syncthreads();  // buffer `buf` is read before the reads of phase ph + kEvictBufs refill it
    }
}

}  // namespace

size_t store_evict_smem_bytes(int K, int mask_stride) { return store_evict_layout(K, mask_stride).total; }

cudaError_t store_set_attributes(size_t evict_smem, size_t append_smem) {
    cudaError_t e = cudaFuncSetAttribute(store_evict_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(evict_smem));
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(store_append_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 static_cast<int>(append_smem));
    return e;
}

size_t store_append_smem_bytes(int mask_stride, int H, int n, int K, bool big) {
    return store_append_layout(mask_stride, big ? H + n : 0, big ? K : 0).total;
}

cudaError_t launch_store_append(const StoreParams& p, int n_layers, cudaStream_t s) {
    const size_t smem = store_append_smem_bytes(p.mask_stride, p.H, p.n, p.K, p.big != 0);
    store_append_kernel<<<dim3(static_cast<unsigned>(p.units), static_cast<unsigned>(n_layers)), kStoreThreads,
                          smem, s>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_store_evict(const StoreParams& p, int n_layers, cudaStream_t s) {
    store_evict_kernel<<<dim3(static_cast<unsigned>(p.units), static_cast<unsigned>(n_layers)), kStoreThreads,
                         store_evict_smem_bytes(p.K, p.mask_stride), s>>>(p);
    return cudaGetLastError();
}

}  // namespace vase
