// Bandwidth kernels of the eviction step: window/cache append, value
// magnitude, selection (reservation + stochastic top-k) and the stable
// in-place compaction of the kept rows.
#include <cfloat>
#include <cuda_bf16.h>

#include "kernels.cuh"
#include "ptx.cuh"

namespace vase {

namespace {

// ------------------------------------------------------------------ append
// One decode step appends one (k, v) pair per KV head and one query per query
// head (Sec. 2, periodic eviction; the last W queries are cached for Eq. (2)).
__global__ void append_kernel(const AppendParams p) {
    const int64_t nq = static_cast<int64_t>(p.n) * p.b * p.Hq * kVecPerRow;
    const int64_t nk = static_cast<int64_t>(p.n) * p.b * p.Hkv * kVecPerRow;
    const int64_t npos = static_cast<int64_t>(p.n) * p.b * p.Hkv;
    const int64_t total = nq + 2 * nk + npos;
    const int first_q = p.n > p.W ? p.n - p.W : 0;  // only the last W queries survive in the ring
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < total;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        if (i < nq) {
            const int seg = static_cast<int>(i % kVecPerRow);
            const int64_t r = i / kVecPerRow;  // (t, s, hq)
            const int hq = static_cast<int>(r % p.Hq);
            const int64_t ts = r / p.Hq;
            const int s = static_cast<int>(ts % p.b);
            const int t = static_cast<int>(ts / p.b);
            if (t < first_q) continue;
            const int slot = static_cast<int>((p.q_seen + t) % p.W);
            p.qwin[((static_cast<int64_t>(s) * p.Hq + hq) * p.W + slot) * kVecPerRow + seg] = p.q[i];
        } else if (i < nq + 2 * nk) {
            const int64_t j = i - nq;
            const bool is_v = j >= nk;
            const int64_t jj = is_v ? j - nk : j;
            const int seg = static_cast<int>(jj % kVecPerRow);
            const int64_t r = jj / kVecPerRow;  // (t, s, h)
            const int h = static_cast<int>(r % p.Hkv);
            const int64_t ts = r / p.Hkv;
            const int s = static_cast<int>(ts % p.b);
            const int t = static_cast<int>(ts / p.b);
            const int64_t dst = ((static_cast<int64_t>(s) * p.Hkv + h) * p.N + p.fill + t) * kVecPerRow + seg;
            if (is_v)
                p.vc[dst] = p.v[jj];
            else
                p.kc[dst] = p.k[jj];
        } else {
            const int64_t r = i - nq - 2 * nk;  // (t, s, h)
            const int h = static_cast<int>(r % p.Hkv);
            const int64_t ts = r / p.Hkv;
            const int s = static_cast<int>(ts % p.b);
            const int t = static_cast<int>(ts / p.b);
            p.pos[(static_cast<int64_t>(s) * p.Hkv + h) * p.N + p.fill + t] = static_cast<int32_t>(p.next_pos + t);
        }
    }
}

// ------------------------------------------------------------------ value magnitude
// Range(v) = max_j v_j - min_j v_j (Eq. (5)); L2 and Var (App. A).  A half
// warp reads one 256-byte row with one 16-byte load per lane.
__device__ __forceinline__ void bf16x8_to_f32(const uint4 u, float (&f)[8]) {
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        f[2 * i] = __uint_as_float(w[i] << 16);
        f[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
    }
}

__global__ void value_score_kernel(const ValueParams p) {
    const int warp = threadIdx.x >> 5;
    const int hsel = (threadIdx.x >> 4) & 1;
    const int l = threadIdx.x & 15;
    const int halves = blockDim.x >> 4;
    const int64_t rows = static_cast<int64_t>(p.units) * p.K;
    // the loop bound is uniform per warp so every shuffle sees all 32 lanes
    for (int64_t r0 = static_cast<int64_t>(blockIdx.x) * halves + 2 * warp; r0 < rows;
         r0 += static_cast<int64_t>(gridDim.x) * halves) {
        const int64_t r = r0 + hsel;
        const bool valid = r < rows;
        const int unit = valid ? static_cast<int>(r / p.K) : 0;
        const int slot = valid ? static_cast<int>(r - static_cast<int64_t>(unit) * p.K) : 0;
        const int64_t row = static_cast<int64_t>(unit) * p.N + slot;
        float f[8];
        bf16x8_to_f32(valid ? __ldg(&p.vc[row * kVecPerRow + l]) : make_uint4(0, 0, 0, 0), f);
        float out;
        if (p.kind == 0) {
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
            out = mx - mn;
        } else if (p.kind == 1) {
            float ss = 0.f;
#pragma unroll
            for (int i = 0; i < 8; ++i) ss = fmaf(f[i], f[i], ss);
#pragma unroll
            for (int o = 8; o >= 1; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
            out = sqrtf(ss);
        } else {
            float sm = 0.f;
#pragma unroll
            for (int i = 0; i < 8; ++i) sm += f[i];
#pragma unroll
            for (int o = 8; o >= 1; o >>= 1) sm += __shfl_xor_sync(0xffffffffu, sm, o);
            const float mu = sm * (1.0f / kHeadDim);
            float ss = 0.f;
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const float dlt = f[i] - mu;
                ss = fmaf(dlt, dlt, ss);
            }
#pragma unroll
            for (int o = 8; o >= 1; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
            out = ss * (1.0f / kHeadDim);
        }
        if (valid && l == 0) p.out[row] = out;
    }
}

// ------------------------------------------------------------------ selection
constexpr int kSelThreads = 512;
constexpr int kSelWarps = kSelThreads / 32;
constexpr uint8_t kFlagValue = 1;
constexpr uint8_t kFlagSampled = 2;

struct SelShared {
    uint32_t hist[256];
    int warp_tot[kSelWarps];
    uint32_t bcast[4];
};

// Exclusive prefix over threads of `v` in thread order; returns the offset and
// writes the block total to *total.  Every thread must call it.
__device__ __forceinline__ int block_exclusive_scan(int v, SelShared& sh, int* total) {
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
        int w = lane < kSelWarps ? sh.warp_tot[lane] : 0;
        int inc = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, inc, o);
            if (lane >= o) inc += y;
        }
        if (lane < kSelWarps) sh.warp_tot[lane] = inc - w;  // exclusive warp offsets
        if (lane == kSelWarps - 1) sh.bcast[3] = static_cast<uint32_t>(inc);
    }
    __syncthreads();
    const int off = sh.warp_tot[warp] + x - v;
    *total = static_cast<int>(sh.bcast[3]);
    __syncthreads();
    return off;
}

// Marks with `flag` the k largest values of ord[0..n) (ties to the lower
// index), by an MSB-first radix select on 8-bit digits followed by a
// slot-ordered rank of the elements equal to the threshold.  Each thread owns
// the contiguous slots [seg_lo, seg_hi).
__device__ void radix_top_k(const uint32_t* ord, int n, int k, uint8_t* flags, uint8_t flag, int seg_lo,
                            int seg_hi, SelShared& sh) {
    if (k <= 0) return;
    const int tid = threadIdx.x;
    uint32_t prefix = 0, mask = 0;
    int remain = k;
    for (int shift = 24; shift >= 0; shift -= 8) {
        for (int i = tid; i < 256; i += kSelThreads) sh.hist[i] = 0;
        __syncthreads();
        for (int i = tid; i < n; i += kSelThreads) {
            const uint32_t x = ord[i];
            if ((x & mask) == prefix) atomicAdd(&sh.hist[(x >> shift) & 0xFFu], 1u);
        }
        __syncthreads();
        if (tid < 32) {
            const int lane = tid;
            uint32_t c[8];
            uint32_t tot = 0;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                c[j] = sh.hist[8 * lane + j];
                tot += c[j];
            }
            uint32_t suf = tot;  // inclusive suffix sum over lanes >= lane
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const uint32_t y = __shfl_down_sync(0xffffffffu, suf, o);
                if (lane + o < 32) suf += y;
            }
            uint32_t above = suf - tot;
#pragma unroll
            for (int j = 7; j >= 0; --j) {
                if (above < static_cast<uint32_t>(remain) && above + c[j] >= static_cast<uint32_t>(remain)) {
                    sh.bcast[0] = static_cast<uint32_t>(8 * lane + j);
                    sh.bcast[1] = above;
                }
                above += c[j];
            }
        }
        __syncthreads();
        const uint32_t digit = sh.bcast[0];
        remain -= static_cast<int>(sh.bcast[1]);
        prefix |= digit << shift;
        mask |= 0xFFu << shift;
        __syncthreads();
    }
    const uint32_t thr = prefix;
    int eq = 0;
    for (int i = seg_lo; i < seg_hi; ++i) eq += ord[i] == thr;
    int total;
    int rank = block_exclusive_scan(eq, sh, &total);
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

// One CTA per unit.  AttnV (Sec. 3.2): R_B = slots >= K; R_V = N_v largest
// value magnitudes among slots < K; the m = K - N_v - B remaining slots are
// the m largest keys pooled_i / E_i over C = [K] \ R_V, E_i = -ln u_i, which is
// weighted sampling without replacement proportional to the pooled score
// (exponential race); with stochastic = 0 the key is the pooled score itself
// (Sec. 4.1).  DKV: the K - B largest leverage products.  Writes the ascending
// list of kept slots.
__global__ void __launch_bounds__(kSelThreads, 1) select_kernel(const SelectParams p) {
    extern __shared__ __align__(16) uint8_t smem_raw[];
    __shared__ SelShared sh;
    const int N = p.N, K = p.K;
    float* a_s = reinterpret_cast<float*>(smem_raw);              // [N] window score (AttnV)
    uint32_t* ord = reinterpret_cast<uint32_t*>(a_s + N);         // [K] orderable keys
    uint8_t* flags = reinterpret_cast<uint8_t*>(ord + K);         // [N]
    const int unit = blockIdx.x;
    const int tid = threadIdx.x;
    const int64_t base = static_cast<int64_t>(unit) * N;
    const int seg = (N + kSelThreads - 1) / kSelThreads;
    const int seg_lo = min(N, tid * seg);
    const int seg_hi = min(N, seg_lo + seg);
    const int kseg_lo = min(K, seg_lo);
    const int kseg_hi = min(K, seg_hi);

    for (int i = tid; i < N; i += kSelThreads) flags[i] = 0;
    if (p.variant == 0) {
        for (int i = tid; i < N; i += kSelThreads) a_s[i] = p.attn[base + i];
        for (int i = tid; i < K; i += kSelThreads) ord[i] = __float_as_uint(p.vscore[base + i]) + 1u;
        __syncthreads();
        radix_top_k(ord, K, p.n_v, flags, kFlagValue, kseg_lo, kseg_hi, sh);
        // keys over the candidates C
        const int h = p.pool / 2;
        const float inv_pool = 1.0f / static_cast<float>(p.pool);
        const uint32_t c2 = static_cast<uint32_t>(p.layer) | (kTagSelect << 24);
        for (int i = tid; i < N; i += kSelThreads) {
            float sum = 0.f;
            const int lo = max(0, i - h), hi = min(N - 1, i + h);
            for (int j = lo; j <= hi; ++j) sum += a_s[j];
            const float pooled = sum * inv_pool;
            if (p.pooled_dbg) p.pooled_dbg[base + i] = pooled;
            if (i >= K) continue;
            float key = -1.f;
            if (flags[i] & kFlagValue) {
                ord[i] = 0u;
            } else {
                key = pooled;
                if (p.stochastic) {
                    const Philox4 w = philox4x32_10(
                        Philox4{static_cast<uint32_t>(p.pos[base + i]), static_cast<uint32_t>(p.rnd), c2,
                                static_cast<uint32_t>(unit)},
                        p.seed_lo, p.seed_hi);
                    key = pooled / (-logf(open_uniform(w.x)));
                }
                ord[i] = __float_as_uint(key) + 1u;
            }
            if (p.key_dbg) p.key_dbg[base + i] = key;
        }
        __syncthreads();
        radix_top_k(ord, K, p.m, flags, kFlagSampled, kseg_lo, kseg_hi, sh);
    } else {
        for (int i = tid; i < K; i += kSelThreads) {
            const float s = p.vscore[base + i];
            ord[i] = __float_as_uint(s) + 1u;
            if (p.key_dbg) p.key_dbg[base + i] = s;
        }
        __syncthreads();
        radix_top_k(ord, K, p.m, flags, kFlagSampled, kseg_lo, kseg_hi, sh);
    }
    // keep = R_B u R_V u sampled; ascending list of kept slots
    int cnt = 0;
    for (int i = seg_lo; i < seg_hi; ++i) cnt += (i >= K) || flags[i];
    int total;
    int dst = block_exclusive_scan(cnt, sh, &total);
    for (int i = seg_lo; i < seg_hi; ++i) {
        const bool keep = (i >= K) || flags[i];
        if (keep) {
            if (dst < K) p.src[static_cast<int64_t>(unit) * K + dst] = i;
            ++dst;
        }
        if (p.keep_dbg) p.keep_dbg[base + i] = keep ? 1 : 0;
        if (p.key_dbg && i >= K) p.key_dbg[base + i] = -1.f;
    }
    if (tid == 0 && total != K) record_error(p.err, kErrSelectCount);
}

// ------------------------------------------------------------------ compaction
// Stable in-place gather of the kept rows into slots 0..K-1 (Sec. 2: the
// cache is restored to K pairs).  New slot j takes old slot src[j] >= j, so a
// CTA that walks destination chunks in ascending order, loading a chunk's
// sources before any of its stores (barrier) and never storing past the
// chunk, never overwrites a row it still has to read.  Each CTA owns one
// 128-byte column half of K or V, so CTAs never touch the same bytes.
constexpr int kCompactThreads = 256;
constexpr int kCompactRowsPerChunk = 256;

__global__ void __launch_bounds__(kCompactThreads) compact_kernel(const CompactParams p) {
    const int unit = blockIdx.x;
    const int part = blockIdx.y;  // 0, 1: K halves; 2, 3: V halves
    uint4* base = (part < 2 ? p.kc : p.vc) + static_cast<int64_t>(unit) * p.N * kVecPerRow;
    const int seg = (part & 1) * 8 + (threadIdx.x & 7);
    const int rsub = threadIdx.x >> 3;  // 0..31
    const bool do_pos = (part == 0) && ((threadIdx.x & 7) == 0);
    int32_t* pos = p.pos + static_cast<int64_t>(unit) * p.N;
    const int32_t* src = p.src + static_cast<int64_t>(unit) * p.K;
    const int n_chunks = (p.K + kCompactRowsPerChunk - 1) / kCompactRowsPerChunk;

    uint4 cur[8], nxt[8];
    int cs[8], ns[8];
    int32_t cp[8], np[8];
    auto load = [&](int c, uint4 (&d)[8], int (&sidx)[8], int32_t (&pv)[8]) {
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            const int j = c * kCompactRowsPerChunk + rsub + 32 * i;
            sidx[i] = -1;
            if (j < p.K) {
                const int s = src[j];
                if (s != j) {
                    sidx[i] = s;
                    d[i] = base[static_cast<int64_t>(s) * kVecPerRow + seg];
                    if (do_pos) pv[i] = pos[s];
                }
            }
        }
    };
    auto store = [&](int c, const uint4 (&d)[8], const int (&sidx)[8], const int32_t (&pv)[8]) {
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            const int j = c * kCompactRowsPerChunk + rsub + 32 * i;
            if (sidx[i] >= 0) {
                base[static_cast<int64_t>(j) * kVecPerRow + seg] = d[i];
                if (do_pos) pos[j] = pv[i];
            }
        }
    };
    if (n_chunks > 0) load(0, cur, cs, cp);
    __syncthreads();
    for (int c = 0; c < n_chunks; ++c) {
        if (c + 1 < n_chunks) load(c + 1, nxt, ns, np);
        store(c, cur, cs, cp);
        __syncthreads();
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            cur[i] = nxt[i];
            cs[i] = ns[i];
            cp[i] = np[i];
        }
    }
    if (part == 0) {
        for (int j = p.K + threadIdx.x; j < p.N; j += kCompactThreads) pos[j] = -1;
    }
}

}  // namespace

cudaError_t launch_append(const AppendParams& p, cudaStream_t s) {
    const int64_t total = static_cast<int64_t>(p.n) * p.b * (p.Hq + 2 * p.Hkv) * kVecPerRow +
                          static_cast<int64_t>(p.n) * p.b * p.Hkv;
    const int threads = 256;
    const int64_t blocks = (total + threads - 1) / threads;
    append_kernel<<<static_cast<unsigned>(blocks < 65535 ? blocks : 65535), threads, 0, s>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_value_score(const ValueParams& p, int num_sms, cudaStream_t s) {
    const int threads = 256;
    const int64_t rows = static_cast<int64_t>(p.units) * p.K;
    int64_t blocks = (rows + (threads / 16) - 1) / (threads / 16);
    const int64_t cap = static_cast<int64_t>(num_sms) * 8;
    if (blocks > cap) blocks = cap;
    value_score_kernel<<<static_cast<unsigned>(blocks), threads, 0, s>>>(p);
    return cudaGetLastError();
}

size_t select_smem_bytes(int N, int K) { return static_cast<size_t>(N) * 4 + static_cast<size_t>(K) * 4 + N + 16; }

cudaError_t select_set_attributes(size_t smem_bytes) {
    return cudaFuncSetAttribute(select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                static_cast<int>(smem_bytes));
}

cudaError_t launch_select(const SelectParams& p, int units, size_t smem_bytes, cudaStream_t s) {
    select_kernel<<<static_cast<unsigned>(units), kSelThreads, smem_bytes, s>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_compact(const CompactParams& p, int units, cudaStream_t s) {
    compact_kernel<<<dim3(static_cast<unsigned>(units), 4), kCompactThreads, 0, s>>>(p);
    return cudaGetLastError();
}

}  // namespace vase
