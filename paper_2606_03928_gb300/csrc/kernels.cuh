// Kernel parameter blocks, launch helpers and the device-side Philox of the
// VaSE eviction step.  Host orchestration lives in api.cu.
#pragma once

#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

namespace vase {

// Error sites recorded in the device error word (low 16 bits).
enum ErrSite : uint32_t {
    kErrScoreQ = 1,
    kErrScoreKFull = 2,
    kErrScoreKEmpty = 3,
    kErrScoreTFull = 4,
    kErrScoreTEmpty = 5,
    kErrScoreDrain = 6,
    kErrSelectCount = 16,
    kErrCompactFull = 17,
    kErrDkvTFull = 32,
    kErrDkvKFull = 33,
    kErrDkvKEmpty = 34,
    kErrDkvTEmpty = 35,
    kErrDkvDrain = 36,
    kErrDecodeFull = 48,
    kErrDecodeEmpty = 49,
    kErrDecodeDrain = 50,
    kErrDecodeMask = 51,
    kErrSmallQ = 64,
    kErrSmallKFull = 65,
    kErrSmallKFree = 66,
    kErrSmallDone = 67,
    kErrStoreOverflow = 80,  // VASE_SITE_STORE_OVERFLOW: an append would overflow the ring after an eviction
    kErrStoreState = 81,     // VASE_SITE_STORE_STATE: ring state or masks out of range (a store not written here)
};

constexpr int kTileTokens = 128;   // tokens per MMA tile (M)
constexpr int kHeadDim = 128;      // d
constexpr int kRowBytes = 256;     // d * sizeof(bf16)
constexpr int kVecPerRow = 16;     // 16-byte vectors per row
constexpr int kDecodeTileRows = 64;   // rows per TMA box of the tensor-core decode attention
constexpr int kDecodeMaxCluster = 8;  // CTAs that split one unit's slots (one thread-block cluster)

// ------------------------------------------------------------------ Philox4x32-10
// Salmon, Moraes, Dror, Shaw, "Parallel random numbers: as easy as 1, 2, 3" (SC'11):
// ten rounds of two 32x32->64-bit multiplies with a Weyl-sequence key schedule.
struct Philox4 {
    uint32_t x, y, z, w;
};

__device__ __forceinline__ Philox4 philox4x32_10(Philox4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
    for (int i = 0; i < 10; ++i) {
        const uint32_t hi0 = __umulhi(0xD2511F53u, c.x);
        const uint32_t lo0 = 0xD2511F53u * c.x;
        const uint32_t hi1 = __umulhi(0xCD9E8D57u, c.z);
        const uint32_t lo1 = 0xCD9E8D57u * c.z;
        c = Philox4{hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0};
        k0 += 0x9E3779B9u;
        k1 += 0xBB67AE85u;
    }
    return c;
}

// u = (2 * (x >> 9) + 1) * 2^-24: strictly inside (0, 1) and exact in fp32.
__device__ __forceinline__ float open_uniform(uint32_t x) {
    return static_cast<float>(2u * (x >> 9) + 1u) * 5.9604644775390625e-08f;
}

constexpr uint32_t kTagSelect = 0u;
constexpr uint32_t kTagDkv = 1u;
constexpr uint32_t kTagReserve = 2u;

// ------------------------------------------------------------------ parameter blocks

// The layers one launch works on: slot z = blockIdx.z (or .y) handles model layer layer[z],
// whose next eviction is round rnd[z].  Workspace arrays are indexed by slot.
constexpr int kMaxLayerBatch = 64;
struct LayerBatch {
    int32_t n;
    int32_t layer[kMaxLayerBatch];
    int32_t rnd[kMaxLayerBatch];
};

struct AppendParams {
    const uint4* q;   // [slot][n][b][Hq][16], layer slots q_stride apart
    const uint4* k;   // [slot][n][b][Hkv][16], layer slots kv_stride apart
    const uint4* v;
    int64_t q_stride, kv_stride;  // 16-byte vectors between consecutive layer slots' inputs
    uint4* qwin;      // base of [L][b][Hq][W][16]
    uint4* kc;        // base of [L][b][Hkv][N][16]
    uint4* vc;
    int32_t* pos;     // base of [L][b][Hkv][N]
    float* vmag;      // base of [L][b][Hkv][N]: value magnitude of each cached token
    int32_t n, b, Hq, Hkv, W, N, kind;
    int32_t steps_per_block;         // decode steps per block (set by launch_append)
    int32_t layer[kMaxLayerBatch];
    int32_t fill[kMaxLayerBatch];
    int64_t next_pos[kMaxLayerBatch];
    int32_t q_ring[kMaxLayerBatch];  // window-ring slot of the layer's next query (queries seen mod W)
};

struct ScoreAttnParams {
    LayerBatch batch;
    int32_t N;              // K + B slots per unit
    int32_t GW;             // window rows per unit (G * W)
    int32_t GWp;            // GW padded: a multiple of 32 up to 256, of 256 beyond
    int32_t NB;             // window rows per pass-B MMA (N of the MMA), <= 256
    int32_t n_rb;           // GWp / NB
    int32_t n_rbA;          // 128-row blocks of window rows in pass A
    int32_t rep;            // copies of the window rows across the 128 pass-A lanes (GWp in {32, 64})
    int32_t q_rows;         // window rows staged in shared memory (>= GWp)
    int32_t q_box;          // rows per TMA box of the window-query map
    int32_t n_tiles;        // ceil(N / 128)
    int32_t tiles_per_cta;  // T
    int32_t work;           // work items: batch.n layer slots x units (item w = slot * units + unit)
    int32_t groups;         // CTA groups (clusters) of the grid; group g takes items g, g + groups, ...
    int32_t q_bufs;         // window-row buffers: 2 when a group takes several items, else 1
    int32_t lead;           // pass-B tiles that open an interleaved phase before its first pass-A tile
    int32_t cluster;        // CTAs per unit
    int32_t stages;         // tile ring depth
    int32_t buf_cols;       // TMEM columns per accumulator buffer
    int32_t nbuf;           // accumulator buffers in TMEM (2 or 4)
    int32_t cgroups;        // consumer warpgroups (2, or 4 with one buffer and one row block each)
    int32_t units;          // units per layer
    int32_t tmem_cols;
    int32_t Hq, Hkv, W, G;
    int64_t layer_rows;     // cache rows per layer (units * N)
    int64_t q_layer_rows;   // window rows per layer (b * Hq * W)
    int32_t head_rows;      // 0: the score sums all G*W window rows; W: per query head, the largest head sum
    int32_t fold_rows;      // rows the score averages over: G*W (mean over the heads) or W (max over the heads)
    float scale_log2;       // log2(e) / sqrt(d)
    float inv_gw;           // 1 / (G * W)
    float* attn;            // [slot][n_rb][units][N] (one part per row block)
    uint32_t* err;
};

struct ValueParams {
    const uint4* vc;        // layer base of [units][N][16]
    float* out;             // layer base of [units][N]
    int32_t N, rows, units, kind;  // slots 0..rows-1 of every unit
};

struct DkvParams {
    LayerBatch batch;
    int32_t N, K, r, Hkv, fixed_g, units;
    int32_t shared_g;       // 1: one G per round for every layer and unit (counter without layer and unit)
    uint32_t seed_lo, seed_hi;
    int32_t n_tiles_k;      // ceil(K / 128)
    int32_t tiles_per_cta;
    int32_t stages;
    int64_t layer_rows;     // cache rows per layer
    float* out;             // [slot][units][N] leverage product, slots < K
    uint32_t* err;
};

struct SelectParams {
    LayerBatch batch;
    const float* attn;      // [slot][n_parts][units][N]: the window score is the sum of the parts
    const float* dkv;       // [slot][units][N] leverage products (DKV)
    float* vmag;            // base of [L][units][N]: value magnitudes (AttnV), compacted in place
    int32_t* pos;           // base of [L][units][N]; compacted in place with the kept list
    uint4* kc;              // base of [L][units][N][16]: K rows, gathered in place
    uint4* vc;              // V rows
    float* vscore_dbg;      // nullable, [slot][units][N]: the value magnitudes of this eviction
    int32_t* src;           // [slot][units][K]
    uint8_t* resv;          // nullable, [slot][units][store_resv_stride(K)]: 1 = new slot j is in R_V u R_B (store)
    float* pooled_dbg;      // nullable, [slot][units][N]
    float* key_dbg;         // nullable
    uint8_t* keep_dbg;      // nullable
    int32_t N, K, B, n_v, m, pool, variant, stochastic, Hkv, n_parts, units;
    int32_t staged;         // 1: every input array of the unit is copied to shared memory up front
    int32_t reserve_random; // 1: R_V = the N_v largest reservation uniforms (App. C ablation) instead of value magnitudes
    int32_t gqa_max;        // 1: the parts of the window score combine by max (GQA max-aggregation), 0: by sum
    uint32_t seed_lo, seed_hi;
    uint32_t* err;
};


// The fused eviction of small units (evict_small_kernel): one CTA per unit scores it, selects and gathers in one
// launch.  sel is the selection's block (one score part, staged); the rest describes the window score.
struct SmallEvictParams {
    SelectParams sel;
    int32_t GW, GWp;        // window rows per unit, padded to 32
    int32_t q_rows;         // window rows per TMA box of the window map and per shared-memory panel (>= GWp)
    int32_t n_tiles;        // ceil(N / 128): 128-token tiles, all resident in TMEM as S = K Q^T
    int32_t stages;         // K tile ring depth
    int32_t tmem_cols;
    int32_t Hq, W, G;
    int32_t head_rows;      // 0: mean over the G*W rows; W: per query head, the largest head mean (GQA max)
    int32_t fold_rows;      // G*W (mean) or W (max)
    int64_t layer_rows;     // cache rows per layer
    int64_t q_layer_rows;   // window rows per layer
    float scale_log2;       // log2(e) / sqrt(d)
    float* attn;            // [slot][units][N]: the window score, written for the debug view (nullable)
    int32_t append;         // 1: each CTA first appends its unit's rows of `ap` (the step's append, fused)
    AppendParams ap;        // the append of every layer slot of the launch (same slot order as sel.batch)
};
constexpr int kSmallThreads = 512;
constexpr int kSmallWarps = kSmallThreads / 32;
constexpr int kSmallMaxTiles = 8;

// Mixed-precision values of one layer: codes of the unreserved kept value rows, their (s, z), and the
// reserved-slot mask (bit t of word w: slot 32 w + t keeps its bf16 row).
struct QuantParams {
    const uint4* vc;        // layer base of [units][N][16]
    const float* vmag;      // layer base of [units][N]: value magnitudes
    uint8_t* codes;         // [units][K][row_bytes]
    float* qparams;         // [units][Kp][2]: (s, z)
    uint32_t* rmask;        // [units][mask_words]
    uint4* hp_rows;         // [units][hp_cap][16]: the reserved rows in slot order
    int32_t N, K, B, n_v, bits, row_bytes, Kp, mask_words, hp_cap;
};

struct DecodeParams {
    const uint4* q;         // [b][Hq][16]: the decode step's query rows (bf16)
    const uint4* kc;        // layer base of [units][N][16]
    const uint4* vc;
    float* out;             // [b][Hq][d] fp32
    int32_t N, fill, G, Hkv, units;
    int32_t n_chunks;       // ceil(fill / chunk) (set by launch_decode for the kernel it picks)
    int32_t cluster;        // CTAs per unit (cluster size, <= n_chunks); CTA r takes chunks r, r + cluster, ...
    int32_t row_base;       // first row of the layer in the K / V tensor maps (layer * units * N)
    float scale_log2;       // log2(e) / sqrt(d)
    uint32_t* err;
    // mixed-precision values (bits > 0): unreserved slots below Kq read from codes
    const uint8_t* codes;   // [units][Kq][code_row]
    const float* qparams;   // [units][Kp][2]
    const uint32_t* rmask;  // [units][mask_words]
    const uint4* hp_rows;   // [units][hp_cap][16]: the reserved rows below Kq in slot order
    // compressed value store: hp_rows is a ring, its entry i at row (head + i) mod hp_cap, head = ring_state[4 u]
    const int32_t* ring_state;  // nullable, [units][4]
    int32_t bits, code_row, Kq, Kp, mask_words, hp_cap;
};

// Bytes per unit of the selection's R_V u R_B flags (K rounded up to 16: whole 16-byte copies per unit).
__host__ __device__ inline int store_resv_stride(int K) { return (K + 15) & ~15; }

// Compressed value store of every layer (the mixed-precision cache Sec. 6 proposes): per layer and unit the
// b-bit codes and (s, z) of every slot, one bit per slot set where the value is held in bf16, the ring of H bf16
// rows holding those values in slot order, and (head, count) of the ring.
struct StoreParams {
    uint8_t* base;          // the store (the V buffer in this mode)
    int64_t layer_bytes;    // bytes per layer
    int64_t codes_off, qp_off, mask_off, ring_off, state_off;  // sub-arrays within a layer
    int32_t units, N, Np, mask_stride, mask_words, H, bits, code_row, K, b, Hkv;
    int32_t layer[kMaxLayerBatch];
    int32_t fill[kMaxLayerBatch];   // append: fill before the call
    int32_t round[kMaxLayerBatch];  // append: evictions so far
    // append: value rows [slot][n][b][Hkv][16], layer slots kv_stride vectors apart
    const uint4* v;
    int64_t kv_stride;
    int32_t n;
    int32_t big;            // 1: the ring may overflow (a first fill past H): the launch carries the overflow's memory
    int32_t n_v;            // N_v: the large-Range values the overflow keeps
    const float* vmag;      // base of [L][units][N]: value magnitudes (appended rows included)
    // eviction: the selection's kept list ([slot][units][K]) and R_V u R_B flags ([slot][units][resv stride])
    const int32_t* src;
    const uint8_t* resv;
    uint32_t* err;
};

// ------------------------------------------------------------------ launchers (return cudaError_t)

cudaError_t launch_append(const AppendParams& p, int n_layers, cudaStream_t s);
cudaError_t launch_value_score(const ValueParams& p, int num_sms, cudaStream_t s);
cudaError_t launch_score_attn(const CUtensorMap& kmap, const CUtensorMap& qmap, const ScoreAttnParams& p,
                              size_t smem_bytes, cudaStream_t s);
cudaError_t launch_dkv(const CUtensorMap& kmap, const CUtensorMap& vmap, const DkvParams& p, int units,
                       size_t smem_bytes, cudaStream_t s);
cudaError_t launch_select(const SelectParams& p, int units, size_t smem_bytes, int threads, cudaStream_t s);
size_t evict_small_smem_bytes(int N, int K, int GWp, int q_rows, int n_tiles, int stages);
cudaError_t evict_small_set_attributes(size_t smem_bytes);
cudaError_t launch_evict_small(const CUtensorMap& kmap, const CUtensorMap& qmap, const SmallEvictParams& p, int units,
                               size_t smem_bytes, cudaStream_t s);
cudaError_t launch_quantize(const QuantParams& p, int units, size_t smem_bytes, cudaStream_t s);
cudaError_t launch_store_append(const StoreParams& p, int n_layers, cudaStream_t s);
cudaError_t launch_store_evict(const StoreParams& p, int n_layers, cudaStream_t s);
size_t store_evict_smem_bytes(int K, int mask_stride);
size_t store_append_smem_bytes(int mask_stride, int H, int n, int K, bool big);
cudaError_t store_set_attributes(size_t evict_smem, size_t append_smem);
size_t quantize_smem_bytes(int K, int B);
cudaError_t quantize_set_attributes(size_t smem_bytes);
cudaError_t launch_decode(const CUtensorMap& kmap, const CUtensorMap& vmap, DecodeParams p, size_t smem_bytes,
                          int num_sms, cudaStream_t s);

size_t score_attn_smem_bytes(int q_rows, int q_bufs, int n_rbA, int GWp, int cluster, int stages, int groups);
size_t dkv_smem_bytes(int stages);
size_t select_smem_bytes(int N, int K, int n_parts, bool staged);
size_t select_static_smem_bytes();  // the selection kernel's static shared memory
cudaError_t score_attn_set_attributes(size_t smem_bytes, int cluster);
cudaError_t dkv_set_attributes(size_t smem_bytes);
cudaError_t select_set_attributes(size_t smem_bytes);
size_t decode_smem_bytes(int G, bool store);
cudaError_t decode_set_attributes(int G, size_t smem_bytes, bool store);
size_t decode_mixed_smem_bytes(int G, int bits, int mask_words);
cudaError_t decode_mixed_set_attributes();
cudaError_t launch_decode_mixed(DecodeParams p, int num_sms, cudaStream_t s);
constexpr int kDecodeMaxMaskWords = 544;  // reserved-slot mask words of a unit the mixed-precision decode holds

}  // namespace vase
