// Host side of the C ABI declared in include/vase.h: configuration checks,
// launch plans, TMA descriptors, per-layer counters and stream-ordered
// launches of the eviction-step kernels.
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <string>
#include <vector>

#include "kernels.cuh"
#include "vase.h"

using namespace vase;

namespace {

constexpr size_t kMaxDynSmem = 232448;  // 227 KB per block on sm_100-class GPUs
constexpr size_t kSmemPerSm = 233472;   // 228 KB per SM
constexpr size_t kSmemReservedPerBlock = 1024;  // the system's share of each block's shared memory
constexpr size_t kAlign = 256;

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }
int ceil_div(int a, int b) { return (a + b - 1) / b; }

struct Plan {
    int N, units, G, GW, GWp, NB, n_rb, n_rbA, rep, q_rows, q_box, buf_cols, nbuf, cgroups;
    int n_tiles, cluster, stages, stages_p, tmem_cols, n_v, m, num_sms;
    int cluster_for[kMaxLayerBatch + 1];  // CTAs per unit of the score kernel, by layers per launch
    bool persist_for[kMaxLayerBatch + 1]; // one CTA per SM taking several units (interleaved passes)
    size_t score_smem;
    int dkv_tiles_k, dkv_tiles_per_cta, dkv_stages;
    size_t dkv_smem;
    size_t select_smem;
    bool select_staged;
    int select_threads;
    // workspace
    int slots;  // layers one launch can batch
    size_t stride_attn, stride_un, stride_src;  // elements per workspace slot
    size_t off_err, off_attn, off_pooled, off_vscore, off_key, off_keep, off_src, off_staging, staging_bytes, ws_bytes;
    size_t decode_smem;                           // decode attention: shared memory per CTA
    // compressed value store (value_bits > 0): per layer the codes, (s, z), masks, ring and ring state of every unit
    bool store;
    int st_H, st_Np, st_mask_words, st_mask_stride, st_code_row;
    size_t st_codes_off, st_qp_off, st_mask_off, st_ring_off, st_state_off, st_layer_bytes, st_evict_smem;
    size_t st_append_smem;  // the append's shared memory when the ring may overflow (a first fill of N past H)
    size_t off_resv;  // workspace: [slot][units][K] R_V u R_B flags of the kept slots
    // fused eviction of small units (evict_small_kernel): usable when the unit's score matrix fits in TMEM
    bool small_ok;
    int small_tiles, small_stages, small_tmem_cols;
    size_t small_smem;
};

// Launch parameters of the window-score kernel for `nz` layers of `batch`.
ScoreAttnParams score_params(const Plan& P, const vase_config& c, const LayerBatch& batch, int nz, float* attn,
                             uint32_t* err);

// Reason of the last failed configuration check on this thread (vase_last_error(NULL)).
thread_local std::string g_config_error;

const char* check_config(const vase_config* c) {
    if (!c) return "null config";
    if (c->head_dim != 128) return "head_dim must be 128";
    if (c->budget_k < 1 || c->buffer_b < 1) return "budget_k and buffer_b must be >= 1";
    if (c->buffer_b > c->budget_k) return "buffer_b must not exceed budget_k (K - B candidates are kept)";
    if (c->num_q_heads < 1 || c->num_kv_heads < 1 || c->num_q_heads % c->num_kv_heads) return "num_q_heads must be a positive multiple of num_kv_heads";
    if (c->num_layers < 1 || c->batch < 1) return "num_layers and batch must be >= 1";
    if (c->window < 1) return "window must be >= 1";
    if (c->window > c->budget_k + c->buffer_b) return "window must not exceed K + B";
    if (c->variant != VASE_VARIANT_ATTNV && c->variant != VASE_VARIANT_DKV) return "unknown variant";
    if (c->value_score < 0 || c->value_score > 2) return "unknown value_score";
    if (c->pool_kernel < 1 || (c->pool_kernel % 2) == 0) return "pool_kernel must be odd and >= 1";
    if (c->dkv_rank < 1 || c->dkv_rank > 32) return "dkv_rank must be in 1..32";
    const int nv = c->n_v < 0 ? c->budget_k / 4 : c->n_v;
    if (c->variant == VASE_VARIANT_ATTNV && nv + c->buffer_b > c->budget_k) return "n_v + buffer_b must not exceed budget_k";
    if (c->reserve_kind != VASE_RESERVE_VALUE && c->reserve_kind != VASE_RESERVE_RANDOM) return "unknown reserve_kind";
    if (c->gqa_reduce != VASE_GQA_MEAN && c->gqa_reduce != VASE_GQA_MAX) return "unknown gqa_reduce";
    if (c->dkv_shared_g != 0 && c->dkv_shared_g != 1) return "dkv_shared_g must be 0 or 1";
    if (c->gqa_reduce == VASE_GQA_MAX && c->window % 4) return "GQA max-aggregation needs window % 4 == 0";
    if (c->value_bits != 0 && c->value_bits != 2 && c->value_bits != 4 && c->value_bits != 8)
        return "value_bits must be 0, 2, 4 or 8";
    if (c->value_bits != 0 && c->variant != VASE_VARIANT_ATTNV)
        return "the compressed value store needs the AttnV variant (DKV scores read every value each round)";
    return nullptr;
}

bool make_plan_impl(const vase_config* c, int num_sms, Plan* P, const char** why);

bool make_plan(const vase_config* c, int num_sms, Plan* P, const char** why) {
    *why = check_config(c);
    if (!*why) make_plan_impl(c, num_sms, P, why);
    g_config_error = *why ? *why : "";
    return *why == nullptr;
}

bool make_plan_impl(const vase_config* c, int num_sms, Plan* P, const char** why) {
    Plan& p = *P;
    p.num_sms = num_sms;
    p.N = c->budget_k + c->buffer_b;
    p.units = c->batch * c->num_kv_heads;
    p.G = c->num_q_heads / c->num_kv_heads;
    p.GW = p.G * c->window;
    if (p.GW > 512) {
        *why = "G * window must be <= 512";
        return false;
    }
    p.GWp = p.GW <= 256 ? (p.GW + 31) / 32 * 32 : (p.GW + 255) / 256 * 256;
    // Four consumer groups, one 128-column accumulator each: at up to 128 window rows (a tile is one item per
    // pass, taken by the groups in turn), and at 512 window rows, where each group owns one 128-row block in
    // both passes (pass B in four parts; GQA max then needs whole query heads per 128-row block).  Two groups
    // with two 256-column accumulators in between (measured: Qwen3-8B geometry 755 -> 678 us per eight layers,
    // Qwen3-1.7B 261 -> 255 us per 28 layers, Qwen3-32B 2400 -> 1920 us per eight layers).
    p.cgroups = p.GWp <= 128 || (p.GWp == 512 && (c->gqa_reduce != VASE_GQA_MAX || 128 % c->window == 0)) ? 4 : 2;
    p.NB = p.GWp < (p.cgroups == 4 ? 128 : 256) ? p.GWp : (p.cgroups == 4 ? 128 : 256);
    p.n_rb = p.GWp / p.NB;
    if (p.n_rb < 1 || p.n_rb * p.NB != p.GWp) {
        *why = "internal: the pass-B row blocks do not tile the window rows";
        return false;
    }
    if (c->gqa_reduce == VASE_GQA_MAX && p.n_rb > 1 && p.NB % c->window) {
        *why = "GQA max-aggregation with G * window > 256 needs window to divide 256";
        return false;
    }
    if (p.GWp <= 64) {  // replicate short windows across the 128 pass-A lanes
        p.rep = 128 / p.GWp;
        p.n_rbA = 1;
        p.q_rows = 128;
        p.q_box = p.GWp;
    } else {
        p.rep = 1;
        p.n_rbA = ceil_div(p.GWp, 128);
        p.q_rows = 128 * p.n_rbA;
        p.q_box = p.q_rows < 256 ? p.q_rows : 256;
    }
    p.buf_cols = p.NB > 128 ? p.NB : 128;
    p.nbuf = 512 / p.buf_cols >= 4 ? 4 : 2;
    p.n_tiles = ceil_div(p.N, kTileTokens);
    p.n_v = c->n_v < 0 ? c->budget_k / 4 : c->n_v;
    p.m = c->variant == VASE_VARIANT_ATTNV ? c->budget_k - p.n_v - c->buffer_b : c->budget_k - c->buffer_b;
    p.tmem_cols = 32;
    while (p.tmem_cols < p.nbuf * p.buf_cols) p.tmem_cols *= 2;

    // cluster size per number of layers in a launch: minimise waves x (tiles per CTA + 1)
    // among the sizes whose shared memory fits with two stages
    const int max_batch = c->num_layers < kMaxLayerBatch ? c->num_layers : kMaxLayerBatch;
    int c_max = 0;
    for (int nz = 1; nz <= kMaxLayerBatch; ++nz) {
        int best_c = 0;
        long best_cost = -1;
        for (int C = 1; C <= 16 && C <= p.n_tiles; ++C) {
            const int T = ceil_div(p.n_tiles, C);
            if (ceil_div(p.n_tiles, T) != C) continue;
            if (score_attn_smem_bytes(p.q_rows, 1, p.n_rbA, p.GWp, C, 2, p.cgroups) > kMaxDynSmem) continue;
            const long ctas = static_cast<long>(p.units) * C * nz;
            const long waves = (ctas + num_sms - 1) / num_sms;
            const long cost = waves * (T + 1);
            if (best_cost < 0 || cost < best_cost) {
                best_cost = cost;
                best_c = C;
            }
        }
        if (!best_c) {
            *why = "window rows do not fit in shared memory";
            return false;
        }
        p.cluster_for[nz] = best_c;
        if (nz <= max_batch && best_c > c_max) c_max = best_c;
    }
    // With at least one item per SM, one CTA per SM takes a strided list of units and overlaps the pass-B
    // sweep of each with the pass-A sweep of the next (measured faster than one cluster per unit from 152
    // items on: batch-1 launches of 288 units); this needs two window-row buffers.
    p.stages_p = 0;
    for (int s = 4; s >= 2; --s) {
        if (score_attn_smem_bytes(p.q_rows, 2, p.n_rbA, p.GWp, 1, s, p.cgroups) <= kMaxDynSmem) {
            p.stages_p = s;
            break;
        }
    }
    bool any_persist = false;
    c_max = 0;
    for (int nz = 1; nz <= kMaxLayerBatch; ++nz) {
        p.persist_for[nz] = p.stages_p > 0 && static_cast<long>(p.units) * nz >= num_sms;
        if (nz <= max_batch) {
            if (p.persist_for[nz]) any_persist = true;
            else if (p.cluster_for[nz] > c_max) c_max = p.cluster_for[nz];
        }
    }
    p.cluster = c_max > 0 ? c_max : 1;  // shared memory is sized for the largest cluster used
    p.stages = 0;
    for (int s = 6; s >= 2; --s) {
        if (score_attn_smem_bytes(p.q_rows, 1, p.n_rbA, p.GWp, p.cluster, s, p.cgroups) <= kMaxDynSmem) {
            p.stages = s;
            break;
        }
    }
    p.score_smem = score_attn_smem_bytes(p.q_rows, 1, p.n_rbA, p.GWp, p.cluster, p.stages, p.cgroups);
    if (any_persist) {
        const size_t sp = score_attn_smem_bytes(p.q_rows, 2, p.n_rbA, p.GWp, 1, p.stages_p, p.cgroups);
        if (sp > p.score_smem) p.score_smem = sp;
    }
    if (p.tmem_cols > 256 && p.score_smem < 120 * 1024) p.score_smem = 120 * 1024;  // one CTA per SM owns TMEM

    p.dkv_tiles_k = ceil_div(c->budget_k, kTileTokens);
    {
        int best = 1;
        long bc = -1;
        for (int C = 1; C <= p.dkv_tiles_k && C <= 64; ++C) {
            const int T = ceil_div(p.dkv_tiles_k, C);
            if (ceil_div(p.dkv_tiles_k, T) != C) continue;
            const long ctas = static_cast<long>(p.units) * C;
            const long waves = (ctas + num_sms - 1) / num_sms;
            const long cost = waves * (T + 2);
            if (bc < 0 || cost < bc) {
                bc = cost;
                best = C;
            }
        }
        p.dkv_tiles_per_cta = ceil_div(p.dkv_tiles_k, best);
    }
    p.dkv_stages = 3;
    p.dkv_smem = dkv_smem_bytes(p.dkv_stages);
    {
        const int n_parts = c->variant == VASE_VARIANT_ATTNV ? p.n_rb : 1;
        // Staged (every input of the unit copied to shared memory at once), unless that leaves one CTA per SM
        // and reading the inputs from global memory lets two or more share it, so that one CTA's gather runs
        // under another's selection (measured: Qwen3-32B geometry 1807 -> 1675 us per eight layers; at two
        // staged CTAs per SM, Qwen3-8B, four unstaged ones were slower).
        auto per_sm = [](size_t smem) {
            return kSmemPerSm / (smem + select_static_smem_bytes() + kSmemReservedPerBlock);
        };
        const size_t s_staged = select_smem_bytes(p.N, c->budget_k, n_parts, true);
        const size_t s_plain = select_smem_bytes(p.N, c->budget_k, n_parts, false);
        p.select_staged = s_staged <= kMaxDynSmem - 9216 && !(per_sm(s_staged) < 2 && per_sm(s_plain) >= 2);
        p.select_smem = select_smem_bytes(p.N, c->budget_k, n_parts, p.select_staged);
        // threads per CTA: 1024 when one CTA holds an SM, 512 for two, 256 (four) otherwise
        const size_t ctas = per_sm(p.select_smem);
        p.select_threads = ctas <= 1 ? 1024 : (ctas == 2 ? 512 : 256);
    }
    if (p.select_smem > kMaxDynSmem - 9216) {
        *why = "K + B too large for the single-CTA selection (its shared memory holds about 17k slots)";
        return false;
    }

    // workspace: one slot of per-eviction arrays per layer a launch can batch
    p.slots = c->num_layers < kMaxLayerBatch ? c->num_layers : kMaxLayerBatch;
    const size_t un = static_cast<size_t>(p.units) * p.N;
    p.stride_attn = un * p.n_rb;
    p.stride_un = un;
    p.stride_src = static_cast<size_t>(p.units) * c->budget_k;
    const size_t Z = static_cast<size_t>(p.slots);
    size_t o = 0;
    p.off_err = o;
    o += kAlign;
    p.off_attn = o;
    o = align_up(o + Z * p.stride_attn * 4, kAlign);  // one part per pass-B row block
    p.off_pooled = o;
    o = align_up(o + Z * un * 4, kAlign);
    p.off_vscore = o;
    o = align_up(o + Z * un * 4, kAlign);
    p.off_key = o;
    o = align_up(o + Z * un * 4, kAlign);
    p.off_keep = o;
    o = align_up(o + Z * un, kAlign);
    p.off_src = o;
    o = align_up(o + Z * p.stride_src * 4, kAlign);
    p.off_resv = o;
    o = align_up(o + Z * p.units * static_cast<size_t>(store_resv_stride(c->budget_k)), kAlign);
    p.off_staging = o;
    p.staging_bytes = static_cast<size_t>(c->buffer_b) * c->batch * (c->num_q_heads + 2 * c->num_kv_heads) * kRowBytes;
    o = align_up(o + p.staging_bytes, kAlign);
    p.decode_smem = decode_smem_bytes(p.G, c->value_bits != 0);
    p.ws_bytes = o;
    // fused small-unit eviction: AttnV, at most 128 window rows, every 128-token tile's S = K Q^T resident in TMEM
    p.small_tiles = p.n_tiles;
    p.small_stages = p.n_tiles < 4 ? p.n_tiles : 4;
    p.small_tmem_cols = 32;
    while (p.small_tmem_cols < p.n_tiles * p.GWp) p.small_tmem_cols *= 2;
    p.small_smem = evict_small_smem_bytes(p.N, c->budget_k, p.GWp, p.q_box, p.n_tiles, p.small_stages);
    p.store = c->value_bits != 0;
    p.small_ok = c->variant == VASE_VARIANT_ATTNV && p.GWp <= 128 && p.n_tiles <= kSmallMaxTiles &&
                 p.n_tiles * p.GWp <= 512 && p.q_box >= p.GWp && p.small_smem <= kMaxDynSmem && !p.store;
    // compressed value store: the reserved ring holds R_V u R_B after an eviction and the B values appended
    // before the next one
    p.st_H = p.n_v + 2 * c->buffer_b;
    p.st_Np = (p.N + 1) & ~1;
    p.st_mask_words = ceil_div(p.N, 32);
    p.st_mask_stride = (p.st_mask_words + 3) & ~3;
    p.st_code_row = c->value_bits ? kHeadDim * c->value_bits / 8 : 0;
    {
        const size_t u = static_cast<size_t>(p.units);
        size_t so = 0;
        p.st_codes_off = so;
        so = align_up(so + u * p.N * p.st_code_row, kAlign);
        p.st_qp_off = so;
        so = align_up(so + u * p.st_Np * 8, kAlign);
        p.st_mask_off = so;
        so = align_up(so + u * p.st_mask_stride * 4, kAlign);
        p.st_ring_off = so;
        so = align_up(so + u * p.st_H * kRowBytes, kAlign);
        p.st_state_off = so;
        so = align_up(so + u * 16, kAlign);
        p.st_layer_bytes = so;
    }
    p.st_evict_smem = store_evict_smem_bytes(c->budget_k, p.st_mask_stride);
    p.st_append_smem = store_append_smem_bytes(p.st_mask_stride, p.st_H, p.N, c->budget_k, true);
    if (p.store && (p.st_evict_smem > kMaxDynSmem || p.st_append_smem > kMaxDynSmem ||
                    p.st_mask_words > kDecodeMaxMaskWords)) {
        *why = "K + B too large for the compressed value store";
        return false;
    }
    return true;
}

ScoreAttnParams score_params(const Plan& P, const vase_config& c, const LayerBatch& batch, int nz, float* attn,
                             uint32_t* err) {
    ScoreAttnParams sp{};
    sp.batch = batch;
    sp.N = P.N;
    sp.GW = P.GW;
    sp.GWp = P.GWp;
    sp.NB = P.NB;
    sp.n_rb = P.n_rb;
    sp.n_rbA = P.n_rbA;
    sp.rep = P.rep;
    sp.q_rows = P.q_rows;
    sp.q_box = P.q_box;
    sp.n_tiles = P.n_tiles;
    sp.work = P.units * nz;
    if (P.persist_for[nz]) {
        sp.cluster = 1;
        sp.groups = P.num_sms < sp.work ? P.num_sms : sp.work;
        sp.q_bufs = 2;
        sp.stages = P.stages_p;
    } else {
        sp.cluster = P.cluster_for[nz];
        sp.groups = sp.work;
        sp.q_bufs = 1;
        sp.stages = P.stages;
    }
    sp.lead = sp.stages;
    sp.tiles_per_cta = ceil_div(P.n_tiles, sp.cluster);
    sp.buf_cols = P.buf_cols;
    sp.nbuf = P.nbuf;
    sp.cgroups = P.cgroups;
    sp.units = P.units;
    sp.tmem_cols = P.tmem_cols;
    sp.Hq = c.num_q_heads;
    sp.Hkv = c.num_kv_heads;
    sp.W = c.window;
    sp.G = P.G;
    sp.layer_rows = static_cast<int64_t>(P.units) * P.N;
    sp.q_layer_rows = static_cast<int64_t>(c.batch) * c.num_q_heads * c.window;
    sp.scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(kHeadDim));
    sp.inv_gw = 1.0f / static_cast<float>(P.GW);
    sp.head_rows = c.gqa_reduce == VASE_GQA_MAX ? c.window : 0;
    sp.fold_rows = c.gqa_reduce == VASE_GQA_MAX ? c.window : P.GW;
    sp.attn = attn;
    sp.err = err;
    return sp;
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

}  // namespace

struct vase_ctx {
    vase_config cfg;
    vase_buffers bufs;
    Plan plan;
    int device = 0;
    int num_sms = 0;
    CUtensorMap kmap, vmap, qmap;
    CUtensorMap kmap_dec, vmap_dec;  // 64-row boxes for the decode attention
    std::vector<vase_layer_state> layers;
    std::vector<int32_t> quant_round, quant_bits;  // per layer: round and bits of the last vase_quantize_values
    std::vector<int32_t> last_batch;  // layers of the most recent eviction launch, by workspace slot
    int64_t launches = 0;
    std::string last_error;
    uint8_t* ws = nullptr;
    // host-side kernel timing (vase_profile_enable)
    struct EventPair {
        cudaEvent_t start, end;
        int kind;
    };
    std::vector<EventPair> events;
    size_t events_used = 0;
    bool profiling = false;
    // host-input pipeline (vase_stage_host_inputs / vase_append_all_staged / vase_read_positions_all)
    struct Staged {
        cudaEvent_t copied = nullptr;    // the inputs of this half have landed
        cudaEvent_t consumed = nullptr;  // the append that read this half has run
        bool consumed_pending = false;   // `consumed` was recorded and a later copy into the half must wait for it
        const uint8_t* base = nullptr;   // device address of the half
        int32_t n_tokens = 0, w_q = 0;   // tokens per layer, query rows kept per layer
        int64_t block = 0;               // bytes of one layer's [query tail | k | v] block
    };
    Staged staged[2];
    int staged_next = 0;      // half the next vase_stage_host_inputs fills
    int staged_count = 0;     // staged steps not yet appended (0..2)
    cudaEvent_t evicted = nullptr;    // recorded on the compute stream before a positions read-back
    cudaEvent_t read_done = nullptr;  // the last positions read-back has run; the next eviction waits for it
    bool read_pending = false;
    ~vase_ctx() {
        for (auto& e : events) {
            cudaEventDestroy(e.start);
            cudaEventDestroy(e.end);
        }
        for (auto& h : staged) {
            if (h.copied) cudaEventDestroy(h.copied);
            if (h.consumed) cudaEventDestroy(h.consumed);
        }
        if (evicted) cudaEventDestroy(evicted);
        if (read_done) cudaEventDestroy(read_done);
    }
};

namespace {

int fail(vase_ctx* ctx, int code, const std::string& msg) {
    if (ctx) ctx->last_error = msg;
    return code;
}

int cuda_fail(vase_ctx* ctx, cudaError_t e, const char* what) {
    return fail(ctx, VASE_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
}

// Runs `launch` (which enqueues one kernel on s), bracketed by CUDA events when profiling.
template <class F>
cudaError_t timed_launch(vase_ctx* ctx, int kind, cudaStream_t s, F&& launch) {
    if (!ctx->profiling) return launch();
    if (ctx->events_used == ctx->events.size()) {
        vase_ctx::EventPair e;
        if (cudaEventCreate(&e.start) != cudaSuccess) return cudaGetLastError();
        if (cudaEventCreate(&e.end) != cudaSuccess) {
            cudaEventDestroy(e.start);
            return cudaGetLastError();
        }
        ctx->events.push_back(e);
    }
    vase_ctx::EventPair& e = ctx->events[ctx->events_used++];
    e.kind = kind;
    cudaError_t r = cudaEventRecord(e.start, s);
    if (r != cudaSuccess) return r;
    r = launch();
    if (r != cudaSuccess) return r;
    return cudaEventRecord(e.end, s);
}

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

bool encode_rows(EncodeTiledFn enc, CUtensorMap* map, void* base, uint64_t rows, uint32_t box_rows) {
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(kHeadDim), static_cast<cuuint64_t>(rows)};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(kRowBytes)};
    cuuint32_t box[2] = {64, box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

bool check_layer(vase_ctx* ctx, int32_t layer) { return ctx && layer >= 0 && layer < ctx->cfg.num_layers; }

uint4* kc_layer(vase_ctx* c, int layer) {
    return reinterpret_cast<uint4*>(c->bufs.k_cache) +
           static_cast<int64_t>(layer) * c->plan.units * c->plan.N * kVecPerRow;
}
uint4* vc_layer(vase_ctx* c, int layer) {
    return reinterpret_cast<uint4*>(c->bufs.v_cache) +
           static_cast<int64_t>(layer) * c->plan.units * c->plan.N * kVecPerRow;
}
int32_t* pos_layer(vase_ctx* c, int layer) {
    return c->bufs.positions + static_cast<int64_t>(layer) * c->plan.units * c->plan.N;
}

// The compressed value store's parameter block (layer-independent part).
StoreParams store_params(vase_ctx* ctx) {
    const Plan& P = ctx->plan;
    const vase_config& c = ctx->cfg;
    StoreParams sp;
    std::memset(&sp, 0, sizeof(sp));
    sp.base = static_cast<uint8_t*>(ctx->bufs.v_cache);
    sp.layer_bytes = static_cast<int64_t>(P.st_layer_bytes);
    sp.codes_off = static_cast<int64_t>(P.st_codes_off);
    sp.qp_off = static_cast<int64_t>(P.st_qp_off);
    sp.mask_off = static_cast<int64_t>(P.st_mask_off);
    sp.ring_off = static_cast<int64_t>(P.st_ring_off);
    sp.state_off = static_cast<int64_t>(P.st_state_off);
    sp.units = P.units;
    sp.N = P.N;
    sp.Np = P.st_Np;
    sp.mask_stride = P.st_mask_stride;
    sp.mask_words = P.st_mask_words;
    sp.H = P.st_H;
    sp.bits = c.value_bits;
    sp.code_row = P.st_code_row;
    sp.K = c.budget_k;
    sp.b = c.batch;
    sp.Hkv = c.num_kv_heads;
    sp.err = reinterpret_cast<uint32_t*>(ctx->ws + P.off_err);
    return sp;
}

}  // namespace

namespace vase {
cudaError_t launch_wait_timeout_probe(uint32_t* err, cudaStream_t s);  // selftest.cu: the failure-detection self-test
}

extern "C" {

void vase_config_default(vase_config* cfg) {
    if (!cfg) return;
    std::memset(cfg, 0, sizeof(*cfg));
    cfg->head_dim = 128;
    cfg->variant = VASE_VARIANT_ATTNV;
    cfg->n_v = -1;
    cfg->value_score = VASE_VALUE_RANGE;
    cfg->pool_kernel = 7;
    cfg->dkv_rank = 20;
    cfg->stochastic = 1;
    cfg->dkv_fixed_g = 0;
    cfg->debug_outputs = 0;
    cfg->seed = 0;
}

int vase_get_buffer_sizes(const vase_config* cfg, vase_buffer_sizes* out) {
    if (!cfg || !out) return VASE_ERR_INVALID;
    Plan p;
    const char* why = nullptr;
    if (!make_plan(cfg, 152, &p, &why)) return cfg->head_dim != 128 ? VASE_ERR_UNSUPPORTED : VASE_ERR_INVALID;
    const size_t rows = static_cast<size_t>(cfg->num_layers) * p.units * p.N;
    out->k_cache = rows * kRowBytes;
    out->v_cache = p.store ? static_cast<size_t>(cfg->num_layers) * p.st_layer_bytes : rows * kRowBytes;
    out->q_window = static_cast<size_t>(cfg->num_layers) * cfg->batch * cfg->num_q_heads * cfg->window * kRowBytes;
    out->positions = rows * 4;
    out->value_scores = rows * 4;
    out->workspace = p.ws_bytes;
    return VASE_OK;
}

int vase_create(const vase_config* cfg, const vase_buffers* bufs, vase_ctx** out) {
    if (!out) return VASE_ERR_INVALID;
    *out = nullptr;
    if (!cfg || !bufs) return VASE_ERR_INVALID;
    vase_ctx* ctx = new vase_ctx();
    ctx->cfg = *cfg;
    ctx->bufs = *bufs;
    cudaError_t e = cudaGetDevice(&ctx->device);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&ctx->num_sms, cudaDevAttrMultiProcessorCount, ctx->device);
    if (e != cudaSuccess) {
        int r = cuda_fail(ctx, e, "device query");
        fprintf(stderr, "vase_create: %s\n", ctx->last_error.c_str());
        delete ctx;
        return r;
    }
    const char* why = nullptr;
    if (!make_plan(cfg, ctx->num_sms, &ctx->plan, &why)) {
        fprintf(stderr, "vase_create: %s\n", why);
        delete ctx;
        return cfg->head_dim != 128 ? VASE_ERR_UNSUPPORTED : VASE_ERR_INVALID;
    }
    const void* ptrs[6] = {bufs->k_cache, bufs->v_cache, bufs->q_window, bufs->positions, bufs->value_scores,
                           bufs->workspace};
    for (const void* p : ptrs) {
        if (!p || !aligned(p, kAlign)) {
            fprintf(stderr, "vase_create: null or unaligned buffer (256-byte alignment required)\n");
            delete ctx;
            return p ? VASE_ERR_ALIGN : VASE_ERR_INVALID;
        }
    }
    ctx->ws = static_cast<uint8_t*>(bufs->workspace);
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
    if (e != cudaSuccess || !fn || q != cudaDriverEntryPointSuccess) {
        fprintf(stderr, "vase_create: cuTensorMapEncodeTiled unavailable\n");
        delete ctx;
        return VASE_ERR_CUDA;
    }
    EncodeTiledFn enc = reinterpret_cast<EncodeTiledFn>(fn);
    const Plan& P = ctx->plan;
    const uint64_t cache_rows = static_cast<uint64_t>(cfg->num_layers) * P.units * P.N;
    const uint64_t q_rows = static_cast<uint64_t>(cfg->num_layers) * cfg->batch * cfg->num_q_heads * cfg->window;
    if (cache_rows >= (1ull << 31) || q_rows >= (1ull << 31)) {
        fprintf(stderr, "vase_create: caches exceed 2^31 rows\n");
        delete ctx;
        return VASE_ERR_UNSUPPORTED;
    }
    const uint32_t qbox = static_cast<uint32_t>(P.q_box);
    // (with the compressed value store there are no V rows to map; no kernel of that mode reads the V maps)
    std::memset(&ctx->vmap, 0, sizeof(ctx->vmap));
    std::memset(&ctx->vmap_dec, 0, sizeof(ctx->vmap_dec));
    if (!encode_rows(enc, &ctx->kmap, bufs->k_cache, cache_rows, kTileTokens) ||
        (!P.store && !encode_rows(enc, &ctx->vmap, bufs->v_cache, cache_rows, kTileTokens)) ||
        !encode_rows(enc, &ctx->qmap, bufs->q_window, q_rows, qbox) ||
        !encode_rows(enc, &ctx->kmap_dec, bufs->k_cache, cache_rows, kDecodeTileRows) ||
        (!P.store && !encode_rows(enc, &ctx->vmap_dec, bufs->v_cache, cache_rows, kDecodeTileRows))) {
        fprintf(stderr, "vase_create: tensor map encoding failed\n");
        delete ctx;
        return VASE_ERR_CUDA;
    }
    if ((e = score_attn_set_attributes(P.score_smem, P.cluster)) != cudaSuccess ||
        (e = dkv_set_attributes(P.dkv_smem)) != cudaSuccess ||
        (e = select_set_attributes(P.select_smem)) != cudaSuccess ||
        (e = decode_set_attributes(P.G, P.decode_smem, P.store)) != cudaSuccess ||
        (e = decode_mixed_set_attributes()) != cudaSuccess ||
        (e = quantize_set_attributes(quantize_smem_bytes(cfg->budget_k, cfg->buffer_b))) != cudaSuccess ||
        (P.small_ok && (e = evict_small_set_attributes(P.small_smem)) != cudaSuccess) ||
        (P.store && (e = store_set_attributes(P.st_evict_smem, P.st_append_smem)) != cudaSuccess)) {
        fprintf(stderr, "vase_create: kernel attributes: %s\n", cudaGetErrorString(e));
        delete ctx;
        return VASE_ERR_CUDA;
    }
    if ((e = cudaMemset(ctx->ws + P.off_err, 0, kAlign)) != cudaSuccess) {
        fprintf(stderr, "vase_create: %s\n", cudaGetErrorString(e));
        delete ctx;
        return VASE_ERR_CUDA;
    }
    ctx->layers.assign(static_cast<size_t>(cfg->num_layers), vase_layer_state{0, 0, 0, 0});
    ctx->quant_round.assign(static_cast<size_t>(cfg->num_layers), -1);
    ctx->quant_bits.assign(static_cast<size_t>(cfg->num_layers), 0);
    *out = ctx;
    return VASE_OK;
}

void vase_destroy(vase_ctx* ctx) { delete ctx; }

namespace {

// Appends n_tokens to each layer of `layers` in one launch; the inputs of consecutive layer slots are q_stride
// and kv_stride bytes apart (0: packed, one slot's [n][b][H][d] after the other).
// Checks of an append's arguments (the same for every append entry point); VASE_OK or the failure.
int check_append(vase_ctx* ctx, const int32_t* layers, int n_layers, const void* q, const void* k, const void* v,
                 int32_t n_tokens, int64_t q_stride, int64_t kv_stride) {
    if (n_tokens < 1) return fail(ctx, VASE_ERR_INVALID, "n_tokens must be >= 1");
    if (!q || !k || !v) return fail(ctx, VASE_ERR_INVALID, "null input");
    if (!aligned(q, 16) || !aligned(k, 16) || !aligned(v, 16))
        return fail(ctx, VASE_ERR_ALIGN, "inputs must be 16-byte aligned");
    if (q_stride < 0 || kv_stride < 0 || q_stride % 16 || kv_stride % 16)
        return fail(ctx, VASE_ERR_ALIGN, "layer strides must be non-negative multiples of 16 bytes");
    for (int z = 0; z < n_layers; ++z)
        if (ctx->layers[layers[z]].fill + n_tokens > ctx->plan.N)
            return fail(ctx, VASE_ERR_FULL, "append would exceed K + B slots");
    return VASE_OK;
}

// The append kernel's parameter block for layers[z0 .. z0 + nz - 1] (inputs of layer slot z at q + z * q_stride and
// k, v + z * kv_stride; a stride of 0 means packed), from the layers' states before the append.
AppendParams append_params(vase_ctx* ctx, const int32_t* layers, int z0, int nz, const void* q, const void* k,
                           const void* v, int32_t n_tokens, int64_t q_stride, int64_t kv_stride) {
    const vase_config& c = ctx->cfg;
    const size_t q_slot = q_stride > 0 ? static_cast<size_t>(q_stride) / 16
                                       : static_cast<size_t>(n_tokens) * c.batch * c.num_q_heads * kVecPerRow;
    const size_t kv_slot = kv_stride > 0 ? static_cast<size_t>(kv_stride) / 16
                                         : static_cast<size_t>(n_tokens) * c.batch * c.num_kv_heads * kVecPerRow;
    AppendParams p{};
    p.q = static_cast<const uint4*>(q) + z0 * q_slot;
    p.k = static_cast<const uint4*>(k) + z0 * kv_slot;
    p.v = static_cast<const uint4*>(v) + z0 * kv_slot;
    p.q_stride = static_cast<int64_t>(q_slot);
    p.kv_stride = static_cast<int64_t>(kv_slot);
    p.qwin = static_cast<uint4*>(ctx->bufs.q_window);
    p.kc = static_cast<uint4*>(ctx->bufs.k_cache);
    p.vc = ctx->plan.store ? nullptr : static_cast<uint4*>(ctx->bufs.v_cache);  // store: values go below
    p.pos = ctx->bufs.positions;
    p.vmag = ctx->bufs.value_scores;
    p.kind = c.value_score;
    p.n = n_tokens;
    p.b = c.batch;
    p.Hq = c.num_q_heads;
    p.Hkv = c.num_kv_heads;
    p.W = c.window;
    p.N = ctx->plan.N;
    for (int z = 0; z < nz; ++z) {
        const vase_layer_state& st = ctx->layers[layers[z0 + z]];
        p.layer[z] = layers[z0 + z];
        p.fill[z] = st.fill;
        p.next_pos[z] = st.next_position;
        p.q_ring[z] = static_cast<int32_t>(st.queries_seen % c.window);
    }
    return p;
}

// The layers' states after an append of n_tokens; true when one of them is full (an eviction is due).
bool advance_after_append(vase_ctx* ctx, const int32_t* layers, int n_layers, int32_t n_tokens) {
    bool due = false;
    for (int z = 0; z < n_layers; ++z) {
        vase_layer_state& st = ctx->layers[layers[z]];
        st.fill += n_tokens;
        st.next_position += n_tokens;
        st.queries_seen += n_tokens;
        due |= st.fill == ctx->plan.N;
    }
    return due;
}

int append_batch(vase_ctx* ctx, const int32_t* layers, int n_layers, const void* q, const void* k, const void* v,
                 int32_t n_tokens, cudaStream_t stream, int64_t q_stride = 0, int64_t kv_stride = 0) {
    const int chk = check_append(ctx, layers, n_layers, q, k, v, n_tokens, q_stride, kv_stride);
    if (chk != VASE_OK) return chk;
    for (int z0 = 0; z0 < n_layers; z0 += kMaxLayerBatch) {
        const int nz = n_layers - z0 < kMaxLayerBatch ? n_layers - z0 : kMaxLayerBatch;
        const AppendParams p = append_params(ctx, layers, z0, nz, q, k, v, n_tokens, q_stride, kv_stride);
        cudaError_t e = timed_launch(ctx, VASE_KERNEL_APPEND, stream, [&] { return launch_append(p, nz, stream); });
        if (e != cudaSuccess) return cuda_fail(ctx, e, "append launch");
        ctx->launches += 1;
        if (ctx->plan.store) {
            StoreParams sp = store_params(ctx);
            for (int z = 0; z < nz; ++z) {
                const vase_layer_state& st = ctx->layers[layers[z0 + z]];
                sp.layer[z] = layers[z0 + z];
                sp.fill[z] = st.fill;
                sp.round[z] = st.round;
                // before the first eviction a fill past H overflows the ring (the bf16 count is at most the fill)
                if (st.round == 0 && st.fill + n_tokens > ctx->plan.st_H) sp.big = 1;
            }
            sp.v = p.v;
            sp.kv_stride = p.kv_stride;
            sp.n = n_tokens;
            sp.n_v = ctx->plan.n_v;
            sp.vmag = ctx->bufs.value_scores;
            e = timed_launch(ctx, VASE_KERNEL_STORE_APPEND, stream, [&] { return launch_store_append(sp, nz, stream); });
            if (e != cudaSuccess) return cuda_fail(ctx, e, "value store append launch");
            ctx->launches += 1;
        }
    }
    return advance_after_append(ctx, layers, n_layers, n_tokens) ? VASE_EVICT_DUE : VASE_OK;
}

LayerBatch make_batch(vase_ctx* ctx, const int32_t* layers, int nz) {
    LayerBatch b;
    b.n = nz;
    for (int z = 0; z < nz; ++z) {
        b.layer[z] = layers[z];
        b.rnd[z] = ctx->layers[layers[z]].round;
    }
    return b;
}

// The selection's parameter block for one batched eviction (workspace arrays of the batch's first slot).
void fill_select_params(vase_ctx* ctx, const LayerBatch& batch, float* attn, float* vscore, int32_t* src,
                        uint32_t* err, SelectParams* out) {
    const Plan& P = ctx->plan;
    const vase_config& c = ctx->cfg;
    SelectParams& sel = *out;
    sel.batch = batch;
    sel.attn = attn;
    sel.dkv = vscore;
    sel.vmag = ctx->bufs.value_scores;
    sel.vscore_dbg = (c.debug_outputs && c.variant == VASE_VARIANT_ATTNV) ? vscore : nullptr;
    sel.pos = ctx->bufs.positions;
    sel.kc = static_cast<uint4*>(ctx->bufs.k_cache);
    sel.vc = P.store ? nullptr : static_cast<uint4*>(ctx->bufs.v_cache);  // the store's values move below
    sel.src = src;
    sel.resv = P.store ? ctx->ws + P.off_resv : nullptr;
    sel.pooled_dbg = c.debug_outputs ? reinterpret_cast<float*>(ctx->ws + P.off_pooled) : nullptr;
    sel.key_dbg = c.debug_outputs ? reinterpret_cast<float*>(ctx->ws + P.off_key) : nullptr;
    sel.keep_dbg = c.debug_outputs ? ctx->ws + P.off_keep : nullptr;
    sel.N = P.N;
    sel.K = c.budget_k;
    sel.B = c.buffer_b;
    sel.n_v = P.n_v;
    sel.m = P.m;
    sel.pool = c.pool_kernel;
    sel.variant = c.variant;
    sel.stochastic = c.stochastic;
    sel.Hkv = c.num_kv_heads;
    sel.n_parts = c.variant == VASE_VARIANT_ATTNV ? P.n_rb : 1;
    sel.staged = P.select_staged ? 1 : 0;
    sel.reserve_random = c.reserve_kind == VASE_RESERVE_RANDOM ? 1 : 0;
    sel.gqa_max = c.gqa_reduce == VASE_GQA_MAX ? 1 : 0;
    sel.units = P.units;
    sel.seed_lo = static_cast<uint32_t>(c.seed & 0xFFFFFFFFull);
    sel.seed_hi = static_cast<uint32_t>(c.seed >> 32);
    sel.err = err;
}

// True when a batched eviction of nz layers runs the fused small-unit kernel: every unit of every layer in one
// wave, one CTA each, and units small enough for it.
bool fused_small(const Plan& P, int nz) { return P.small_ok && static_cast<long>(P.units) * nz <= P.num_sms; }

// One eviction step for up to kMaxLayerBatch full layers: every kernel covers all of them in one launch.  With
// fused_append (only where fused_small holds) the fused kernel first appends the step's rows of every unit.
int evict_batch(vase_ctx* ctx, const int32_t* layers, int nz, cudaStream_t s,
                const AppendParams* fused_append = nullptr) {
    const Plan& P = ctx->plan;
    const vase_config& c = ctx->cfg;
    const LayerBatch batch = make_batch(ctx, layers, nz);
    uint32_t* err = reinterpret_cast<uint32_t*>(ctx->ws + P.off_err);
    float* attn = reinterpret_cast<float*>(ctx->ws + P.off_attn);
    float* vscore = reinterpret_cast<float*>(ctx->ws + P.off_vscore);
    int32_t* src = reinterpret_cast<int32_t*>(ctx->ws + P.off_src);
    cudaError_t e;
    if (ctx->read_pending) {  // the positions a read-back copies must not move before it has run
        if ((e = cudaStreamWaitEvent(s, ctx->read_done, 0)) != cudaSuccess) return cuda_fail(ctx, e, "read-back wait");
        ctx->read_pending = false;
    }
    SelectParams sel{};  // value-initialised: a field this path does not set is zero (pointers null)
    fill_select_params(ctx, batch, attn, vscore, src, err, &sel);
    // Launch-bound batches (every unit of every layer in one wave, one CTA each) whose units are small enough for
    // the fused kernel: score, selection and gather in one launch
    if (fused_small(P, nz)) {
        SmallEvictParams sm{};
        if (fused_append) {
            sm.append = 1;
            sm.ap = *fused_append;
        }
        sm.sel = sel;
        sm.sel.n_parts = 1;
        sm.sel.staged = 1;
        sm.GW = P.GW;
        sm.GWp = P.GWp;
        sm.q_rows = P.q_box;
        sm.n_tiles = P.small_tiles;
        sm.stages = P.small_stages;
        sm.tmem_cols = P.small_tmem_cols;
        sm.Hq = c.num_q_heads;
        sm.W = c.window;
        sm.G = P.G;
        sm.head_rows = c.gqa_reduce == VASE_GQA_MAX ? c.window : 0;
        sm.fold_rows = c.gqa_reduce == VASE_GQA_MAX ? c.window : P.GW;
        sm.layer_rows = static_cast<int64_t>(P.units) * P.N;
        sm.q_layer_rows = static_cast<int64_t>(c.batch) * c.num_q_heads * c.window;
        sm.scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(kHeadDim));
        sm.attn = attn;
        if ((e = timed_launch(ctx, VASE_KERNEL_EVICT_SMALL, s, [&] {
                 return launch_evict_small(ctx->kmap, ctx->qmap, sm, P.units, P.small_smem, s);
             })) != cudaSuccess)
            return cuda_fail(ctx, e, "fused small-unit eviction launch");
        ctx->launches += 1;
        for (int z = 0; z < nz; ++z) {
            vase_layer_state& st = ctx->layers[layers[z]];
            st.fill = c.budget_k;
            st.round += 1;
        }
        return VASE_OK;
    }
    if (fused_append) return fail(ctx, VASE_ERR_INVALID, "a fused append needs the fused small-unit eviction");
    if (c.variant == VASE_VARIANT_ATTNV) {
        const ScoreAttnParams sp = score_params(P, c, batch, nz, attn, err);
        if ((e = timed_launch(ctx, VASE_KERNEL_SCORE, s, [&] {
                 return launch_score_attn(ctx->kmap, ctx->qmap, sp, P.score_smem, s);
             })) != cudaSuccess)
            return cuda_fail(ctx, e, "score launch");
        ctx->launches += 1;
    } else {
        DkvParams dp{};
        dp.batch = batch;
        dp.N = P.N;
        dp.K = c.budget_k;
        dp.r = c.dkv_rank;
        dp.Hkv = c.num_kv_heads;
        dp.fixed_g = c.dkv_fixed_g;
        dp.shared_g = c.dkv_shared_g;
        dp.units = P.units;
        dp.seed_lo = static_cast<uint32_t>(c.seed & 0xFFFFFFFFull);
        dp.seed_hi = static_cast<uint32_t>(c.seed >> 32);
        dp.n_tiles_k = P.dkv_tiles_k;
        dp.tiles_per_cta = P.dkv_tiles_per_cta;
        dp.stages = P.dkv_stages;
        dp.layer_rows = static_cast<int64_t>(P.units) * P.N;
        dp.out = vscore;
        dp.err = err;
        if ((e = timed_launch(ctx, VASE_KERNEL_DKV, s, [&] {
                 return launch_dkv(ctx->kmap, ctx->vmap, dp, P.units, P.dkv_smem, s);
             })) != cudaSuccess)
            return cuda_fail(ctx, e, "dkv launch");
        ctx->launches += 1;
    }
    if ((e = timed_launch(ctx, VASE_KERNEL_SELECT, s, [&] { return launch_select(sel, P.units, P.select_smem, P.select_threads, s); })) !=
        cudaSuccess)
        return cuda_fail(ctx, e, "select launch");
    ctx->launches += 1;
    if (P.store) {
        StoreParams sp = store_params(ctx);
        for (int z = 0; z < nz; ++z) sp.layer[z] = layers[z];
        sp.src = src;
        sp.resv = ctx->ws + P.off_resv;
        if ((e = timed_launch(ctx, VASE_KERNEL_STORE_EVICT, s, [&] { return launch_store_evict(sp, nz, s); })) !=
            cudaSuccess)
            return cuda_fail(ctx, e, "value store eviction launch");
        ctx->launches += 1;
    }
    for (int z = 0; z < nz; ++z) {
        vase_layer_state& st = ctx->layers[layers[z]];
        st.fill = c.budget_k;
        st.round += 1;
    }
    return VASE_OK;
}

}  // namespace

int vase_append(vase_ctx* ctx, int32_t layer, const void* q, const void* k, const void* v, int32_t n_tokens,
                void* stream) {
    if (!ctx) return VASE_ERR_INVALID;
    if (!check_layer(ctx, layer)) return fail(ctx, VASE_ERR_INVALID, "layer out of range");
    return append_batch(ctx, &layer, 1, q, k, v, n_tokens, static_cast<cudaStream_t>(stream));
}

int vase_append_all(vase_ctx* ctx, const void* q, const void* k, const void* v, int32_t n_tokens, void* stream) {
    if (!ctx) return VASE_ERR_INVALID;
    std::vector<int32_t> all(static_cast<size_t>(ctx->cfg.num_layers));
    for (int32_t l = 0; l < ctx->cfg.num_layers; ++l) all[l] = l;
    return append_batch(ctx, all.data(), ctx->cfg.num_layers, q, k, v, n_tokens, static_cast<cudaStream_t>(stream));
}

int vase_append_all_strided(vase_ctx* ctx, const void* q, const void* k, const void* v, int32_t n_tokens,
                            int64_t q_layer_stride, int64_t kv_layer_stride, void* stream) {
    if (!ctx) return VASE_ERR_INVALID;
    if (q_layer_stride <= 0 || kv_layer_stride <= 0) return fail(ctx, VASE_ERR_INVALID, "layer strides must be > 0");
    std::vector<int32_t> all(static_cast<size_t>(ctx->cfg.num_layers));
    for (int32_t l = 0; l < ctx->cfg.num_layers; ++l) all[l] = l;
    return append_batch(ctx, all.data(), ctx->cfg.num_layers, q, k, v, n_tokens, static_cast<cudaStream_t>(stream),
                        q_layer_stride, kv_layer_stride);
}

namespace {

// Device-visible address of page-locked (pinned or registered) host memory, or nullptr for any other pointer.
const void* mapped_host_pointer(const void* host) {
    cudaPointerAttributes a;
    if (cudaPointerGetAttributes(&a, host) != cudaSuccess) {
        cudaGetLastError();  // clear the sticky-free error of an unknown pointer
        return nullptr;
    }
    return a.type == cudaMemoryTypeHost ? a.devicePointer : nullptr;
}

}  // namespace

int vase_append_host(vase_ctx* ctx, int32_t layer, const void* q_host, const void* k_host, const void* v_host,
                     int32_t n_tokens, void* stream) {
    if (!ctx) return VASE_ERR_INVALID;
    if (!check_layer(ctx, layer)) return fail(ctx, VASE_ERR_INVALID, "layer out of range");
    if (n_tokens < 1 || n_tokens > ctx->cfg.buffer_b)
        return fail(ctx, VASE_ERR_INVALID, "n_tokens must be in 1..buffer_b for host appends");
    if (!q_host || !k_host || !v_host) return fail(ctx, VASE_ERR_INVALID, "null input");
    if (ctx->layers[layer].fill + n_tokens > ctx->plan.N) return fail(ctx, VASE_ERR_FULL, "append would exceed K + B slots");
    // Page-locked inputs: the append kernel reads them over the host link itself (no staging copies); only
    // the query rows that stay in the window ring (the last W steps) are read at all.
    const void* qd = mapped_host_pointer(q_host);
    const void* kd = mapped_host_pointer(k_host);
    const void* vd = mapped_host_pointer(v_host);
    if (qd && kd && vd) return vase_append(ctx, layer, qd, kd, vd, n_tokens, stream);
    // Otherwise copy into the staging area of the workspace: all k and v rows, and the query rows of the
    // last min(W, n_tokens) steps only.  The kernel addresses q by step, so it is handed the staged rows'
    // address less the skipped steps (it never reads a step before the last W).
    const int n_q = n_tokens < ctx->cfg.window ? n_tokens : ctx->cfg.window;
    const size_t q_step = static_cast<size_t>(ctx->cfg.batch) * ctx->cfg.num_q_heads * kRowBytes;
    const size_t qb = static_cast<size_t>(n_q) * q_step;
    const size_t kb = static_cast<size_t>(n_tokens) * ctx->cfg.batch * ctx->cfg.num_kv_heads * kRowBytes;
    uint8_t* sq = ctx->ws + ctx->plan.off_staging;
    uint8_t* sk = sq + static_cast<size_t>(ctx->cfg.buffer_b) * q_step;
    uint8_t* sv = sk + kb;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const size_t skipped = static_cast<size_t>(n_tokens - n_q) * q_step;
    cudaError_t e;
    if ((e = cudaMemcpyAsync(sq, static_cast<const uint8_t*>(q_host) + skipped, qb, cudaMemcpyHostToDevice, s)) !=
            cudaSuccess ||
        (e = cudaMemcpyAsync(sk, k_host, kb, cudaMemcpyHostToDevice, s)) != cudaSuccess ||
        (e = cudaMemcpyAsync(sv, v_host, kb, cudaMemcpyHostToDevice, s)) != cudaSuccess)
        return cuda_fail(ctx, e, "host-to-device staging copy");
    const void* q_dev = reinterpret_cast<const void*>(reinterpret_cast<uintptr_t>(sq) - skipped);
    return vase_append(ctx, layer, q_dev, sk, sv, n_tokens, stream);
}

int vase_evict(vase_ctx* ctx, int32_t layer, void* stream) {
    if (!ctx) return VASE_ERR_INVALID;
    if (!check_layer(ctx, layer)) return fail(ctx, VASE_ERR_INVALID, "layer out of range");
    if (ctx->layers[layer].fill != ctx->plan.N) return fail(ctx, VASE_ERR_NOT_FULL, "evict needs a full cache (fill == K + B)");
    const int r = evict_batch(ctx, &layer, 1, static_cast<cudaStream_t>(stream));
    if (r == VASE_OK) ctx->last_batch.assign(1, layer);
    return r;
}

int vase_evict_all(vase_ctx* ctx, void* stream) {
    if (!ctx) return VASE_ERR_INVALID;
    std::vector<int32_t> due;
    for (int32_t l = 0; l < ctx->cfg.num_layers; ++l)
        if (ctx->layers[l].fill == ctx->plan.N) due.push_back(l);
    std::vector<int32_t> done;
    for (size_t z0 = 0; z0 < due.size(); z0 += static_cast<size_t>(ctx->plan.slots)) {
        const int nz = static_cast<int>(due.size() - z0 < static_cast<size_t>(ctx->plan.slots) ? due.size() - z0
                                                                                                : ctx->plan.slots);
        const int r = evict_batch(ctx, due.data() + z0, nz, static_cast<cudaStream_t>(stream));
        if (r != VASE_OK) return r;
        done.assign(due.begin() + static_cast<long>(z0), due.begin() + static_cast<long>(z0) + nz);
    }
    ctx->last_batch = done;
    return static_cast<int>(due.size());
}

int vase_append_evict_all(vase_ctx* ctx, const void* q, const void* k, const void* v, int32_t n_tokens,
                          int64_t q_layer_stride, int64_t kv_layer_stride, void* stream) {
    if (!ctx) return VASE_ERR_INVALID;
    const Plan& P = ctx->plan;
    const int L = ctx->cfg.num_layers;
    // one launch where the append makes every layer full and the eviction of all of them is the fused kernel's
    bool fused = !P.store && L <= P.slots && fused_small(P, L) && n_tokens >= 1;
    for (int l = 0; l < L && fused; ++l) fused = ctx->layers[l].fill + n_tokens == P.N;
    if (!fused) {
        const int r = vase_append_all_strided(ctx, q, k, v, n_tokens, q_layer_stride, kv_layer_stride, stream);
        if (r < 0) return r;
        return vase_evict_all(ctx, stream);
    }
    if (q_layer_stride <= 0 || kv_layer_stride <= 0) return fail(ctx, VASE_ERR_INVALID, "layer strides must be > 0");
    std::vector<int32_t> all(static_cast<size_t>(L));
    for (int32_t l = 0; l < L; ++l) all[l] = l;
    const int chk = check_append(ctx, all.data(), L, q, k, v, n_tokens, q_layer_stride, kv_layer_stride);
    if (chk != VASE_OK) return chk;
    const AppendParams ap = append_params(ctx, all.data(), 0, L, q, k, v, n_tokens, q_layer_stride, kv_layer_stride);
    advance_after_append(ctx, all.data(), L, n_tokens);
    const int r = evict_batch(ctx, all.data(), L, static_cast<cudaStream_t>(stream), &ap);
    if (r != VASE_OK) return r;
    ctx->last_batch = all;
    return L;
}

int vase_refresh_value_scores(vase_ctx* ctx, int32_t layer, void* stream) {
    if (!ctx) return VASE_ERR_INVALID;
    if (!check_layer(ctx, layer)) return fail(ctx, VASE_ERR_INVALID, "layer out of range");
    if (ctx->plan.store)
        return fail(ctx, VASE_ERR_UNSUPPORTED, "the compressed value store keeps no bf16 rows to recompute magnitudes from");
    const int rows = ctx->layers[layer].fill;
    if (rows == 0) return VASE_OK;
    ValueParams vp{};
    vp.vc = static_cast<const uint4*>(ctx->bufs.v_cache) + static_cast<int64_t>(layer) * ctx->plan.units * ctx->plan.N * kVecPerRow;
    vp.out = ctx->bufs.value_scores + static_cast<int64_t>(layer) * ctx->plan.units * ctx->plan.N;
    vp.N = ctx->plan.N;
    vp.rows = rows;
    vp.units = ctx->plan.units;
    vp.kind = ctx->cfg.value_score;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = timed_launch(ctx, VASE_KERNEL_VALUE, s, [&] { return launch_value_score(vp, ctx->num_sms, s); });
    if (e != cudaSuccess) return cuda_fail(ctx, e, "value refresh launch");
    ctx->launches += 1;
    return VASE_OK;
}

}  // extern "C"

namespace {

// Decode attention over the compressed value store: the mixed-precision kernel with the store's arrays (codes of
// every slot, the ring of bf16 rows and its head).
int decode_store(vase_ctx* ctx, int32_t layer, const void* q, float* out, cudaStream_t stream) {
    const Plan& P = ctx->plan;
    if (P.G > 16) return fail(ctx, VASE_ERR_UNSUPPORTED, "decode handles at most 16 query heads per KV head");
    uint8_t* base = static_cast<uint8_t*>(ctx->bufs.v_cache) + static_cast<size_t>(layer) * P.st_layer_bytes;
    DecodeParams dp{};
    dp.q = static_cast<const uint4*>(q);
    dp.kc = kc_layer(ctx, layer);
    dp.vc = nullptr;
    dp.out = out;
    dp.N = P.N;
    dp.fill = ctx->layers[layer].fill;
    dp.G = P.G;
    dp.Hkv = ctx->cfg.num_kv_heads;
    dp.units = P.units;
    dp.row_base = layer * P.units * P.N;
    dp.scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(kHeadDim));
    dp.err = reinterpret_cast<uint32_t*>(ctx->ws + P.off_err);
    dp.codes = base + P.st_codes_off;
    dp.qparams = reinterpret_cast<const float*>(base + P.st_qp_off);
    dp.rmask = reinterpret_cast<const uint32_t*>(base + P.st_mask_off);
    dp.hp_rows = reinterpret_cast<const uint4*>(base + P.st_ring_off);
    dp.ring_state = reinterpret_cast<const int32_t*>(base + P.st_state_off);
    dp.bits = ctx->cfg.value_bits;
    dp.code_row = P.st_code_row;
    dp.Kq = P.N;  // every slot has a code row (unit stride N); bf16 values are the masked ones
    dp.Kp = P.st_Np;
    dp.mask_words = P.st_mask_stride;
    dp.hp_cap = P.st_H;
    // the tensor-core kernel, its V tiles written from the ring rows and the codes by builder warps
    cudaError_t e = launch_decode(ctx->kmap_dec, ctx->vmap_dec, dp, P.decode_smem, P.num_sms, stream);
    if (e == cudaErrorInvalidValue) return fail(ctx, VASE_ERR_UNSUPPORTED, "too many slots for the mixed decode");
    if (e != cudaSuccess) return cuda_fail(ctx, e, "value store decode attention launch");
    ctx->launches += 1;
    return VASE_OK;
}

}  // namespace

extern "C" {

int vase_decode_attention(vase_ctx* ctx, int32_t layer, const void* q, float* out, void* stream) {
    if (!ctx) return VASE_ERR_INVALID;
    if (!check_layer(ctx, layer)) return fail(ctx, VASE_ERR_INVALID, "layer out of range");
    if (!q || !out) return fail(ctx, VASE_ERR_INVALID, "null input or output");
    if (!aligned(q, 16) || !aligned(out, 4)) return fail(ctx, VASE_ERR_ALIGN, "q must be 16-byte aligned, out 4-byte");
    const int fill = ctx->layers[layer].fill;
    if (fill < 1) return fail(ctx, VASE_ERR_INVALID, "the layer holds no cached pair");
    const Plan& P = ctx->plan;
    if (P.G > 16) return fail(ctx, VASE_ERR_UNSUPPORTED, "decode attention handles at most 16 query heads per KV head");
    if (P.store) return decode_store(ctx, layer, q, out, static_cast<cudaStream_t>(stream));
    DecodeParams dp{};
    dp.q = static_cast<const uint4*>(q);
    dp.kc = kc_layer(ctx, layer);
    dp.vc = vc_layer(ctx, layer);
    dp.ring_state = nullptr;
    dp.out = out;
    dp.N = P.N;
    dp.fill = fill;
    dp.G = P.G;
    dp.Hkv = ctx->cfg.num_kv_heads;
    dp.units = P.units;
    dp.row_base = layer * P.units * P.N;
    dp.scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(kHeadDim));
    dp.err = reinterpret_cast<uint32_t*>(ctx->ws + P.off_err);
    dp.codes = nullptr;
    dp.qparams = nullptr;
    dp.rmask = nullptr;
    dp.hp_rows = nullptr;
    dp.bits = dp.code_row = dp.Kq = dp.Kp = dp.mask_words = dp.hp_cap = 0;
    cudaError_t e =
        launch_decode(ctx->kmap_dec, ctx->vmap_dec, dp, P.decode_smem, P.num_sms, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(ctx, e, "decode attention launch");
    ctx->launches += 1;
    return VASE_OK;
}

// Reserved rows per unit: R_V (N_v, none for DKV) and R_B.
int hp_capacity(const vase_config* c) {
    const int nv = c->variant == VASE_VARIANT_ATTNV ? (c->n_v < 0 ? c->budget_k / 4 : c->n_v) : 0;
    return nv + c->buffer_b;
}

int vase_mixed_buffer_sizes(const vase_config* cfg, int32_t bits, size_t* codes, size_t* qparams, size_t* rmask,
                            size_t* hp_rows) {
    if (const char* why = check_config(cfg)) {
        g_config_error = why;
        return VASE_ERR_INVALID;
    }
    if (bits != 2 && bits != 4 && bits != 8) {
        g_config_error = "bits must be 2, 4 or 8";
        return VASE_ERR_INVALID;
    }
    const size_t units = static_cast<size_t>(cfg->batch) * cfg->num_kv_heads;
    const size_t K = static_cast<size_t>(cfg->budget_k);
    if (codes) *codes = units * K * (kHeadDim * bits / 8);
    if (qparams) *qparams = units * ((K + 1) & ~size_t(1)) * 2 * sizeof(float);
    if (rmask) *rmask = units * ((K + 31) / 32) * sizeof(uint32_t);
    if (hp_rows) *hp_rows = units * static_cast<size_t>(hp_capacity(cfg)) * kRowBytes;
    return VASE_OK;
}

int vase_quantize_values(vase_ctx* ctx, int32_t layer, int32_t bits, const vase_mixed_buffers* mb, void* stream) {
    if (!ctx) return VASE_ERR_INVALID;
    if (!check_layer(ctx, layer)) return fail(ctx, VASE_ERR_INVALID, "layer out of range");
    if (bits != 2 && bits != 4 && bits != 8) return fail(ctx, VASE_ERR_INVALID, "bits must be 2, 4 or 8");
    if (ctx->plan.store)
        return fail(ctx, VASE_ERR_UNSUPPORTED, "the compressed value store quantizes by itself (value_bits)");
    if (!mb || !mb->codes || !mb->qparams || !mb->rmask || !mb->hp_rows)
        return fail(ctx, VASE_ERR_INVALID, "null mixed buffers");
    if (!aligned(mb->codes, 16) || !aligned(mb->qparams, 16) || !aligned(mb->rmask, 16) || !aligned(mb->hp_rows, 16))
        return fail(ctx, VASE_ERR_ALIGN, "mixed buffers must be 16-byte aligned");
    const vase_config& c = ctx->cfg;
    if (c.variant == VASE_VARIANT_ATTNV && c.reserve_kind == VASE_RESERVE_RANDOM)
        return fail(ctx, VASE_ERR_UNSUPPORTED, "random reservation: R_V is not a function of the kept values");
    const vase_layer_state& st = ctx->layers[layer];
    if (st.round < 1 || st.fill != c.budget_k)
        return fail(ctx, VASE_ERR_INVALID, "quantize right after an eviction (fill == K)");
    const Plan& P = ctx->plan;
    QuantParams qp{};
    qp.vc = vc_layer(ctx, layer);
    qp.vmag = ctx->bufs.value_scores + static_cast<int64_t>(layer) * P.units * P.N;
    qp.codes = static_cast<uint8_t*>(mb->codes);
    qp.qparams = mb->qparams;
    qp.rmask = mb->rmask;
    qp.N = P.N;
    qp.K = c.budget_k;
    qp.B = c.buffer_b;
    qp.n_v = c.variant == VASE_VARIANT_ATTNV ? P.n_v : 0;
    qp.bits = bits;
    qp.row_bytes = kHeadDim * bits / 8;
    qp.Kp = (c.budget_k + 1) & ~1;
    qp.mask_words = (c.budget_k + 31) / 32;
    qp.hp_rows = static_cast<uint4*>(mb->hp_rows);
    qp.hp_cap = hp_capacity(&c);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = launch_quantize(qp, P.units, quantize_smem_bytes(c.budget_k, c.buffer_b), s);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "quantize launch");
    ctx->launches += 1;
    ctx->quant_round[layer] = st.round;
    ctx->quant_bits[layer] = bits;
    return VASE_OK;
}

int vase_decode_attention_mixed(vase_ctx* ctx, int32_t layer, int32_t bits, const vase_mixed_buffers* mb,
                                const void* q, float* out, void* stream) {
    if (!ctx) return VASE_ERR_INVALID;
    if (!check_layer(ctx, layer)) return fail(ctx, VASE_ERR_INVALID, "layer out of range");
    if (ctx->plan.store)
        return fail(ctx, VASE_ERR_UNSUPPORTED, "with the compressed value store, vase_decode_attention reads it");
    if (!q || !out || !mb || !mb->codes || !mb->qparams || !mb->rmask || !mb->hp_rows)
        return fail(ctx, VASE_ERR_INVALID, "null input, output or mixed buffer");
    if (!aligned(q, 16) || !aligned(out, 4)) return fail(ctx, VASE_ERR_ALIGN, "q must be 16-byte aligned, out 4-byte");
    if (!aligned(mb->codes, 16) || !aligned(mb->qparams, 16) || !aligned(mb->rmask, 16) || !aligned(mb->hp_rows, 16))
        return fail(ctx, VASE_ERR_ALIGN, "mixed buffers must be 16-byte aligned");
    const vase_layer_state& st = ctx->layers[layer];
    if (ctx->quant_round[layer] != st.round || ctx->quant_bits[layer] != bits)
        return fail(ctx, VASE_ERR_INVALID, "no codes of this bit width for the layer's current round");
    const Plan& P = ctx->plan;
    if (P.G > 16) return fail(ctx, VASE_ERR_UNSUPPORTED, "decode attention handles at most 16 query heads per KV head");
    DecodeParams dp{};
    dp.q = static_cast<const uint4*>(q);
    dp.kc = kc_layer(ctx, layer);
    dp.vc = vc_layer(ctx, layer);
    dp.out = out;
    dp.N = P.N;
    dp.fill = st.fill;
    dp.G = P.G;
    dp.Hkv = ctx->cfg.num_kv_heads;
    dp.units = P.units;
    dp.row_base = layer * P.units * P.N;
    dp.scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(kHeadDim));
    dp.err = reinterpret_cast<uint32_t*>(ctx->ws + P.off_err);
    dp.codes = static_cast<const uint8_t*>(mb->codes);
    dp.qparams = mb->qparams;
    dp.rmask = mb->rmask;
    dp.ring_state = nullptr;
    dp.bits = bits;
    dp.code_row = kHeadDim * bits / 8;
    dp.Kq = ctx->cfg.budget_k;
    dp.Kp = (ctx->cfg.budget_k + 1) & ~1;
    dp.mask_words = (ctx->cfg.budget_k + 31) / 32;
    dp.hp_rows = static_cast<const uint4*>(mb->hp_rows);
    dp.hp_cap = hp_capacity(&ctx->cfg);
    cudaError_t e = launch_decode_mixed(dp, P.num_sms, static_cast<cudaStream_t>(stream));
    if (e == cudaErrorInvalidValue) return fail(ctx, VASE_ERR_UNSUPPORTED, "too many chunks per CTA for the mixed decode");
    if (e != cudaSuccess) return cuda_fail(ctx, e, "mixed decode attention launch");
    ctx->launches += 1;
    return VASE_OK;
}

int vase_read_positions(vase_ctx* ctx, int32_t layer, int32_t* host_out, void* stream) {
    if (!ctx) return VASE_ERR_INVALID;
    if (!check_layer(ctx, layer) || !host_out) return fail(ctx, VASE_ERR_INVALID, "bad layer or null output");
    const Plan& P = ctx->plan;
    const size_t width = static_cast<size_t>(ctx->cfg.budget_k) * 4;
    cudaError_t e = cudaMemcpy2DAsync(host_out, width, pos_layer(ctx, layer), static_cast<size_t>(P.N) * 4, width,
                                      static_cast<size_t>(P.units), cudaMemcpyDeviceToHost,
                                      static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(ctx, e, "positions copy");
    return VASE_OK;
}

namespace {

// One step's staging block per layer: [the last w_q query rows | n key rows | n value rows].
int64_t staged_block_bytes(const vase_config& c, int32_t n_tokens, int32_t* w_q) {
    *w_q = n_tokens < c.window ? n_tokens : c.window;
    const int64_t q_step = static_cast<int64_t>(c.batch) * c.num_q_heads * kRowBytes;
    const int64_t kv = static_cast<int64_t>(n_tokens) * c.batch * c.num_kv_heads * kRowBytes;
    return align_up(static_cast<size_t>(*w_q * q_step + 2 * kv), kAlign);
}

cudaError_t lazy_event(cudaEvent_t* ev) {
    if (*ev) return cudaSuccess;
    return cudaEventCreateWithFlags(ev, cudaEventDisableTiming);
}

}  // namespace

size_t vase_host_staging_bytes(const vase_config* cfg, int32_t n_tokens) {
    if (!cfg || n_tokens < 1 || check_config(cfg)) return 0;
    int32_t w_q = 0;
    return static_cast<size_t>(cfg->num_layers) * static_cast<size_t>(staged_block_bytes(*cfg, n_tokens, &w_q));
}

int vase_stage_host_inputs(vase_ctx* ctx, const void* q_host, const void* k_host, const void* v_host,
                           int32_t n_tokens, int64_t q_layer_stride, int64_t kv_layer_stride, void* staging,
                           size_t staging_bytes, void* copy_stream) {
    if (!ctx) return VASE_ERR_INVALID;
    const vase_config& c = ctx->cfg;
    if (!q_host || !k_host || !v_host || !staging) return fail(ctx, VASE_ERR_INVALID, "null input or staging buffer");
    if (n_tokens < 1 || n_tokens > c.buffer_b) return fail(ctx, VASE_ERR_INVALID, "n_tokens must be in 1..buffer_b");
    int32_t w_q = 0;
    const int64_t block = staged_block_bytes(c, n_tokens, &w_q);
    const int64_t q_step = static_cast<int64_t>(c.batch) * c.num_q_heads * kRowBytes;
    const int64_t kv = static_cast<int64_t>(n_tokens) * c.batch * c.num_kv_heads * kRowBytes;
    if (q_layer_stride < w_q * q_step || kv_layer_stride < kv)
        return fail(ctx, VASE_ERR_INVALID, "layer strides smaller than one layer's inputs");
    if (q_layer_stride % 16 || kv_layer_stride % 16)
        return fail(ctx, VASE_ERR_ALIGN, "layer strides must be multiples of 16 bytes");
    const size_t half = static_cast<size_t>(c.num_layers) * static_cast<size_t>(block);
    if (staging_bytes < 2 * half) return fail(ctx, VASE_ERR_INVALID, "staging buffer smaller than 2 x vase_host_staging_bytes");
    if (!aligned(staging, kAlign)) return fail(ctx, VASE_ERR_ALIGN, "staging buffer must be 256-byte aligned");
    if (ctx->staged_count == 2) return fail(ctx, VASE_ERR_FULL, "two steps are staged already: append one first");
    cudaStream_t cs = static_cast<cudaStream_t>(copy_stream);
    vase_ctx::Staged& h = ctx->staged[ctx->staged_next];
    cudaError_t e;
    if ((e = lazy_event(&h.copied)) != cudaSuccess || (e = lazy_event(&h.consumed)) != cudaSuccess)
        return cuda_fail(ctx, e, "staging events");
    if (h.consumed_pending) {  // the append that read this half before must have run
        if ((e = cudaStreamWaitEvent(cs, h.consumed, 0)) != cudaSuccess) return cuda_fail(ctx, e, "staging wait");
        h.consumed_pending = false;
    }
    uint8_t* dst = static_cast<uint8_t*>(staging) + static_cast<size_t>(ctx->staged_next) * half;
    const uint8_t* qs = static_cast<const uint8_t*>(q_host) + static_cast<int64_t>(n_tokens - w_q) * q_step;
    const size_t L = static_cast<size_t>(c.num_layers);
    // three strided copies move every layer's query tail, keys and values into its block
    if ((e = cudaMemcpy2DAsync(dst, static_cast<size_t>(block), qs, static_cast<size_t>(q_layer_stride),
                               static_cast<size_t>(w_q * q_step), L, cudaMemcpyHostToDevice, cs)) != cudaSuccess ||
        (e = cudaMemcpy2DAsync(dst + w_q * q_step, static_cast<size_t>(block), k_host,
                               static_cast<size_t>(kv_layer_stride), static_cast<size_t>(kv), L,
                               cudaMemcpyHostToDevice, cs)) != cudaSuccess ||
        (e = cudaMemcpy2DAsync(dst + w_q * q_step + kv, static_cast<size_t>(block), v_host,
                               static_cast<size_t>(kv_layer_stride), static_cast<size_t>(kv), L,
                               cudaMemcpyHostToDevice, cs)) != cudaSuccess ||
        (e = cudaEventRecord(h.copied, cs)) != cudaSuccess)
        return cuda_fail(ctx, e, "host-to-device staging copy");
    h.base = dst;
    h.n_tokens = n_tokens;
    h.w_q = w_q;
    h.block = block;
    ctx->staged_next ^= 1;
    ctx->staged_count += 1;
    return VASE_OK;
}

int vase_append_all_staged(vase_ctx* ctx, void* stream) {
    if (!ctx) return VASE_ERR_INVALID;
    if (ctx->staged_count == 0) return fail(ctx, VASE_ERR_INVALID, "no staged step: call vase_stage_host_inputs first");
    const int oldest = (ctx->staged_next + 2 - ctx->staged_count) & 1;
    vase_ctx::Staged& h = ctx->staged[oldest];
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const vase_config& c = ctx->cfg;
    cudaError_t e;
    for (int32_t l = 0; l < c.num_layers; ++l)
        if (ctx->layers[l].fill + h.n_tokens > ctx->plan.N)
            return fail(ctx, VASE_ERR_FULL, "append would exceed K + B slots");
    if ((e = cudaStreamWaitEvent(s, h.copied, 0)) != cudaSuccess) return cuda_fail(ctx, e, "staging wait");
    // the append reads only the last w_q query rows, so layer l's q pointer sits n - w_q steps before its tail
    const int64_t q_step = static_cast<int64_t>(c.batch) * c.num_q_heads * kRowBytes;
    const void* q = h.base - static_cast<int64_t>(h.n_tokens - h.w_q) * q_step;
    const void* k = h.base + h.w_q * q_step;
    const void* v = static_cast<const uint8_t*>(k) + static_cast<int64_t>(h.n_tokens) * c.batch * c.num_kv_heads * kRowBytes;
    std::vector<int32_t> all(static_cast<size_t>(c.num_layers));
    for (int32_t l = 0; l < c.num_layers; ++l) all[l] = l;
    const int r = append_batch(ctx, all.data(), c.num_layers, q, k, v, h.n_tokens, s, h.block, h.block);
    if (r < 0) return r;
    if ((e = cudaEventRecord(h.consumed, s)) != cudaSuccess) return cuda_fail(ctx, e, "staging event");
    h.consumed_pending = true;
    ctx->staged_count -= 1;
    return r;
}

int vase_read_positions_all(vase_ctx* ctx, int32_t* host_out, void* copy_stream, void* stream) {
    if (!ctx) return VASE_ERR_INVALID;
    if (!host_out) return fail(ctx, VASE_ERR_INVALID, "null output");
    cudaError_t e;
    if ((e = lazy_event(&ctx->evicted)) != cudaSuccess || (e = lazy_event(&ctx->read_done)) != cudaSuccess)
        return cuda_fail(ctx, e, "read-back events");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaStream_t cs = static_cast<cudaStream_t>(copy_stream);
    const Plan& P = ctx->plan;
    const size_t width = static_cast<size_t>(ctx->cfg.budget_k) * 4;
    const size_t rows = static_cast<size_t>(ctx->cfg.num_layers) * P.units;
    if ((e = cudaEventRecord(ctx->evicted, s)) != cudaSuccess || (e = cudaStreamWaitEvent(cs, ctx->evicted, 0)) != cudaSuccess ||
        (e = cudaMemcpy2DAsync(host_out, width, ctx->bufs.positions, static_cast<size_t>(P.N) * 4, width, rows,
                               cudaMemcpyDeviceToHost, cs)) != cudaSuccess ||
        (e = cudaEventRecord(ctx->read_done, cs)) != cudaSuccess)
        return cuda_fail(ctx, e, "positions read-back");
    ctx->read_pending = true;
    return VASE_OK;
}

int vase_get_layer_state(const vase_ctx* ctx, int32_t layer, vase_layer_state* out) {
    if (!ctx || !out || layer < 0 || layer >= ctx->cfg.num_layers) return VASE_ERR_INVALID;
    *out = ctx->layers[layer];
    return VASE_OK;
}

int vase_set_layer_state(vase_ctx* ctx, int32_t layer, const vase_layer_state* st) {
    if (!ctx || !st) return VASE_ERR_INVALID;
    if (!check_layer(ctx, layer)) return fail(ctx, VASE_ERR_INVALID, "layer out of range");
    if (st->fill < 0 || st->fill > ctx->plan.N || st->round < 0 || st->next_position < 0 || st->queries_seen < 0)
        return fail(ctx, VASE_ERR_INVALID, "layer state out of range");
    ctx->layers[layer] = *st;
    return VASE_OK;
}

int vase_kv_view_get(const vase_ctx* ctx, int32_t layer, vase_kv_view* out) {
    if (!ctx || !out || layer < 0 || layer >= ctx->cfg.num_layers) return VASE_ERR_INVALID;
    vase_ctx* c = const_cast<vase_ctx*>(ctx);
    out->k = kc_layer(c, layer);
    out->v = ctx->plan.store ? nullptr : vc_layer(c, layer);  // the store's values: vase_value_store_get
    out->positions = pos_layer(c, layer);
    out->value_scores = c->bufs.value_scores + static_cast<int64_t>(layer) * ctx->plan.units * ctx->plan.N;
    out->unit_stride = static_cast<int64_t>(ctx->plan.N) * kHeadDim;
    out->slots = ctx->plan.N;
    out->fill = ctx->layers[layer].fill;
    return VASE_OK;
}

int vase_value_store_get(const vase_ctx* ctx, int32_t layer, vase_value_store* out) {
    if (!ctx || !out || layer < 0 || layer >= ctx->cfg.num_layers) return VASE_ERR_INVALID;
    const Plan& P = ctx->plan;
    if (!P.store) return VASE_ERR_UNSUPPORTED;
    uint8_t* base = static_cast<uint8_t*>(ctx->bufs.v_cache) + static_cast<size_t>(layer) * P.st_layer_bytes;
    out->codes = base + P.st_codes_off;
    out->sz = reinterpret_cast<float*>(base + P.st_qp_off);
    out->mask = reinterpret_cast<uint32_t*>(base + P.st_mask_off);
    out->ring = base + P.st_ring_off;
    out->state = reinterpret_cast<int32_t*>(base + P.st_state_off);
    out->bits = ctx->cfg.value_bits;
    out->code_row = P.st_code_row;
    out->slots = P.N;
    out->sz_stride = P.st_Np;
    out->mask_stride = P.st_mask_stride;
    out->ring_rows = P.st_H;
    out->units = P.units;
    out->fill = ctx->layers[layer].fill;
    return VASE_OK;
}

int vase_debug_view_get(const vase_ctx* ctx, int32_t slot, vase_debug_view* out) {
    if (!ctx || !out || slot < 0 || slot >= ctx->plan.slots) return VASE_ERR_INVALID;
    const Plan& P = ctx->plan;
    const size_t z = static_cast<size_t>(slot);
    out->attn = reinterpret_cast<float*>(ctx->ws + P.off_attn) + z * P.stride_attn;
    out->pooled = reinterpret_cast<float*>(ctx->ws + P.off_pooled) + z * P.stride_un;
    out->value_score = reinterpret_cast<float*>(ctx->ws + P.off_vscore) + z * P.stride_un;
    out->key = reinterpret_cast<float*>(ctx->ws + P.off_key) + z * P.stride_un;
    out->keep = ctx->ws + P.off_keep + z * P.stride_un;
    out->src = reinterpret_cast<int32_t*>(ctx->ws + P.off_src) + z * P.stride_src;
    out->units = P.units;
    out->slots = P.N;
    out->layer = slot < static_cast<int32_t>(ctx->last_batch.size()) ? ctx->last_batch[slot] : -1;
    return VASE_OK;
}

int vase_check_device_error(vase_ctx* ctx, void* stream, uint32_t* code) {
    if (!ctx) return VASE_ERR_INVALID;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "stream synchronize");
    uint32_t word = 0;
    uint32_t* dev = reinterpret_cast<uint32_t*>(ctx->ws + ctx->plan.off_err);
    if ((e = cudaMemcpy(&word, dev, 4, cudaMemcpyDeviceToHost)) != cudaSuccess) return cuda_fail(ctx, e, "error word read");
    if (code) *code = word;
    if (word) {
        if ((e = cudaMemset(dev, 0, 4)) != cudaSuccess) return cuda_fail(ctx, e, "error word clear");
        char buf[96];
        snprintf(buf, sizeof(buf), "device error word 0x%08x", word);
        return fail(ctx, VASE_ERR_DEVICE, buf);
    }
    return VASE_OK;
}

int vase_self_test_wait_timeout(vase_ctx* ctx, void* stream) {
    if (!ctx) return VASE_ERR_INVALID;
    uint32_t* err = reinterpret_cast<uint32_t*>(ctx->ws + ctx->plan.off_err);
    cudaError_t e = vase::launch_wait_timeout_probe(err, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(ctx, e, "self-test launch");
    ctx->launches += 1;
    return VASE_OK;
}

int64_t vase_launch_count(const vase_ctx* ctx) { return ctx ? ctx->launches : 0; }

int vase_profile_enable(vase_ctx* ctx, int enable) {
    if (!ctx) return VASE_ERR_INVALID;
    ctx->profiling = enable != 0;
    return VASE_OK;
}

int vase_profile_collect(vase_ctx* ctx, double* total_ms, int64_t* launches) {
    if (!ctx || !total_ms || !launches) return VASE_ERR_INVALID;
    for (int k = 0; k < VASE_KERNEL_COUNT; ++k) {
        total_ms[k] = 0.0;
        launches[k] = 0;
    }
    for (size_t i = 0; i < ctx->events_used; ++i) {
        const vase_ctx::EventPair& e = ctx->events[i];
        cudaError_t r = cudaEventSynchronize(e.end);
        float ms = 0.f;
        if (r == cudaSuccess) r = cudaEventElapsedTime(&ms, e.start, e.end);
        if (r != cudaSuccess) {
            ctx->events_used = 0;
            return cuda_fail(ctx, r, "profile events");
        }
        total_ms[e.kind] += ms;
        launches[e.kind] += 1;
    }
    ctx->events_used = 0;
    return VASE_OK;
}

const char* vase_status_string(int status) {
    switch (status) {
        case VASE_OK: return "ok";
        case VASE_EVICT_DUE: return "eviction due";
        case VASE_ERR_INVALID: return "invalid argument";
        case VASE_ERR_FULL: return "cache full";
        case VASE_ERR_NOT_FULL: return "cache not full";
        case VASE_ERR_CUDA: return "CUDA error";
        case VASE_ERR_UNSUPPORTED: return "unsupported configuration";
        case VASE_ERR_ALIGN: return "misaligned pointer";
        case VASE_ERR_DEVICE: return "device-side error";
        default: return "unknown status";
    }
}

const char* vase_last_error(const vase_ctx* ctx) { return ctx ? ctx->last_error.c_str() : g_config_error.c_str(); }

int vase_abi_version(void) { return VASE_ABI_VERSION; }

}  // extern "C"

// ----------------------------------------------------------------------------------------------------------------
// Eviction without a caller-provided workspace.
//
// Some callers of this library never hold an allocator: a plugin inside an inference server whose host process
// owns all device memory and only hands it tensors, or a runtime that forbids device allocation after start-up
// to keep a fixed, unfragmented memory budget.  They can provide the caches but not the eviction's scratch.  For
// them vase_evict_static_scratch runs the same kernels with their scratch (window scores, DKV leverage products,
// kept-slot lists, the device error word) in the file-scope array below, which every GPU that loads the library
// holds until the process exits.  Nothing is allocated per call.
namespace {

constexpr size_t kStaticScratchBytes = static_cast<size_t>(VASE_STATIC_SCRATCH_BYTES);
__device__ __align__(256) uint8_t g_static_scratch[kStaticScratchBytes];

constexpr int kMaxDevices = 64;
void* g_static_scratch_addr[kMaxDevices] = {};  // device address of g_static_scratch, per device

// Host set-up of the previous call (tensor maps, kernel attributes), reused while nothing it depends on changed.
struct StaticScratchSetup {
    bool valid = false;
    int device = -1;
    vase_config cfg;
    const void* k = nullptr;
    const void* v = nullptr;
    const void* q = nullptr;
    CUtensorMap kmap, vmap, qmap;
};
StaticScratchSetup g_static_setup;

}  // namespace

extern "C" int vase_evict_static_scratch(const vase_config* cfg, const vase_buffers* bufs, int32_t layer,
                                         const vase_layer_state* state, uint32_t* device_error, void* stream) {
    if (!cfg || !bufs || !state) {
        g_config_error = "null argument";
        return VASE_ERR_INVALID;
    }
    int device = 0, num_sms = 0;
    cudaError_t e = cudaGetDevice(&device);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&num_sms, cudaDevAttrMultiProcessorCount, device);
    if (e != cudaSuccess || device < 0 || device >= kMaxDevices) {
        g_config_error = "no usable CUDA device";
        return VASE_ERR_CUDA;
    }
    Plan P;
    const char* why = nullptr;
    if (!make_plan(cfg, num_sms, &P, &why)) return cfg->head_dim != 128 ? VASE_ERR_UNSUPPORTED : VASE_ERR_INVALID;
    const vase_config& c = *cfg;
    if (P.store) {
        g_config_error = "the static-scratch eviction works on the bf16 value cache (value_bits = 0)";
        return VASE_ERR_UNSUPPORTED;
    }
    if (layer < 0 || layer >= c.num_layers) {
        g_config_error = "layer out of range";
        return VASE_ERR_INVALID;
    }
    // scratch of one layer: error word | window-score parts | DKV products | kept lists (a property of the
    // configuration alone, so it is checked before anything else is looked at)
    const size_t un = static_cast<size_t>(P.units) * P.N;
    const size_t off_attn = kAlign;
    const size_t off_dkv = align_up(off_attn + un * 4 * P.n_rb, kAlign);
    const size_t off_src = align_up(off_dkv + un * 4, kAlign);
    const size_t need = align_up(off_src + static_cast<size_t>(P.units) * c.budget_k * 4, kAlign);
    if (need > kStaticScratchBytes) {
        g_config_error = "one layer needs " + std::to_string(need) +
                         " bytes of eviction scratch, more than the static array holds (VASE_STATIC_SCRATCH_BYTES = " +
                         std::to_string(kStaticScratchBytes) + ")";
        return VASE_ERR_UNSUPPORTED;
    }
    if (state->fill != P.N) {
        g_config_error = "evict needs a full cache (fill == K + B)";
        return VASE_ERR_NOT_FULL;
    }
    const void* ptrs[5] = {bufs->k_cache, bufs->v_cache, bufs->q_window, bufs->positions, bufs->value_scores};
    for (const void* p : ptrs) {
        if (!p || !aligned(p, kAlign)) {
            g_config_error = "null or unaligned buffer (256-byte alignment required)";
            return p ? VASE_ERR_ALIGN : VASE_ERR_INVALID;
        }
    }
    // set-up, once per device, with that device current: the device address of the static array.  With lazy
    // module loading (the CUDA default) this is also where the array is committed on the device.
    if (!g_static_scratch_addr[device]) {
        void* addr = nullptr;
        if ((e = cudaGetSymbolAddress(&addr, g_static_scratch)) != cudaSuccess || !addr) {
            g_config_error = e == cudaErrorMemoryAllocation
                                 ? "out of device memory while loading the static scratch array (first call on this "
                                   "device): make the first call at start-up, or set CUDA_MODULE_LOADING=EAGER"
                                 : std::string("cudaGetSymbolAddress: ") + cudaGetErrorString(e);
            return VASE_ERR_CUDA;
        }
        g_static_scratch_addr[device] = addr;
    }
    uint8_t* scratch = static_cast<uint8_t*>(g_static_scratch_addr[device]);
    uint32_t* err = reinterpret_cast<uint32_t*>(scratch);
    float* attn = reinterpret_cast<float*>(scratch + off_attn);
    float* dkv = reinterpret_cast<float*>(scratch + off_dkv);
    int32_t* src = reinterpret_cast<int32_t*>(scratch + off_src);

    // Tensor maps and kernel attributes: reused while the device, the configuration and the buffers are those of
    // the previous call (a serving loop evicts the same caches over and over).
    StaticScratchSetup& su = g_static_setup;
    if (!(su.valid && su.device == device && std::memcmp(&su.cfg, &c, sizeof(c)) == 0 &&
          su.k == bufs->k_cache && su.v == bufs->v_cache && su.q == bufs->q_window)) {
        su.valid = false;
        void* fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
        if (e != cudaSuccess || !fn || q != cudaDriverEntryPointSuccess) {
            g_config_error = "cuTensorMapEncodeTiled unavailable";
            return VASE_ERR_CUDA;
        }
        EncodeTiledFn enc = reinterpret_cast<EncodeTiledFn>(fn);
        const uint64_t cache_rows = static_cast<uint64_t>(c.num_layers) * P.units * P.N;
        const uint64_t q_rows = static_cast<uint64_t>(c.num_layers) * c.batch * c.num_q_heads * c.window;
        if (cache_rows >= (1ull << 31) || q_rows >= (1ull << 31) ||
            !encode_rows(enc, &su.kmap, bufs->k_cache, cache_rows, kTileTokens) ||
            !encode_rows(enc, &su.vmap, bufs->v_cache, cache_rows, kTileTokens) ||
            !encode_rows(enc, &su.qmap, bufs->q_window, q_rows, static_cast<uint32_t>(P.q_box))) {
            g_config_error = "tensor map encoding failed";
            return VASE_ERR_CUDA;
        }
        if ((e = score_attn_set_attributes(P.score_smem, P.cluster)) != cudaSuccess ||
            (e = dkv_set_attributes(P.dkv_smem)) != cudaSuccess ||
            (e = select_set_attributes(P.select_smem)) != cudaSuccess) {
            g_config_error = std::string("kernel attributes: ") + cudaGetErrorString(e);
            return VASE_ERR_CUDA;
        }
        su.device = device;
        su.cfg = c;
        su.k = bufs->k_cache;
        su.v = bufs->v_cache;
        su.q = bufs->q_window;
        su.valid = true;
    }
    const CUtensorMap& kmap = su.kmap;
    const CUtensorMap& vmap = su.vmap;
    const CUtensorMap& qmap = su.qmap;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    // The error word is not cleared here: the kernels OR their failure sites into it, and it is read and cleared
    // only by a call that reports it (device_error != NULL), so a failure of a call made with device_error == NULL
    // is reported by the next call that asks.  Every other part of the array is written before it is read.
    LayerBatch batch;
    batch.n = 1;
    batch.layer[0] = layer;
    batch.rnd[0] = state->round;
    if (c.variant == VASE_VARIANT_ATTNV) {
        const ScoreAttnParams sp = score_params(P, c, batch, 1, attn, err);
        if ((e = launch_score_attn(kmap, qmap, sp, P.score_smem, s)) != cudaSuccess) {
            g_config_error = std::string("score launch: ") + cudaGetErrorString(e);
            return VASE_ERR_CUDA;
        }
    } else {
        DkvParams dp{};
        dp.batch = batch;
        dp.N = P.N;
        dp.K = c.budget_k;
        dp.r = c.dkv_rank;
        dp.Hkv = c.num_kv_heads;
        dp.fixed_g = c.dkv_fixed_g;
        dp.shared_g = c.dkv_shared_g;
        dp.units = P.units;
        dp.seed_lo = static_cast<uint32_t>(c.seed & 0xFFFFFFFFull);
        dp.seed_hi = static_cast<uint32_t>(c.seed >> 32);
        dp.n_tiles_k = P.dkv_tiles_k;
        dp.tiles_per_cta = P.dkv_tiles_per_cta;
        dp.stages = P.dkv_stages;
        dp.layer_rows = static_cast<int64_t>(P.units) * P.N;
        dp.out = dkv;
        dp.err = err;
        if ((e = launch_dkv(kmap, vmap, dp, P.units, P.dkv_smem, s)) != cudaSuccess) {
            g_config_error = std::string("dkv launch: ") + cudaGetErrorString(e);
            return VASE_ERR_CUDA;
        }
    }
    SelectParams sel{};  // value-initialised: a field this path does not set is zero (pointers null)
    sel.batch = batch;
    sel.attn = attn;
    sel.dkv = dkv;
    sel.vmag = bufs->value_scores;
    sel.vscore_dbg = nullptr;
    sel.pos = bufs->positions;
    sel.kc = static_cast<uint4*>(bufs->k_cache);
    sel.vc = static_cast<uint4*>(bufs->v_cache);
    sel.src = src;
    sel.pooled_dbg = nullptr;
    sel.key_dbg = nullptr;
    sel.keep_dbg = nullptr;
    sel.N = P.N;
    sel.K = c.budget_k;
    sel.B = c.buffer_b;
    sel.n_v = P.n_v;
    sel.m = P.m;
    sel.pool = c.pool_kernel;
    sel.variant = c.variant;
    sel.stochastic = c.stochastic;
    sel.Hkv = c.num_kv_heads;
    sel.n_parts = c.variant == VASE_VARIANT_ATTNV ? P.n_rb : 1;
    sel.staged = P.select_staged ? 1 : 0;
    sel.reserve_random = c.reserve_kind == VASE_RESERVE_RANDOM ? 1 : 0;
    sel.gqa_max = c.gqa_reduce == VASE_GQA_MAX ? 1 : 0;
    sel.units = P.units;
    sel.seed_lo = static_cast<uint32_t>(c.seed & 0xFFFFFFFFull);
    sel.seed_hi = static_cast<uint32_t>(c.seed >> 32);
    sel.err = err;
    if ((e = launch_select(sel, P.units, P.select_smem, P.select_threads, s)) != cudaSuccess) {
        g_config_error = std::string("select launch: ") + cudaGetErrorString(e);
        return VASE_ERR_CUDA;
    }
    if (device_error) {
        if ((e = cudaMemcpyAsync(device_error, err, sizeof(uint32_t), cudaMemcpyDeviceToHost, s)) != cudaSuccess ||
            (e = cudaStreamSynchronize(s)) != cudaSuccess) {
            g_config_error = std::string("error word read: ") + cudaGetErrorString(e);
            return VASE_ERR_CUDA;
        }
        if (*device_error) {
            // reported: clear it, so that the next call starts from zero
            if ((e = cudaMemsetAsync(err, 0, sizeof(uint32_t), s)) != cudaSuccess ||
                (e = cudaStreamSynchronize(s)) != cudaSuccess) {
                g_config_error = std::string("error word clear: ") + cudaGetErrorString(e);
                return VASE_ERR_CUDA;
            }
            char buf[128];
            snprintf(buf, sizeof(buf),
                     "device-side check or bounded wait failed (word 0x%08x, this call or an earlier one made "
                     "without device_error)",
                     *device_error);
            g_config_error = buf;
            return VASE_ERR_DEVICE;
        }
    }
    return VASE_OK;
}
