/*
 * vase.h -- C ABI of the VaSE eviction step on one GPU (sm_103a).
 *
 * VaSE (Value-aware Stochastic KV cache Eviction, arXiv 2606.03928) runs a
 * periodic eviction step on each layer's KV cache (Sec. 2, "Periodic eviction
 * with budget K and buffer B"): every decode step appends one (k, v) pair per
 * KV head; once the cache holds N = K + B pairs the eviction step keeps the B
 * most recent pairs, scores the other K candidates, drops B of them and
 * compacts the cache back to K slots.  The scores and the rule are those of
 * Sec. 3.2: VaSE-AttnV (window attention score, Eq. (2), with N_v slots
 * reserved for the largest value magnitudes, Eq. (5), and weighted sampling
 * without replacement for the rest) and VaSE-DKV (CurDKV leverage scores,
 * Eq. (4), under a Gaussian projection redrawn every round).
 *
 * Conventions shared by every entry point:
 *   - Every pointer named "device" is a CUDA device pointer owned by the
 *     caller; the library never allocates or frees device memory and never
 *     synchronises a stream except in vase_check_device_error.
 *   - "stream" is a cudaStream_t passed as void* (NULL = legacy default stream).
 *     All work is enqueued on it in call order; every call on one context
 *     must be ordered on one stream (the workspace is shared by all layers).
 *   - bf16 tensors are row-major with head_dim = 128 contiguous elements
 *     (256 bytes) per row; every device base pointer must be 256-byte aligned.
 *   - Return values: VASE_OK (0), VASE_EVICT_DUE (> 0, informational) or a
 *     negative VASE_ERR_* code.  On error nothing is enqueued and the
 *     context's counters are unchanged; vase_last_error() explains.
 *   - A context is not thread-safe.
 */
#ifndef VASE_H
#define VASE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define VASE_ABI_VERSION 3

#define VASE_OK 0
#define VASE_EVICT_DUE 1          /* the layer's cache is full: call vase_evict before the next append */
#define VASE_ERR_INVALID (-1)     /* bad argument or configuration */
#define VASE_ERR_FULL (-2)        /* append would exceed K + B slots */
#define VASE_ERR_NOT_FULL (-3)    /* evict called before the cache holds K + B pairs */
#define VASE_ERR_CUDA (-4)        /* a CUDA runtime call failed (message in vase_last_error) */
#define VASE_ERR_UNSUPPORTED (-5) /* valid but outside what the kernels implement (e.g. head_dim != 128) */
#define VASE_ERR_ALIGN (-6)       /* a device pointer is not 256-byte aligned */
#define VASE_ERR_DEVICE (-7)      /* a device-side check or bounded wait failed (vase_check_device_error) */

#define VASE_VARIANT_ATTNV 0      /* Sec. 3.2, VaSE-AttnV */
#define VASE_VARIANT_DKV 1        /* Sec. 3.2, VaSE-DKV */

#define VASE_VALUE_RANGE 0        /* Eq. (5): max_j v_j - min_j v_j */
#define VASE_VALUE_L2 1           /* App. A: ||v||_2 */
#define VASE_VALUE_VAR 2          /* App. A: (1/d) sum_j (v_j - mean)^2 */

#define VASE_RESERVE_VALUE 0      /* R_V = the N_v candidates of largest value magnitude (Sec. 3.1) */
#define VASE_RESERVE_RANDOM 1     /* R_V = N_v candidates drawn uniformly at random (the ablation of App. C) */

#define VASE_GQA_MEAN 0           /* window score of a KV head: mean over its G query heads' G*W window rows */
#define VASE_GQA_MAX 1            /* ... the largest over its G query heads of each head's mean over W rows */

typedef struct vase_config {
    int32_t budget_k;      /* K: persistent budget (Sec. 2) */
    int32_t buffer_b;      /* B: recency buffer, always kept (Sec. 2) */
    int32_t window;        /* W: cached decode queries per query head (Eq. (2) footnote; the paper uses W = B) */
    int32_t num_q_heads;   /* Hq */
    int32_t num_kv_heads;  /* Hkv; Hq % Hkv == 0, query head j reads KV head j / (Hq / Hkv) */
    int32_t head_dim;      /* d; must be 128 */
    int32_t num_layers;    /* L */
    int32_t batch;         /* b: sequences */
    int32_t variant;       /* VASE_VARIANT_* */
    int32_t n_v;           /* N_v value-reserved slots (AttnV); -1 = K/4 (App. B) */
    int32_t value_score;   /* VASE_VALUE_*: the value magnitude used for R_V (AttnV) */
    int32_t pool_kernel;   /* odd average-pooling width over the slot axis (Eq. (2) footnote); 1 = off */
    int32_t dkv_rank;      /* r of G in R^{d x r} (Eq. (4)); 1..32, 20 in App. B */
    int32_t stochastic;    /* AttnV: 1 = weighted sampling without replacement (Sec. 3.2), 0 = top-k (Sec. 4.1) */
    int32_t dkv_fixed_g;   /* DKV: 1 = one G for the whole stream (CurDKV), 0 = G_t redrawn per round (VaSE-DKV) */
    int32_t debug_outputs; /* 1 = also write pooled scores, selection keys and the keep mask to the workspace */
    uint64_t seed;         /* key of the Philox4x32-10 noise stream */
    int32_t reserve_kind;  /* AttnV: VASE_RESERVE_* (how R_V is chosen) */
    int32_t gqa_reduce;    /* AttnV: VASE_GQA_*; VASE_GQA_MAX needs W % 4 == 0 and, when G*W > 256, 256 % W == 0 */
    int32_t dkv_shared_g;  /* DKV: 1 = one G per round shared by every layer, sequence and KV head; 0 = per unit */
    int32_t value_bits;    /* AttnV: 0 = bf16 value cache; 2, 4 or 8 = the compressed value store (below) */
} vase_config;

/* Sizes in bytes of the caller-allocated device buffers for a configuration. */
typedef struct vase_buffer_sizes {
    size_t k_cache;    /* bf16 [L][b][Hkv][K+B][d] */
    size_t v_cache;    /* bf16 [L][b][Hkv][K+B][d]; with value_bits > 0 the compressed value store of every layer */
    size_t q_window;   /* bf16 [L][b][Hq][W][d], a ring over the last W decode queries */
    size_t positions;  /* int32 [L][b][Hkv][K+B], absolute stream position of each slot, -1 if empty */
    size_t value_scores; /* fp32 [L][b][Hkv][K+B], value magnitude of the token in each slot */
    size_t workspace;  /* scratch for one eviction at a time plus the host-append staging area */
} vase_buffer_sizes;

typedef struct vase_buffers {
    void* k_cache;     /* device */
    void* v_cache;     /* device */
    void* q_window;    /* device */
    int32_t* positions;/* device */
    float* value_scores; /* device; filled by the appends, moved by the evictions */
    void* workspace;   /* device; contents are the library's between calls */
} vase_buffers;

/* Per-layer host counters: everything besides the buffers that a resume needs. */
typedef struct vase_layer_state {
    int32_t fill;          /* occupied slots, 0..K+B */
    int32_t round;         /* evictions done so far (keys the noise of the next one) */
    int64_t next_position; /* stream position of the next appended token */
    int64_t queries_seen;  /* queries appended so far (ring write index = queries_seen % W) */
} vase_layer_state;

/* Where a decode attention kernel finds one layer's cache after eviction. */
typedef struct vase_kv_view {
    void* k;               /* device, bf16; row (s, h, slot) at k + ((s*Hkv + h)*unit_stride + slot)*d */
    void* v;
    int32_t* positions;
    float* value_scores;   /* per slot, same layout as positions */
    int64_t unit_stride;   /* elements between consecutive (s, h) units = (K+B)*d */
    int32_t slots;         /* K + B */
    int32_t fill;          /* valid slots 0..fill-1, in stream order */
} vase_kv_view;

/* Device pointers to the workspace results of one layer of the most recent eviction call
 * (valid until the next one).  Slot z is the z-th layer that call evicted (0 for vase_evict). */
typedef struct vase_debug_view {
    float* attn;           /* [b*Hkv][K+B] window score before pooling (AttnV) */
    float* pooled;         /* [b*Hkv][K+B] pooled score (AttnV, debug_outputs) */
    float* value_score;    /* [b*Hkv][K+B] Range/L2/Var (AttnV) or leverage product s_i (DKV), slots < K */
    float* key;            /* [b*Hkv][K+B] selection key per candidate, -1 if not a candidate (debug_outputs) */
    uint8_t* keep;         /* [b*Hkv][K+B] 1 = kept (debug_outputs) */
    int32_t* src;          /* [b*Hkv][K] ascending kept slots: new slot j holds old slot src[j] */
    int32_t units;         /* b*Hkv */
    int32_t slots;         /* K + B */
    int32_t layer;         /* the layer whose eviction these are, -1 if the slot was not used */
} vase_debug_view;

typedef struct vase_ctx vase_ctx;

/* Fills *cfg with the paper's defaults (App. B): n_v = -1 (K/4), r = 20, pool 7,
 * stochastic, fresh G per round, Range value score.  Geometry fields are zeroed. */
void vase_config_default(vase_config* cfg);

/* Validates *cfg and reports the buffer sizes it needs.  No device work.  The caches
 * hold N = K + B slots per (layer, sequence, KV head) -- the budget K and buffer B of
 * Sec. 2's periodic eviction -- and the window ring the W cached decode queries per
 * query head that Eq. (2) and its footnote score against.  Errors: VASE_ERR_INVALID
 * (inconsistent configuration; vase_last_error(NULL) says which check),
 * VASE_ERR_UNSUPPORTED (head_dim != 128). */
int vase_get_buffer_sizes(const vase_config* cfg, vase_buffer_sizes* out);

/* Creates a context over caller-owned buffers (sizes from vase_buffer_sizes): the
 * per-layer KV caches of budget K plus buffer B that Sec. 2's periodic eviction works
 * on.  Reads the current CUDA device; encodes the TMA descriptors of the caches.
 * Every layer starts empty (fill 0, round 0).  The buffers are not cleared and stay
 * the caller's; the context keeps only pointers.  Errors: VASE_ERR_INVALID (bad
 * configuration or null buffer), VASE_ERR_ALIGN (a buffer not 256-byte aligned),
 * VASE_ERR_UNSUPPORTED, VASE_ERR_CUDA; *out is NULL then. */
int vase_create(const vase_config* cfg, const vase_buffers* bufs, vase_ctx** out);

/* Frees the context's host state.  Caller memory is untouched.  NULL is a no-op. */
void vase_destroy(vase_ctx* ctx);

/* Appends n_tokens consecutive decode steps of one layer (Sec. 2: each decode
 * step adds one pair per KV head).  Device inputs, row-major:
 *   q [n_tokens][b][Hq][d], k and v [n_tokens][b][Hkv][d]  (bf16).
 * q goes to the window ring, k and v to slots fill..fill+n_tokens-1 with their
 * stream positions.  Only the last min(W, n_tokens) query rows are read (the
 * ring keeps no others); the rows before them need not hold data.  Returns
 * VASE_EVICT_DUE when the layer becomes full, VASE_ERR_FULL (nothing written)
 * when fill + n_tokens > K + B. */
int vase_append(vase_ctx* ctx, int32_t layer, const void* q, const void* k, const void* v,
                int32_t n_tokens, void* stream);

/* vase_append for every layer at once, in one launch: q [L][n_tokens][b][Hq][d],
 * k and v [L][n_tokens][b][Hkv][d] (device, bf16).  All layers must have room. */
int vase_append_all(vase_ctx* ctx, const void* q, const void* k, const void* v, int32_t n_tokens, void* stream);

/* vase_append_all with the layers' inputs at any fixed distance: layer l's
 * [n_tokens][b][Hq][d] query rows start at q + l * q_layer_stride bytes and its
 * [n_tokens][b][Hkv][d] key and value rows at k + l * kv_layer_stride and
 * v + l * kv_layer_stride (device, bf16).  As in vase_append only the last
 * min(W, n_tokens) query rows of each layer are read, so a layer's block may
 * hold its query tail alone (q pointing W rows before it) next to its keys and
 * values, and one copy can bring every layer's inputs.  Strides must be positive
 * multiples of 16 bytes (VASE_ERR_INVALID / VASE_ERR_ALIGN otherwise, nothing
 * written); all layers must have room (VASE_ERR_FULL). */
int vase_append_all_strided(vase_ctx* ctx, const void* q, const void* k, const void* v, int32_t n_tokens,
                            int64_t q_layer_stride, int64_t kv_layer_stride, void* stream);

/* Same as vase_append with HOST inputs (at most B tokens per call).  Page-locked
 * inputs (pinned or registered) are read by the append kernel in place over the
 * host link, asynchronously on `stream`; other host memory is first copied into
 * the staging area of the workspace.  Either way only the query rows of the last
 * W steps cross (earlier queries never reach the window ring).  As with
 * cudaMemcpyAsync, the inputs must stay unchanged until the stream has run the
 * append. */
int vase_append_host(vase_ctx* ctx, int32_t layer, const void* q_host, const void* k_host,
                     const void* v_host, int32_t n_tokens, void* stream);

/* One eviction step of one layer (Sec. 2 and Sec. 3.2): requires fill == K+B;
 * afterwards fill == K, round += 1, slots 0..K-1 hold the kept pairs in stream
 * order and positions of slots K..K+B-1 are -1. */
int vase_evict(vase_ctx* ctx, int32_t layer, void* stream);

/* The eviction step of every full layer (all layers fill at the same decode step), batched:
 * each kernel covers up to 64 layers per launch.  Returns the number of layers evicted (>= 0)
 * or a negative error. */
int vase_evict_all(vase_ctx* ctx, void* stream);

/* One whole step of the periodic eviction (Sec. 2): vase_append_all_strided of
 * n_tokens decode steps (arguments, layout, checks and errors as there), then
 * vase_evict_all, with the same results.  Where the append makes every layer full
 * and the eviction of all of them fits one wave of the fused small-unit kernel
 * (AttnV, bf16 values, one CTA per unit), both run in that kernel's one launch:
 * each CTA appends its unit's key, value and window-query rows, then scores,
 * selects and compacts the unit.  Returns the number of layers evicted (>= 0) or
 * a negative error.  If the fused launch itself fails (VASE_ERR_CUDA) the layers'
 * states already count the append. */
int vase_append_evict_all(vase_ctx* ctx, const void* q, const void* k, const void* v, int32_t n_tokens,
                          int64_t q_layer_stride, int64_t kv_layer_stride, void* stream);

/* The value magnitude (Range, L2 or Var of the value row, Eq. (5) / App. A) of every cached
 * token is computed once, by the append that writes the row, and kept per slot in
 * value_scores; the AttnV eviction reads it instead of the V cache.  A caller that writes
 * V rows directly (restoring a checkpoint, say) recomputes slots 0..fill-1 of one layer
 * with this call. */
int vase_refresh_value_scores(vase_ctx* ctx, int32_t layer, void* stream);

/* Attention output of one decode step over the pairs the cache holds now (Eq. (1), Sec. 2):
 * for every sequence and query head, o = sum_i alpha_i v_i with alpha_i the softmax of
 * q . k_i / sqrt(d) over slots 0..fill-1 of the query head's KV head (GQA: query head
 * g*G + j reads KV head g).  This is the consumer of the layout the eviction keeps, read
 * in place.  q: device, bf16 [b][Hq][d], 16-byte aligned; out: device, fp32 [b][Hq][d].
 * The caller owns q and out; the call uses no workspace (the slots of each KV head are split
 * over the CTAs of one thread-block cluster, whose states are folded in shared memory), so
 * calls may overlap with each other but not with an append or eviction of the same layer.
 * With the compressed value store (value_bits > 0) the values are read from it on the tensor cores: bf16 rows
 * from the reserved ring, every other value as Q s + z from its codes.
 * Errors: VASE_ERR_INVALID (bad layer, null pointer, empty layer), VASE_ERR_ALIGN,
 * VASE_ERR_UNSUPPORTED (more than 16 query heads per KV head). */
int vase_decode_attention(vase_ctx* ctx, int32_t layer, const void* q, float* out, void* stream);

/* ---- Mixed-precision values: the b-bit per-token quantizer of Sec. 4.4 and the reserved cache of Sec. 6.
 * After an eviction the reserved values -- R_V (the N_v largest value magnitudes) and the recency buffer
 * R_B -- keep their bf16 rows; every other kept value is read back from b-bit codes (b = 2, 4 or 8):
 * z = min v, s = Range(v) / (2^b - 1), Q = round((v - z) / s) (half to even, decided in fp32),
 * v' = Q s + z.  The bf16 cache stays the record the evictions work on; the codes serve the decode reads.
 * The caller owns these buffers, one set per layer, all device memory: */
typedef struct vase_mixed_buffers {
    void* codes;      /* uint8 [b][Hkv][K][d * bits / 8]: lane-packed codes, dims 4i .. 4i+3 in 4*bits bits */
    float* qparams;   /* fp32 [b][Hkv][Kp][2], Kp = K rounded up to even: (s, z) of each quantized slot */
    uint32_t* rmask;  /* [b][Hkv][ceil(K / 32)]: bit t of word w set = slot 32 w + t keeps its bf16 value */
    void* hp_rows;    /* bf16 [b][Hkv][N_v + B][d]: the reserved cache, the bf16 rows of the reserved slots in
                         slot order (N_v = 0 for DKV) */
} vase_mixed_buffers;

/* Sizes in bytes of the four buffers of one layer (NULL outputs are skipped). */
int vase_mixed_buffer_sizes(const vase_config* cfg, int32_t bits, size_t* codes, size_t* qparams, size_t* rmask,
                            size_t* hp_rows);

/* Writes the codes, parameters and reserved mask of `layer` right after its eviction (fill == K); the
 * codes serve vase_decode_attention_mixed until the layer's next eviction.  Errors: VASE_ERR_INVALID (bad
 * layer or bits, null buffers, fill != K or no eviction yet), VASE_ERR_UNSUPPORTED (reserve_kind random:
 * its R_V is not a function of the kept values), VASE_ERR_ALIGN (buffers not 16-byte aligned). */
int vase_quantize_values(vase_ctx* ctx, int32_t layer, int32_t bits, const vase_mixed_buffers* mb, void* stream);

/* vase_decode_attention with the values of unreserved slots below K read from the codes of the layer's
 * current round (slots appended since the eviction and reserved slots read bf16).  Errors as
 * vase_decode_attention, plus VASE_ERR_INVALID when the codes were not written for this round and bits. */
int vase_decode_attention_mixed(vase_ctx* ctx, int32_t layer, int32_t bits, const vase_mixed_buffers* mb,
                                const void* q, float* out, void* stream);

/* Copies the K positions of every unit of one layer to host memory
 * (int32 [b][Hkv][K]), enqueued on the stream; the host buffer is valid after
 * the stream completes. */
int vase_read_positions(vase_ctx* ctx, int32_t layer, int32_t* host_out, void* stream);

/* ---- Host-buffer pipeline: a decode loop whose inputs and results live in host memory.
 *
 * Sec. 2's loop appends one (q, k, v) per decode step and evicts every B steps; here one call
 * stages a whole round's inputs (n_tokens <= B steps of every layer) from host memory, the next
 * appends them, and the kept positions go back to the host after the eviction.  The copies run on
 * a caller-given copy stream, so the copies of round r + 1 overlap the kernels of round r when the
 * caller stages r + 1 before it appends r:
 *     stage(r = 0); for r: { stage(r + 1); append_all_staged; evict_all; read_positions_all }
 * The library records events to order the two streams; it allocates no device memory (the caller
 * passes the staging buffer).  For the copies to be asynchronous the host inputs and outputs must
 * be page-locked (pinned or registered). */

/* Bytes of ONE staged step for n_tokens per layer: per layer, the last min(W, n_tokens) query
 * rows and the n_tokens key and value rows, each layer's block rounded up to 256 bytes.  The
 * staging buffer of vase_stage_host_inputs holds two steps (2 x this).  0 for a bad config. */
size_t vase_host_staging_bytes(const vase_config* cfg, int32_t n_tokens);

/* Enqueues on copy_stream the host-to-device copies of one step's inputs of every layer into the
 * next half of `staging` (device, 256-byte aligned, >= 2 x vase_host_staging_bytes(cfg, n_tokens)
 * bytes, caller-owned; pass the same buffer on every call).  Host inputs, bf16 rows of 256 bytes:
 * layer l's q [n_tokens][b][Hq][d] at q_host + l * q_layer_stride bytes, its k and v
 * [n_tokens][b][Hkv][d] at k_host / v_host + l * kv_layer_stride.  Only the query rows of the last
 * min(W, n_tokens) steps are copied (the window ring keeps no others), so a layer's host block may
 * hold its query tail alone (q_host pointing n_tokens - min(W, n_tokens) steps before it, a stride of
 * at least the tail; strides are multiples of 16 bytes).  A half is refilled only
 * after the append that read it has run (the copy stream waits for it).  At most two steps can be
 * staged and not yet appended (VASE_ERR_FULL otherwise).  The host inputs may change once
 * copy_stream has run the copies.  Errors: VASE_ERR_INVALID (null pointer, n_tokens outside
 * 1..B, strides smaller than a layer's inputs, staging too small), VASE_ERR_ALIGN, VASE_ERR_FULL,
 * VASE_ERR_CUDA. */
int vase_stage_host_inputs(vase_ctx* ctx, const void* q_host, const void* k_host, const void* v_host,
                           int32_t n_tokens, int64_t q_layer_stride, int64_t kv_layer_stride, void* staging,
                           size_t staging_bytes, void* copy_stream);

/* Appends the oldest staged step to every layer on `stream` (vase_append_all from the staging
 * buffer; `stream` first waits for that step's copies).  Returns as vase_append_all
 * (VASE_EVICT_DUE when the layers become full), VASE_ERR_INVALID when nothing is staged. */
int vase_append_all_staged(vase_ctx* ctx, void* stream);

/* Copies the K positions of every unit of every layer (int32 [L][b][Hkv][K]) to host_out on
 * copy_stream, after everything enqueued on `stream` so far (call it after vase_evict_all).  The
 * next eviction on this context waits for the copy, so the positions it reads cannot move under
 * it.  host_out is valid once copy_stream has run the copy. */
int vase_read_positions_all(vase_ctx* ctx, int32_t* host_out, void* copy_stream, void* stream);

int vase_get_layer_state(const vase_ctx* ctx, int32_t layer, vase_layer_state* out);
/* Sets one layer's counters (resume from a checkpoint, or tests that write the buffers directly). */
int vase_set_layer_state(vase_ctx* ctx, int32_t layer, const vase_layer_state* st);

/* Where a decode kernel reads one layer's kept pairs (slots 0..fill-1 in stream order, the
 * layout Sec. 2's compaction back to K slots leaves).  Host call, no device work. */
int vase_kv_view_get(const vase_ctx* ctx, int32_t layer, vase_kv_view* out);
/* Device pointers to the intermediate results of the most recent eviction call: the window
 * score of Eq. (2) before and after pooling, the value magnitudes of Eq. (5) (or the DKV
 * products of Eq. (4)), the selection keys of Sec. 3.2 and the kept list.  The arrays stay
 * in the workspace; the caller copies what it needs before the next eviction. */
int vase_debug_view_get(const vase_ctx* ctx, int32_t slot, vase_debug_view* out);

/* ---- Compressed value store (value_bits = 2, 4 or 8; AttnV only).  The mixed-precision value cache that Sec. 6
 * proposes, built on the per-token asymmetric b-bit quantizer of Sec. 4.4 (z = min v, s = Range(v) / (2^b - 1),
 * Q = round((v - z) / s) half to even, decided in fp32, v' = Q s + z).  Keys stay in the bf16 K cache; a value is
 * held either as a bf16 row in the unit's reserved cache or as its codes:
 *   - the reserved cache is a ring of H = N_v + 2B rows: R_V and R_B after an eviction (Sec. 3.1 and Sec. 2, at
 *     most N_v + B values) and the B values appended before the next eviction;
 *   - every appended value enters the ring in bf16; an append that finds the ring full quantizes its earliest
 *     value into the codes (the rule of Sec. 6), which happens only before the layer's first eviction;
 *   - an eviction moves the kept values with their slots and quantizes the kept bf16 values that are not in the
 *     new R_V u R_B (a quantized value never returns to bf16).
 * The V buffer holds, per layer (layer stride and offsets in vase_value_store), for each of the b*Hkv units:
 * codes uint8 [K+B][16 b] (lane-packed: dims 4i .. 4i+3 in 4b bits at byte i*b/2), (s, z) fp32 [sz_stride][2],
 * mask uint32 [mask_stride] (bit t of word w set = slot 32 w + t is held in bf16), ring bf16 [H][d] (the bf16
 * values in slot order, the i-th at row (head + i) mod H), state int32 [4] = (head, count, 0, 0).  The library
 * writes all of it; the first append of a layer (fill 0) starts it empty.  vase_decode_attention reads it;
 * vase_kv_view_get reports v = NULL.  Not available in this mode (VASE_ERR_UNSUPPORTED): the DKV variant (its
 * score reads every value each round), vase_refresh_value_scores, vase_quantize_values,
 * vase_decode_attention_mixed (the bf16-cache read path) and vase_evict_static_scratch. */
typedef struct vase_value_store {
    uint8_t* codes;        /* device, layer's [units][slots][code_row] */
    float* sz;             /* device, [units][sz_stride][2] */
    uint32_t* mask;        /* device, [units][mask_stride] */
    void* ring;            /* device, bf16 [units][ring_rows][d] */
    int32_t* state;        /* device, [units][4]: ring head, ring count */
    int32_t bits, code_row, slots, sz_stride, mask_stride, ring_rows, units, fill;
} vase_value_store;

/* Device pointers to one layer's compressed value store.  Errors: VASE_ERR_INVALID (null or bad layer),
 * VASE_ERR_UNSUPPORTED (value_bits = 0). */
int vase_value_store_get(const vase_ctx* ctx, int32_t layer, vase_value_store* out);

/* Synchronises the stream, then reads and clears the device error word that
 * bounded waits and device-side checks set.  Returns VASE_OK or VASE_ERR_DEVICE
 * (with *code, if non-NULL, set to the raw word). */
int vase_check_device_error(vase_ctx* ctx, void* stream, uint32_t* code);
/* Sites (code & 0xffff) of the compressed value store: an append or eviction found a ring state or bf16 masks
 * it did not write (head or count out of range) and wrote nothing; an append would overflow the ring after an
 * eviction (a fill that skipped an eviction).  The decode reads such a store with head 0 and records its own site. */
#define VASE_SITE_STORE_OVERFLOW 80
#define VASE_SITE_STORE_STATE 81

/* Self-test of the failure detection: launches on `stream` a one-thread kernel whose
 * bounded wait on an mbarrier that nothing completes runs out (about two seconds,
 * the wait limit of every kernel here); the kernel records VASE_SITE_SELF_TEST in
 * the context's device error word and returns, without a fault.  A following
 * vase_check_device_error then returns VASE_ERR_DEVICE with (code & 0xffff) ==
 * VASE_SITE_SELF_TEST and clears the word; the context stays usable.  Returns
 * VASE_OK once launched. */
#define VASE_SITE_SELF_TEST 127
int vase_self_test_wait_timeout(vase_ctx* ctx, void* stream);

/* Number of kernels the library launched on this context since creation. */
int64_t vase_launch_count(const vase_ctx* ctx);

/* Kernel kinds reported by vase_profile_collect. */
#define VASE_KERNEL_APPEND 0
#define VASE_KERNEL_SCORE 1   /* window attention score (tcgen05) */
#define VASE_KERNEL_VALUE 2   /* value magnitude refresh (vase_refresh_value_scores) */
#define VASE_KERNEL_DKV 3     /* DKV leverage scores (tcgen05) */
#define VASE_KERNEL_SELECT 4  /* reservation + sampling + kept list + stable in-place gather of the kept rows */
#define VASE_KERNEL_EVICT_SMALL 5 /* window score + selection + gather in one launch (launch-bound batches of small units) */
#define VASE_KERNEL_STORE_APPEND 6 /* compressed value store: new values into the reserved ring (earliest out when full) */
#define VASE_KERNEL_STORE_EVICT 7  /* compressed value store: codes and ring compacted, values leaving R_V u R_B quantized */
#define VASE_KERNEL_COUNT 8

/* enable = 1: from now on record a CUDA event pair on the launch stream around
 * every kernel (host-side instrumentation, no change to the kernels);
 * enable = 0: stop recording.  Events are created by the library. */
int vase_profile_enable(vase_ctx* ctx, int enable);

/* Waits for the recorded events, writes per kernel kind the summed device time
 * in milliseconds (total_ms[VASE_KERNEL_COUNT]) and the number of launches
 * (launches[VASE_KERNEL_COUNT]), then forgets the recorded events. */
int vase_profile_collect(vase_ctx* ctx, double* total_ms, int64_t* launches);

/* Eviction for callers that cannot allocate device memory.
 *
 * Some callers own no device allocator: a plugin inside an inference server whose host
 * process owns all device memory and hands it only tensors, or a runtime that forbids
 * device allocation after start-up to keep a fixed, unfragmented memory budget.  They can
 * pass the caches but not the workspace that vase_create asks for.  This entry point runs
 * one eviction step of one layer (the same kernels and results as vase_evict) with its
 * scratch -- window scores, DKV leverage products, kept-slot lists and the device error
 * word -- in a static device array of VASE_STATIC_SCRATCH_BYTES that every GPU loading the
 * library holds until the process exits.  It calls no cudaMalloc, cudaFree or other
 * allocating routine and needs no context.  The paper has no counterpart; it is a
 * deployment convenience of this library.
 *
 *   cfg, bufs: as for vase_create; bufs->workspace is ignored and may be NULL.
 *   state:     the layer's counters as the caller tracks them; state->fill must be K + B and
 *              state->round keys the noise.  The call does not update them: afterwards the
 *              caller sets fill = K and round + 1.
 *   device_error: NULL, or a host word.  Non-NULL: the call waits for the stream, stores the
 *              device error word there, and if it is non-zero clears it and returns
 *              VASE_ERR_DEVICE.  NULL: the call neither waits nor reads the word; a failure
 *              stays recorded in the array (the kernels only set bits in it) and is returned
 *              by the next call made with a non-NULL device_error, so a caller that passes
 *              NULL on its hot path can ask now and then.
 * Layers needing more scratch than the array holds (256 + (b*Hkv) * (K+B) * 4 * (1 + parts)
 * + (b*Hkv) * K * 4 bytes, parts = 4 when G*W > 256 (2 with GQA max-aggregation and a window
 * that does not divide 128), else 1, each term rounded up to 256)
 * are rejected with VASE_ERR_UNSUPPORTED before any buffer is looked at; the Qwen3-32B
 * geometry at batch 16 (about 17 MB) is one.  The first call on a device looks up the array's
 * device address (cudaGetSymbolAddress) with that device current; make that first call before
 * any stream capture.  Under the CUDA default of lazy module loading that first call is also
 * when the device commits the VASE_STATIC_SCRATCH_BYTES of the array, and it fails with
 * VASE_ERR_CUDA (an out-of-memory message) if the device's memory is already taken: make it
 * at start-up, or set CUDA_MODULE_LOADING=EAGER so that the array is committed when the
 * library loads.  Every call shares the one array and leaves its contents behind: calls that
 * can overlap on the GPU (different streams, or several host threads) race on it and must be
 * serialised by the caller.  Errors are explained by vase_last_error(NULL). */
#define VASE_STATIC_SCRATCH_BYTES (16u << 20)
int vase_evict_static_scratch(const vase_config* cfg, const vase_buffers* bufs, int32_t layer,
                              const vase_layer_state* state, uint32_t* device_error, void* stream);

const char* vase_status_string(int status);
/* Message of the last failed call on ctx; with ctx == NULL, the reason the last
 * configuration check on this thread (vase_get_buffer_sizes, vase_create) failed. */
const char* vase_last_error(const vase_ctx* ctx);
int vase_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* VASE_H */
