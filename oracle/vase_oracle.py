"""Plain fp64 CPU oracle of one VaSE eviction step (arXiv 2606.03928).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline / reference legs of ``bench.py`` may import this module.  The
product path (the CUDA library and its Python binding) never calls it and
shares no code with it.

Every step follows the paper's definitions in the paper's order, one unit at a
time, where a *unit* is one (layer, sequence, KV head):

* attention weights of a window query over all N = K + B cached keys -- Eq. (1), Sec. 2;
* the SnapKV score, the mean of those weights over the window queries, with
  average pooling and non-causal cached queries -- Eq. (2) and its footnote, Sec. 2;
* the value magnitude Range(v) -- Eq. (5), Sec. 3.1 -- and the L2 / Var variants -- App. A;
* VaSE-AttnV: reserve the buffer R_B and the N_v largest-Range candidates R_V,
  then fill the K - |R| remaining slots by weighted sampling without
  replacement with weights proportional to the pooled score -- Sec. 3.2;
* the deterministic "+V without sampling" ablation -- Sec. 4.1;
* VaSE-DKV: the CurDKV product of key and value leverage scores under a
  Gaussian projection G_t ~ N(0, 1/r) that is redrawn every eviction round,
  then the top K - B candidates -- Eq. (4), Sec. 2 and Sec. 3.2;
* the periodic-eviction framing (protect the B most recent tokens, keep
  exactly K of the K + B cached tokens) -- Sec. 2, "Periodic eviction";
* the decode step's attention output over the kept cache, o = sum_i alpha_i v_i
  -- Eq. (1), Sec. 2 (the consumer of the cache the eviction leaves);
* variants: the random-reservation ablation (N_v candidates drawn uniformly
  at random instead of the largest Range) -- App. C, first paragraph; GQA
  max-aggregation over the query heads of a KV head; one Gaussian projection
  per round shared by every unit (shared-G DKV);
* per-token asymmetric b-bit quantization of value rows, z = min v,
  s = Range(v) / (2^b - 1), Q(v) = round((v - z) / s), v' = Q s + z -- the
  equation of Sec. 4.4 -- and the mixed-precision value cache that Sec. 6
  proposes: the reserved large-Range values (R_V) and the recency buffer keep
  their bf16 rows, every other kept value is read back from its b-bit codes;
* the compressed value store built on that proposal: the bf16 rows live only
  in a reserved cache of N_v + 2B rows (a ring in slot order), every other
  cached value only as its codes; an append that finds the reserved cache full
  quantizes its earliest value that is not large-Range into the low-precision
  cache (the rule Sec. 6 states), and an eviction quantizes the kept values
  that leave R_V u R_B.

Readings where the paper is silent (each is listed with its reason in the
design notes of the repository):

* GQA: the window rows of a KV head are the W cached queries of each of its
  G query heads (head-major: rows g*W .. g*W+W-1 belong to query head g); the
  score is the mean over all G*W rows, or (gqa="max") the largest over the G
  heads of each head's mean over its W rows.
* Window: W is its own parameter (the paper sets W = B); the divisor is G*W.
* Pooling: odd kernel kappa, stride 1, zero padding, divisor kappa, along the
  slot axis over all N slots, before restricting to candidates.
* Weighted sampling without replacement is successive sampling (draw one
  token with probability proportional to the remaining weights, remove it,
  repeat).  It is realised as the exponential race: keep the m largest
  alpha_i / E_i with E_i = -ln u_i (Efraimidis and Spirakis, 2006), which has
  the same joint law.  The tests pin that equivalence by exact enumeration.
* Ties in any ranking go to the lower slot (the older token).
* Noise: u_i comes from Philox4x32-10 (Salmon et al., SC'11) with key
  (seed_lo, seed_hi) and counter (position, round, layer | tag << 24,
  seq * Hkv + head); tag 0 = selection noise, tag 1 = DKV Gaussian, tag 2 =
  random-reservation noise.
  u = (2 * (x >> 9) + 1) * 2**-24 from word 0, exact in fp32 and fp64.
  Gaussian entries use Box-Muller (1958) on words 0 and 1 with counter
  word 0 = a * r + b; the fixed-G (CurDKV) option puts 0 in the round word,
  and the shared-G option puts 0 in the layer bits and the unit word.
* DKV has no value reservation; the value awareness is the value leverage.
* Quantization codes are integers decided by floating point, so they are
  computed in fp32 (the kernels' precision): v - z, the division by s and
  the rounding (half to even) each in fp32.  A row of equal values has s = 0
  and codes 0.  After an eviction the reserved (bf16) values are R_B, the
  last B kept slots, and R_V, which is again the N_v largest value
  magnitudes among the first K - B kept slots (R_V is kept whole and the
  compaction keeps the order).
* Compressed value store: keys stay bf16 (Sec. 4.4 and Sec. 6 speak of value
  states).  The reserved cache holds R_V u R_B after an eviction (at most
  N_v + B rows) and the B values appended before the next one, so its
  capacity is H = N_v + 2B; only the appends before the first eviction can
  find it full.  The values the rule of Sec. 6 spills when it is full are
  "the earliest" among those that are not large-Range: the large-Range values
  are the N_v largest value magnitudes among the slots the next eviction
  draws R_V from (slots below K, ties to the lower slot), the set R_V would be
  now.  (Taken over all values, a long first fill would quantize the
  large-Range values of its earliest tokens before the first eviction could
  reserve them, which is what the proposal is there to prevent.)  So the
  first eviction finds R_V in bf16, and so does every later one.  A value
  that leaves R_V u R_B at an eviction while kept is quantized then (it no
  longer holds a reserved slot).  A quantized value never returns to bf16: a
  later R_V is drawn from the earlier R_V and the newly appended values only,
  since R_V is kept whole.
"""

from __future__ import annotations

import numpy as np

# ----------------------------------------------------------------------------
# Philox4x32-10 (Salmon, Moraes, Dror, Shaw: "Parallel random numbers: as easy
# as 1, 2, 3", SC'11): two 32x32->64 multiplies per round, the Weyl key
# schedule, ten rounds.
# ----------------------------------------------------------------------------

_MASK32 = np.uint64(0xFFFFFFFF)
_PHILOX_M0 = np.uint64(0xD2511F53)
_PHILOX_M1 = np.uint64(0xCD9E8D57)
_PHILOX_W0 = np.uint64(0x9E3779B9)
_PHILOX_W1 = np.uint64(0xBB67AE85)

TAG_SELECT = 0
TAG_DKV = 1
TAG_RESERVE = 2


def philox4x32_10(c0, c1, c2, c3, k0, k1):
    """Philox4x32 with 10 rounds on arrays of 32-bit counters; returns 4 uint32 arrays."""
    c0, c1, c2, c3 = (np.asarray(c, dtype=np.uint64) & _MASK32 for c in (c0, c1, c2, c3))
    c0, c1, c2, c3 = np.broadcast_arrays(c0, c1, c2, c3)
    k0 = np.uint64(int(k0) & 0xFFFFFFFF)
    k1 = np.uint64(int(k1) & 0xFFFFFFFF)
    for _ in range(10):
        p0 = _PHILOX_M0 * c0
        p1 = _PHILOX_M1 * c2
        hi0, lo0 = p0 >> np.uint64(32), p0 & _MASK32
        hi1, lo1 = p1 >> np.uint64(32), p1 & _MASK32
        c0, c1, c2, c3 = hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0
        k0 = (k0 + _PHILOX_W0) & _MASK32
        k1 = (k1 + _PHILOX_W1) & _MASK32
    return tuple(x.astype(np.uint32) for x in (c0, c1, c2, c3))


def uniform_open01(word):
    """Map a 32-bit word to u = (2 * (x >> 9) + 1) * 2**-24, strictly inside (0, 1)."""
    x = np.asarray(word, dtype=np.uint64) >> np.uint64(9)
    return (2.0 * x.astype(np.float64) + 1.0) * 2.0 ** -24


def _noise_key(seed):
    seed = int(seed) & 0xFFFFFFFFFFFFFFFF
    return seed & 0xFFFFFFFF, seed >> 32


def selection_uniforms(seed, layer, seq, head, num_kv_heads, rnd, positions):
    """u_i for the sampling race of one unit, keyed by each token's stream position."""
    k0, k1 = _noise_key(seed)
    pos = np.asarray(positions, dtype=np.int64).astype(np.uint64)
    w0, _, _, _ = philox4x32_10(pos, rnd, (layer | (TAG_SELECT << 24)), seq * num_kv_heads + head, k0, k1)
    return uniform_open01(w0)


def reservation_uniforms(seed, layer, seq, head, num_kv_heads, rnd, positions):
    """Uniform keys of the random-reservation ablation (App. C): the N_v largest pick R_V."""
    k0, k1 = _noise_key(seed)
    pos = np.asarray(positions, dtype=np.int64).astype(np.uint64)
    w0, _, _, _ = philox4x32_10(pos, rnd, (layer | (TAG_RESERVE << 24)), seq * num_kv_heads + head, k0, k1)
    return uniform_open01(w0)


def gaussian_projection(seed, layer, seq, head, num_kv_heads, rnd, d, r, fixed_g=False, shared_g=False):
    """G in R^{d x r} with i.i.d. N(0, 1/r) entries -- Eq. (4), Sec. 2; redrawn per round -- Sec. 3.2.

    Entry (a, b) takes Philox counter (a * r + b, round, layer | 1 << 24, seq * Hkv + head)
    and Box-Muller on words 0 and 1: z = sqrt(-2 ln u1) cos(2 pi u2).  fixed_g puts 0 in the round
    word (one G for the whole stream); shared_g puts 0 in the layer bits and the unit word (one G
    per round for every layer, sequence and KV head).
    """
    k0, k1 = _noise_key(seed)
    idx = np.arange(d * r, dtype=np.uint64)
    rr = 0 if fixed_g else rnd
    c2 = (0 if shared_g else layer) | (TAG_DKV << 24)
    c3 = 0 if shared_g else seq * num_kv_heads + head
    w0, w1, _, _ = philox4x32_10(idx, rr, c2, c3, k0, k1)
    u1 = uniform_open01(w0)
    u2 = uniform_open01(w1)
    z = np.sqrt(-2.0 * np.log(u1)) * np.cos(2.0 * np.pi * u2)
    return (z / np.sqrt(r)).reshape(d, r)


# ----------------------------------------------------------------------------
# bf16 widening (exact) -- inputs arrive as raw bf16 bit patterns.
# ----------------------------------------------------------------------------

def bf16_bits_to_f64(bits):
    b = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return b.view(np.float32).astype(np.float64)


# ----------------------------------------------------------------------------
# Scores
# ----------------------------------------------------------------------------

def attention_weights(q_rows, keys):
    """alpha[r, i] of Eq. (1): softmax over all N cached keys of q_r . k_i / sqrt(d)."""
    d = keys.shape[1]
    logits = (q_rows @ keys.T) / np.sqrt(d)
    logits = logits - logits.max(axis=1, keepdims=True)
    e = np.exp(logits)
    return e / e.sum(axis=1, keepdims=True)


def window_attention_score(q_rows, keys, group=1, gqa="mean"):
    """The window score of Eq. (2) (non-causal cached queries), before pooling.

    q_rows holds the W window queries of each of the `group` query heads, head-major.  "mean": the
    mean of alpha over all G*W rows.  "max": each head's mean over its W rows, then the largest over
    the G heads (GQA max-aggregation)."""
    a = attention_weights(q_rows, keys)
    if gqa == "mean":
        return a.mean(axis=0)
    if gqa == "max":
        G = int(group)
        per_head = a.reshape(G, a.shape[0] // G, a.shape[1]).mean(axis=1)
        return per_head.max(axis=0)
    raise ValueError(f"unknown GQA reduction {gqa}")


def average_pool(scores, kernel):
    """Stride-1 average pooling along the slot axis, zero padded, divisor = kernel."""
    kernel = int(kernel)
    if kernel <= 1:
        return np.asarray(scores, dtype=np.float64).copy()
    return np.convolve(scores, np.ones(kernel) / kernel, mode="same")


VALUE_RANGE, VALUE_L2, VALUE_VAR = 0, 1, 2


def value_magnitude(values, kind=VALUE_RANGE):
    """Range(v) = max_j v_j - min_j v_j (Eq. (5)); L2 and Var variants of App. A."""
    if kind == VALUE_RANGE:
        return values.max(axis=1) - values.min(axis=1)
    if kind == VALUE_L2:
        return np.sqrt((values * values).sum(axis=1))
    if kind == VALUE_VAR:
        mu = values.mean(axis=1, keepdims=True)
        return ((values - mu) ** 2).mean(axis=1)
    raise ValueError(f"unknown value score kind {kind}")


def leverage_scores(keys, values, G):
    """CurDKV product score s_i = ||G^T k_i||^2 * ||G^T v_i||^2 (Eq. (4))."""
    lk = ((keys @ G) ** 2).sum(axis=1)
    lv = ((values @ G) ** 2).sum(axis=1)
    return lk * lv, lk, lv


# ----------------------------------------------------------------------------
# Selection
# ----------------------------------------------------------------------------

def top_k_slots(scores, k, eligible=None):
    """Indices of the k largest scores among eligible slots; ties go to the lower slot."""
    scores = np.asarray(scores, dtype=np.float64)
    idx = np.arange(scores.shape[0])
    if eligible is not None:
        idx = idx[np.asarray(eligible, dtype=bool)]
    order = np.lexsort((idx, -scores[idx]))
    return np.sort(idx[order[:k]])


def evict_unit(q_rows, keys, values, positions, *, budget_k, buffer_b, variant="attnv",
               n_v=None, value_score=VALUE_RANGE, pool_kernel=7, stochastic=True,
               dkv_rank=20, dkv_fixed_g=False, seed=0, layer=0, seq=0, head=0,
               num_kv_heads=1, rnd=0, group=1, gqa="mean", reserve="value", dkv_shared_g=False):
    """One eviction step for one unit, in fp64.

    q_rows [G*W, d], keys/values [K+B, d] (fp64, exact bf16 values), positions [K+B].
    Returns a dict with the scores, the keep mask, the ascending kept-slot list
    and the compacted keys, values and positions.
    """
    K, B = int(budget_k), int(buffer_b)
    N = K + B
    assert keys.shape[0] == N and values.shape[0] == N and len(positions) == N
    out = {}
    keep = np.zeros(N, dtype=bool)
    keep[K:] = True                       # R_B: the B most recent tokens are protected (Sec. 2)
    if variant == "attnv":
        nv = K // 4 if n_v is None or n_v < 0 else int(n_v)
        m = K - nv - B                    # the K - |R| sampled slots (Sec. 3.2)
        assert m >= 0
        a = window_attention_score(q_rows, keys, group, gqa)
        abar = average_pool(a, pool_kernel)
        vmag = value_magnitude(values[:K], value_score)
        if reserve == "value":
            r_v = top_k_slots(vmag, nv)   # R_V: N_v largest Range among the K candidates
        elif reserve == "random":         # the ablation of App. C: N_v candidates uniformly at random
            r_v = top_k_slots(reservation_uniforms(seed, layer, seq, head, num_kv_heads, rnd, positions[:K]), nv)
        else:
            raise ValueError(reserve)
        in_c = np.ones(K, dtype=bool)
        in_c[r_v] = False                 # C = [K] \ R_V
        if stochastic:
            u = selection_uniforms(seed, layer, seq, head, num_kv_heads, rnd, positions[:K])
            key = abar[:K] / (-np.log(u))
        else:
            key = abar[:K].copy()
        sel = top_k_slots(key, m, eligible=in_c)
        keep[r_v] = True
        keep[sel] = True
        key_full = np.full(N, -1.0)
        key_full[:K] = np.where(in_c, key, -1.0)
        out.update(attn=a, pooled=abar, value_score=vmag, key=key_full, reserved_v=r_v)
    elif variant == "dkv":
        d = keys.shape[1]
        G = gaussian_projection(seed, layer, seq, head, num_kv_heads, rnd, d, dkv_rank, dkv_fixed_g, dkv_shared_g)
        s, lk, lv = leverage_scores(keys[:K], values[:K], G)
        sel = top_k_slots(s, K - B)
        keep[sel] = True
        key_full = np.full(N, -1.0)
        key_full[:K] = s
        out.update(value_score=s, lk=lk, lv=lv, key=key_full, G=G)
    else:
        raise ValueError(variant)
    src = np.flatnonzero(keep)
    assert src.shape[0] == K, "exactly K tokens are kept"
    out.update(keep=keep, src=src, keys_new=keys[src], values_new=values[src],
               positions_new=np.asarray(positions)[src])
    return out


# ----------------------------------------------------------------------------
# Decode attention over the kept cache (the consumer of the eviction's layout)
# ----------------------------------------------------------------------------

def decode_attention(q, keys, values):
    """Output of a decode step for query rows q over the cached pairs, Eq. (1), Sec. 2:
    o = sum_i alpha_i v_i with alpha_i the softmax over the cached keys of q . k_i / sqrt(d).
    q [rows, d] (the G query heads of one KV head), keys / values [n, d] (the n filled slots)."""
    return attention_weights(q, keys) @ values


def decode_attention_bound(q, keys, values):
    """sum_i alpha_i |v_i| per output element: the scale of an fp32 weighted sum's rounding error."""
    return attention_weights(q, keys) @ np.abs(values)


def decode_attention_bits(q_bits, k_bits, v_bits):
    """decode_attention on raw bf16 bit arrays; returns (output, its error scale)."""
    q, k, v = bf16_bits_to_f64(q_bits), bf16_bits_to_f64(k_bits), bf16_bits_to_f64(v_bits)
    return decode_attention(q, k, v), decode_attention_bound(q, k, v)


# ----------------------------------------------------------------------------
# Mixed-precision values (Sec. 4.4 equation, Sec. 6 proposal)
# ----------------------------------------------------------------------------

def quantize_values(values, bits):
    """Per-token asymmetric b-bit quantization of value rows [n, d] (exact bf16 values), in fp32.

    Returns codes [n, d] (uint8, 0 .. 2^b - 1), s [n] and z [n] (fp32)."""
    v = np.asarray(values, dtype=np.float32)
    lo = v.min(axis=1)
    hi = v.max(axis=1)
    levels = np.float32(2 ** int(bits) - 1)
    s = ((hi - lo) / levels).astype(np.float32)
    safe = np.where(s > 0, s, np.float32(1)).astype(np.float32)
    t = ((v - lo[:, None]) / safe[:, None]).astype(np.float32)
    codes = np.where(s[:, None] > 0, np.clip(np.rint(t), 0, levels), 0).astype(np.uint8)
    return codes, s, lo.astype(np.float32)


def dequantize_values(codes, s, z):
    """v' = Q s + z (Sec. 4.4), in fp64 from the fp32 parameters."""
    return np.asarray(codes, dtype=np.float64) * np.asarray(s, dtype=np.float64)[:, None] + \
        np.asarray(z, dtype=np.float64)[:, None]


def reserved_after_eviction(value_scores, budget_k, buffer_b, n_v):
    """Mask [K] of the kept slots whose bf16 value rows stay after an eviction: R_B (the last B slots)
    and R_V (the N_v largest value magnitudes among the first K - B kept slots; ties to the lower slot)."""
    K, B = int(budget_k), int(buffer_b)
    mask = np.zeros(K, dtype=bool)
    mask[K - B:] = True
    if n_v > 0:
        mask[top_k_slots(np.asarray(value_scores)[:K - B], int(n_v))] = True
    return mask


def decode_attention_mixed(q, keys, values, reserved, bits):
    """Decode attention where the values of unreserved slots are read back from their b-bit codes.

    Returns the output and its error scale: sum_i alpha_i |v_i| over the bf16 rows and, for a coded row,
    sum_i alpha_i (|Q_i s_i| + |z_i|), the size of the terms an fp32 evaluation of Q s + z rounds."""
    codes, s, z = quantize_values(values, bits)
    res = np.asarray(reserved, dtype=bool)[:, None]
    v_eff = np.where(res, values, dequantize_values(codes, s, z))
    scale = np.where(res, np.abs(values), np.abs(codes * np.asarray(s, dtype=np.float64)[:, None]) +
                     np.abs(np.asarray(z, dtype=np.float64))[:, None])
    return decode_attention(q, keys, v_eff), attention_weights(q, keys) @ scale


def evict_unit_bits(q_bits, k_bits, v_bits, positions, **kw):
    """evict_unit on raw bf16 bit arrays; compacted rows are returned as the same bits."""
    res = evict_unit(bf16_bits_to_f64(q_bits), bf16_bits_to_f64(k_bits), bf16_bits_to_f64(v_bits),
                     positions, **kw)
    src = res["src"]
    res["k_bits_new"] = np.asarray(k_bits)[src]
    res["v_bits_new"] = np.asarray(v_bits)[src]
    return res


# ----------------------------------------------------------------------------
# Compressed value store (Sec. 6: high-precision reserved cache, low-precision rest)
# ----------------------------------------------------------------------------

def store_capacity(budget_k, buffer_b, n_v):
    """Rows of the reserved (bf16) cache: R_V u R_B after an eviction plus the B values appended before the
    next one, H = N_v + 2B."""
    return int(n_v) + 2 * int(buffer_b)


def store_new(capacity):
    """An empty store: the reserved cache is a ring of `capacity` rows whose entries are the bf16 slots in slot
    order, entry i at ring position (head + i) mod capacity."""
    return {"H": int(capacity), "head": 0, "slots": []}


def store_large_range(value_scores, n_slots, budget_k, n_v):
    """The large-Range values of a cache of n_slots: the N_v largest value magnitudes among the slots below K
    (the candidates of R_V, Eq. (5)); ties to the lower slot."""
    c = min(int(n_slots), int(budget_k))
    return set(top_k_slots(np.asarray(value_scores, dtype=np.float64)[:c], min(int(n_v), c)).tolist())


def store_append(store, fill, n, value_scores=None, budget_k=0, n_v=0):
    """Appends slots fill .. fill + n - 1 (their values enter the reserved cache in bf16).  When the reserved
    cache would hold more than H values, its earliest values that are not large-Range (store_large_range over
    the filled slots, value_scores indexed by slot) are quantized into the low-precision cache (Sec. 6), as many
    as it is over.  The entries keep their slot order behind an unchanged head.  Returns the slots quantized by
    this call, in slot order."""
    H = store["H"]
    store["slots"] += [int(fill) + t for t in range(int(n))]
    over = len(store["slots"]) - H
    if over <= 0:
        return []
    keep = store_large_range(value_scores, fill + n, budget_k, n_v) if n_v else set()
    spilled = [s for s in store["slots"] if s not in keep][:over]
    gone = set(spilled)
    store["slots"] = [s for s in store["slots"] if s not in gone]
    return spilled


def store_evict(store, src, reserved_new):
    """The eviction's effect on the store: new slot j holds old slot src[j]; its value stays bf16 when it was
    bf16 and j is in R_V u R_B (reserved_new[j]), and is quantized when it was bf16 and is not.  The ring keeps
    its head; the retained entries close up in slot order.  Returns the new slots quantized by the eviction."""
    old = set(store["slots"])
    kept, spilled = [], []
    for j, s in enumerate(np.asarray(src).tolist()):
        if s in old:
            (kept if reserved_new[j] else spilled).append(j)
    store["slots"] = kept
    return spilled


def store_ring_positions(store):
    """Ring position of each bf16 slot: {slot: (head + i) mod H}."""
    H, h = store["H"], store["head"]
    return {s: (h + i) % H for i, s in enumerate(store["slots"])}


def store_reserved_mask(store, n_slots):
    """Mask [n_slots]: True where the slot's value is held in bf16."""
    mask = np.zeros(int(n_slots), dtype=bool)
    mask[np.asarray(store["slots"], dtype=np.int64)] = True
    return mask


def store_bytes(n_slots, capacity, d, bits):
    """Bytes of one unit's compressed value store (codes and (s, z) of every slot, the reserved cache)
    against the n_slots bf16 rows it replaces."""
    return int(n_slots) * (d * int(bits) // 8 + 8) + int(capacity) * 2 * d, int(n_slots) * 2 * d
