"""Seeded synthetic workloads for the VaSE eviction step.

This module only draws inputs: it holds none of the method's arithmetic and
imports neither the CUDA binding nor the oracle, so both sides can consume
the same bytes.  Every array is produced from a numpy generator keyed by
(seed, kind, layer, sequence, head), so any single unit can be regenerated
on its own, at any size, by whoever needs it.

The distributions follow the workloads of the paper's setting: Qwen3
attention geometries at about 4x compression with large-magnitude value
outliers (Sec. 3.1, Fig. 2; App. A) and channel outliers in keys/queries.
"""

from __future__ import annotations

from dataclasses import dataclass, field, replace

import numpy as np

_KIND_Q, _KIND_K, _KIND_V, _KIND_CH, _KIND_POS, _KIND_VOUT = 1, 2, 3, 4, 5, 6


@dataclass(frozen=True)
class Workload:
    name: str
    num_layers: int
    batch: int
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    budget_k: int
    buffer_b: int
    window: int
    stream_tokens: int
    key_channel_outliers: bool = False
    query_channel_outliers: bool = False
    value_outlier_rate: float = 0.005
    value_outlier_scale: tuple = (20.0, 20.0)   # (lo, hi); lo < hi -> log-uniform
    variants: tuple = ("attnv",)
    outlier_channels: int = 4
    channel_scale: float = 8.0

    @property
    def group(self):
        return self.num_q_heads // self.num_kv_heads

    @property
    def slots(self):
        return self.budget_k + self.buffer_b

    @property
    def window_rows(self):
        return self.group * self.window

    @property
    def units_per_layer(self):
        return self.batch * self.num_kv_heads

    @property
    def rounds_per_layer(self):
        """Eviction rounds in the stream: the first at K+B tokens, then every B tokens."""
        if self.stream_tokens < self.slots:
            return 0
        return 1 + (self.stream_tokens - self.slots) // self.buffer_b


WORKLOADS = {
    # one layer, batch 1, 16/8 heads, K+B = 256+64, W = 32; keys and queries with channel outliers
    "single_layer_k256": Workload("single_layer_k256", 1, 1, 16, 8, 128, 256, 64, 32, 320,
                                  key_channel_outliers=True, query_channel_outliers=True,
                                  value_outlier_rate=0.005, value_outlier_scale=(20.0, 20.0)),
    # Qwen3-1.7B attention geometry, 8192-token stream, 48 rounds per layer
    "qwen3_1p7b_k2048": Workload("qwen3_1p7b_k2048", 28, 8, 16, 8, 128, 2048, 128, 32, 8192,
                                 value_outlier_rate=0.005, value_outlier_scale=(20.0, 20.0)),
    # Qwen3-8B attention geometry, 16384-token stream, AttnV and DKV
    "qwen3_8b_k4096": Workload("qwen3_8b_k4096", 36, 32, 32, 8, 128, 4096, 128, 32, 16384,
                               key_channel_outliers=True,
                               value_outlier_rate=0.005, value_outlier_scale=(20.0, 20.0),
                               variants=("attnv", "dkv")),
    # Qwen3-32B attention geometry, 32768-token stream, 1% of value rows at x10-x50 (log-uniform)
    "qwen3_32b_k8192": Workload("qwen3_32b_k8192", 64, 16, 64, 8, 128, 8192, 256, 64, 32768,
                                key_channel_outliers=True,
                                value_outlier_rate=0.01, value_outlier_scale=(10.0, 50.0)),
}


def sweep_point(budget_k, buffer_b, batch, outlier_rate):
    """One point of the Qwen3-8B sweep (36 layers, 32/8 heads, d = 128, W = 32)."""
    return Workload(f"qwen3_8b_sweep_k{budget_k}_b{buffer_b}_bs{batch}_o{outlier_rate}", 36, batch, 32, 8,
                    128, budget_k, buffer_b, 32, 4 * budget_k, key_channel_outliers=True,
                    value_outlier_rate=outlier_rate, value_outlier_scale=(20.0, 20.0))


def shrink(wl: Workload, **kw) -> Workload:
    return replace(wl, **kw)


# ----------------------------------------------------------------------------
# bf16 bit patterns (round to nearest even)
# ----------------------------------------------------------------------------

def f32_to_bf16_bits(x):
    b = np.ascontiguousarray(np.asarray(x, dtype=np.float32)).view(np.uint32).astype(np.uint64)
    r = (b + np.uint64(0x7FFF) + ((b >> np.uint64(16)) & np.uint64(1))) >> np.uint64(16)
    return r.astype(np.uint16)


def _rng(seed, kind, layer, seq, head):
    return np.random.default_rng([int(seed) & 0xFFFFFFFF, kind, layer, seq, head])


def outlier_channels(wl: Workload, seed, layer, kv_head):
    """The channel-outlier set of one (layer, KV head), shared by its G query heads."""
    g = _rng(seed, _KIND_CH, layer, 0, kv_head)
    return np.sort(g.choice(wl.head_dim, wl.outlier_channels, replace=False))


def _keys(wl, seed, layer, seq, head, n, salt=0):
    x = _rng(seed, _KIND_K, layer, seq, head * 1000003 + salt).standard_normal((n, wl.head_dim))
    if wl.key_channel_outliers:
        x[:, outlier_channels(wl, seed, layer, head)] *= wl.channel_scale
    return x


def _values(wl, seed, layer, seq, head, n, salt=0):
    g = _rng(seed, _KIND_V, layer, seq, head * 1000003 + salt)
    x = g.standard_normal((n, wl.head_dim))
    rows = g.random(n) < wl.value_outlier_rate
    lo, hi = wl.value_outlier_scale
    if hi > lo:
        scale = np.exp(g.uniform(np.log(lo), np.log(hi), n))
    else:
        scale = np.full(n, lo)
    x[rows] *= scale[rows, None]
    return x


def _queries(wl, seed, layer, seq, kv_head, rows_per_head, salt=0):
    q = np.empty((wl.group, rows_per_head, wl.head_dim))
    for g in range(wl.group):
        qh = kv_head * wl.group + g
        q[g] = _rng(seed, _KIND_Q, layer, seq, qh * 1000003 + salt).standard_normal((rows_per_head, wl.head_dim))
    if wl.query_channel_outliers:
        q[:, :, outlier_channels(wl, seed, layer, kv_head)] *= wl.channel_scale
    return q


def unit_state(wl: Workload, seed, layer, seq, head, round_index=0, positions="gapped"):
    """Pre-eviction state of one unit, as raw bf16 bits.

    Returns q_bits [G, W, d] (the window queries of the unit's query heads),
    k_bits / v_bits [K+B, d] and positions int64 [K+B].  With
    positions="gapped" the K persistent slots hold an increasing random subset
    of the earlier stream positions and the buffer the B most recent ones,
    as after ``round_index`` earlier rounds; "dense" gives 0..K+B-1.
    """
    N = wl.slots
    salt = round_index
    k = f32_to_bf16_bits(_keys(wl, seed, layer, seq, head, N, salt))
    v = f32_to_bf16_bits(_values(wl, seed, layer, seq, head, N, salt))
    q = f32_to_bf16_bits(_queries(wl, seed, layer, seq, head, wl.window, salt))
    if positions == "dense" or round_index == 0:
        pos = np.arange(N, dtype=np.int64)
    else:
        first = wl.budget_k + round_index * wl.buffer_b
        g = _rng(seed, _KIND_POS, layer, seq, head * 1000003 + salt)
        persistent = np.sort(g.choice(first, wl.budget_k, replace=False))
        pos = np.concatenate([persistent, np.arange(first, first + wl.buffer_b)]).astype(np.int64)
    return {"q_bits": q, "k_bits": k, "v_bits": v, "positions": pos}


def layer_state(wl: Workload, seed, layer, round_index=0, positions="gapped"):
    """All units of one layer in the cache layouts of the library:

    q_bits [b, Hq, W, d], k_bits / v_bits [b, Hkv, K+B, d], positions [b, Hkv, K+B].
    """
    b, Hkv, G, W, d, N = wl.batch, wl.num_kv_heads, wl.group, wl.window, wl.head_dim, wl.slots
    q = np.empty((b, Hkv * G, W, d), dtype=np.uint16)
    k = np.empty((b, Hkv, N, d), dtype=np.uint16)
    v = np.empty((b, Hkv, N, d), dtype=np.uint16)
    pos = np.empty((b, Hkv, N), dtype=np.int64)
    for s in range(b):
        for h in range(Hkv):
            u = unit_state(wl, seed, layer, s, h, round_index, positions)
            q[s, h * G:(h + 1) * G] = u["q_bits"]
            k[s, h] = u["k_bits"]
            v[s, h] = u["v_bits"]
            pos[s, h] = u["positions"]
    return {"q_bits": q, "k_bits": k, "v_bits": v, "positions": pos}


def stream_chunk(wl: Workload, seed, layer, first_token, n_tokens):
    """New decode tokens of one layer as the decode loop emits them:

    q_bits [n, b, Hq, d], k_bits / v_bits [n, b, Hkv, d] for stream tokens
    first_token .. first_token + n - 1.
    """
    b, Hq, Hkv, d = wl.batch, wl.num_q_heads, wl.num_kv_heads, wl.head_dim
    q = np.empty((n_tokens, b, Hq, d), dtype=np.uint16)
    k = np.empty((n_tokens, b, Hkv, d), dtype=np.uint16)
    v = np.empty((n_tokens, b, Hkv, d), dtype=np.uint16)
    for s in range(b):
        for h in range(Hkv):
            k[:, s, h] = f32_to_bf16_bits(_keys(wl, seed, layer, s, h, n_tokens, 7919 + first_token))
            v[:, s, h] = f32_to_bf16_bits(_values(wl, seed, layer, s, h, n_tokens, 7919 + first_token))
            qq = _queries(wl, seed, layer, s, h, n_tokens, 7919 + first_token)
            for g in range(wl.group):
                q[:, s, h * wl.group + g] = f32_to_bf16_bits(qq[g])
    return {"q_bits": q, "k_bits": k, "v_bits": v}
