"""The seeded input recipe (no GPU): bf16 rounding, keyed determinism, the value-outlier rows and their scale,
the key channel outliers, the gapped positions of a round and the layer layout of the unit states."""

import numpy as np
import pytest

from paper_2606_03928_gb300 import workloads as W


def test_bf16_bits_round_to_nearest_even():
    x = np.array([1.0, 1.0 + 2.0 ** -8, 1.0 + 3.0 * 2.0 ** -8, 1.0 + 2.0 ** -7, -2.5, 0.0], dtype=np.float32)
    # 1 + 2^-8 lies halfway between 1 (0x3F80) and 1 + 2^-7 (0x3F81): ties go to the even 0x3F80;
    # 1 + 3 * 2^-8 lies halfway between 0x3F81 and 0x3F82: to the even 0x3F82
    assert W.f32_to_bf16_bits(x).tolist() == [0x3F80, 0x3F80, 0x3F82, 0x3F81, 0xC020, 0x0000]


def test_unit_states_are_keyed_and_reproducible():
    wl = W.WORKLOADS["single_layer_k256"]
    a = W.unit_state(wl, 0, 0, 0, 3, round_index=2)
    b = W.unit_state(wl, 0, 0, 0, 3, round_index=2)
    for key in ("q_bits", "k_bits", "v_bits", "positions"):
        assert np.array_equal(a[key], b[key])
    for other in (W.unit_state(wl, 0, 0, 0, 4, 2), W.unit_state(wl, 1, 0, 0, 3, 2), W.unit_state(wl, 0, 0, 0, 3, 3)):
        assert not np.array_equal(a["k_bits"], other["k_bits"])


def _norms(v_bits):
    v = (v_bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    return np.linalg.norm(v, axis=-1)


def test_value_outlier_rows_follow_the_rate_and_scale():
    # rows x20 at a rate of 0.5 %: over 64 units of 2176 rows the count is within 5 sigma of the binomial mean
    wl = W.WORKLOADS["qwen3_1p7b_k2048"]
    norms = np.concatenate([_norms(W.unit_state(wl, 0, 0, s, h)["v_bits"]) for s in range(8) for h in range(8)])
    n, p = norms.size, wl.value_outlier_rate
    big = norms > 5.0 * np.sqrt(wl.head_dim)  # N(0, 1) rows have norms near sqrt(d); x20 rows near 20 sqrt(d)
    assert abs(big.sum() - n * p) < 5 * np.sqrt(n * p * (1 - p))
    assert np.all(np.abs(norms[big] / np.sqrt(wl.head_dim) - 20.0) < 5.0)


def test_log_uniform_outlier_scale_of_the_large_geometry():
    # 1 % of rows scaled by a log-uniform factor in [10, 50]
    wl = W.WORKLOADS["qwen3_32b_k8192"]
    norms = np.concatenate([_norms(W.unit_state(wl, 0, 0, s, 0)["v_bits"]) for s in range(4)])
    big = norms > 5.0 * np.sqrt(wl.head_dim)
    scale = norms[big] / np.sqrt(wl.head_dim)
    assert abs(big.mean() - 0.01) < 0.004
    assert scale.min() > 10.0 * 0.7 and scale.max() < 50.0 * 1.3
    assert np.median(np.log(scale)) == pytest.approx(0.5 * (np.log(10.0) + np.log(50.0)), abs=0.35)


def test_key_channel_outliers_are_four_channels_scaled_by_eight():
    wl = W.WORKLOADS["qwen3_8b_k4096"]
    k = (W.unit_state(wl, 0, 2, 1, 5)["k_bits"].astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    ch = W.outlier_channels(wl, 0, 2, 5)
    assert ch.size == 4
    std = k.std(axis=0)
    rest = np.setdiff1d(np.arange(wl.head_dim), ch)
    assert np.all(np.abs(std[ch] - 8.0) < 0.6) and np.all(np.abs(std[rest] - 1.0) < 0.1)


def test_gapped_positions_of_a_round():
    wl = W.shrink(W.WORKLOADS["single_layer_k256"], budget_k=64, buffer_b=16)
    r = 3
    pos = W.unit_state(wl, 0, 0, 0, 0, round_index=r)["positions"]
    first = wl.budget_k + r * wl.buffer_b  # stream position of the round's first new token
    assert np.all(np.diff(pos[:wl.budget_k]) > 0) and pos[wl.budget_k - 1] < first  # a sorted subset of the past
    assert np.array_equal(pos[wl.budget_k:], np.arange(first, first + wl.buffer_b))  # the B newest, in order
    assert np.array_equal(W.unit_state(wl, 0, 0, 0, 0, round_index=0)["positions"], np.arange(wl.slots))


def test_layer_state_places_every_unit_at_its_head():
    wl = W.shrink(W.WORKLOADS["single_layer_k256"], batch=2)
    st = W.layer_state(wl, 0, 0, 2)
    u = W.unit_state(wl, 0, 0, 1, 5, 2)
    G = wl.group
    assert np.array_equal(st["k_bits"][1, 5], u["k_bits"]) and np.array_equal(st["v_bits"][1, 5], u["v_bits"])
    assert np.array_equal(st["q_bits"][1, 5 * G:6 * G], u["q_bits"]) and np.array_equal(st["positions"][1, 5], u["positions"])
