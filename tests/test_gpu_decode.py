"""GPU parity of the decode-step attention over the kept cache (vase_decode_attention, Eq. (1) of the
paper) against the fp64 oracle.

Tolerance: |o_gpu - o_ref| <= 1e-4 * sum_i alpha_i |v_i| per output element (+1e-7), a bound for an fp32
weighted sum of bf16 values whose weights come from fp32 dot products and exponentials."""

import numpy as np
import pytest
import torch

from oracle import vase_oracle as O
from paper_2606_03928_gb300 import workloads as W
import parity_utils as PU

pytestmark = pytest.mark.gpu

DEC_RTOL = 1e-4
DEC_ATOL = 1e-7

SMALL = W.WORKLOADS["single_layer_k256"]


def _cache(wl, num_layers):
    from paper_2606_03928_gb300.vase import VaseCache
    return VaseCache(PU.geometry_of(wl, num_layers), debug_outputs=False)


def _queries(wl, seed):
    rng = np.random.default_rng(seed)
    q = rng.standard_normal((wl.batch, wl.num_q_heads, wl.head_dim)).astype(np.float32)
    bits = W.f32_to_bf16_bits(q)
    return bits, PU.bits_to_bf16_tensor(bits, "cuda")


def _check(wl, cache, layer, q_bits, out, fill, units=None):
    k_bits = cache.k_cache[layer].view(torch.int16).cpu().numpy().view(np.uint16)
    v_bits = cache.v_cache[layer].view(torch.int16).cpu().numpy().view(np.uint16)
    got = out.cpu().numpy().astype(np.float64)
    G = wl.group
    todo = units if units is not None else [(s, h) for s in range(wl.batch) for h in range(wl.num_kv_heads)]
    for s, h in todo:
        ref, bound = O.decode_attention_bits(q_bits[s, h * G:(h + 1) * G], k_bits[s, h, :fill], v_bits[s, h, :fill])
        g = got[s, h * G:(h + 1) * G]
        bad = np.abs(g - ref) > DEC_RTOL * bound + DEC_ATOL
        assert not bad.any(), f"unit ({s}, {h}): {bad.sum()} outputs off, worst {np.abs(g - ref).max():.3e}"


@pytest.mark.parametrize("fill_kind", ["full", "ragged_one", "ragged_chunk"])
def test_decode_matches_oracle_small(fill_kind):
    wl = W.shrink(SMALL, budget_k=256, buffer_b=64, window=32, batch=2, num_layers=2)
    cache = _cache(wl, 2)
    st = W.layer_state(wl, 3, 1, 0, "gapped")
    PU.upload_layer(cache, 1, st, 0)
    fill = {"full": wl.slots, "ragged_one": 1, "ragged_chunk": 200}[fill_kind]
    cache.set_layer_state(1, fill, 0, fill, 10 ** 6)
    q_bits, q = _queries(wl, 5)
    out = cache.decode_attention(1, q)
    torch.cuda.synchronize()
    _check(wl, cache, 1, q_bits, out, fill)


def test_decode_after_eviction_reads_the_kept_cache():
    wl = W.shrink(SMALL, budget_k=192, buffer_b=64, window=16, batch=2, num_layers=1)
    cache = _cache(wl, 1)
    st = W.layer_state(wl, 8, 0, 2, "gapped")
    PU.upload_layer(cache, 0, st, 2)
    cache.evict(0)
    assert cache.layer_state(0)["fill"] == wl.budget_k
    q_bits, q = _queries(wl, 6)
    out = cache.decode_attention(0, q)
    torch.cuda.synchronize()
    _check(wl, cache, 0, q_bits, out, wl.budget_k)


def test_decode_with_eight_query_heads_per_kv_head():
    wl = W.shrink(SMALL, budget_k=320, buffer_b=96, window=16, num_q_heads=64, num_kv_heads=8, batch=1,
                  num_layers=1)
    cache = _cache(wl, 1)
    st = W.layer_state(wl, 9, 0, 0, "dense")
    PU.upload_layer(cache, 0, st, 0)
    q_bits, q = _queries(wl, 7)
    out = cache.decode_attention(0, q)
    torch.cuda.synchronize()
    _check(wl, cache, 0, q_bits, out, wl.slots)


def test_decode_full_size_layer_sampled_units():
    wl = W.WORKLOADS["qwen3_1p7b_k2048"]
    cache = _cache(wl, 2)
    st = W.layer_state(wl, 12, 1, 5, "gapped")
    PU.upload_layer(cache, 1, st, 5)
    cache.evict(1)
    q_bits, q = _queries(wl, 8)
    out = cache.decode_attention(1, q)
    torch.cuda.synchronize()
    _check(wl, cache, 1, q_bits, out, wl.budget_k, units=[(0, 0), (3, 5), (7, 7)])


def test_decode_rejects_an_empty_layer():
    from paper_2606_03928_gb300.vase import VaseError
    wl = W.shrink(SMALL, budget_k=64, buffer_b=16, window=8, batch=1, num_layers=1)
    cache = _cache(wl, 1)
    _, q = _queries(wl, 1)
    with pytest.raises(VaseError):
        cache.decode_attention(0, q)


# (query heads, KV heads): G = 1 and 2 take the CUDA-core kernel, G >= 3 the tensor-core kernel (5 and 16 also
# pad the head columns: 16 columns of P for G <= 8, 32 beyond)
@pytest.mark.parametrize("heads", [(8, 8), (24, 8), (32, 8), (40, 8), (64, 4)])
@pytest.mark.parametrize("fill_kind", ["full", "ragged"])
def test_decode_group_sizes(heads, fill_kind):
    Hq, Hkv = heads
    wl = W.shrink(SMALL, budget_k=448, buffer_b=64, window=16, num_q_heads=Hq, num_kv_heads=Hkv, batch=2,
                  num_layers=1)
    cache = _cache(wl, 1)
    st = W.layer_state(wl, 21, 0, 0, "gapped")
    PU.upload_layer(cache, 0, st, 0)
    fill = wl.slots if fill_kind == "full" else wl.slots - 37
    cache.set_layer_state(0, fill, 0, fill, 10 ** 6)
    q_bits, q = _queries(wl, 22)
    out = cache.decode_attention(0, q)
    torch.cuda.synchronize()
    _check(wl, cache, 0, q_bits, out, fill)


def test_decode_sees_the_append_launched_before_it():
    # the decode launch may start before the preceding kernel ends (programmatic dependent launch) but reads
    # nothing before that kernel's writes are visible: the second call must see the appended pairs
    wl = W.shrink(SMALL, budget_k=256, buffer_b=64, window=16, num_q_heads=32, num_kv_heads=8, batch=2,
                  num_layers=1)
    cache = _cache(wl, 1)
    st = W.layer_state(wl, 31, 0, 0, "gapped")
    PU.upload_layer(cache, 0, st, 0)
    cache.set_layer_state(0, 200, 0, 200, 10 ** 6)
    q_bits, q = _queries(wl, 32)
    first = cache.decode_attention(0, q)
    gen = torch.Generator(device="cuda")
    gen.manual_seed(33)
    n = 100
    qa = torch.randn((n, wl.batch, wl.num_q_heads, wl.head_dim), generator=gen, device="cuda").to(torch.bfloat16)
    ka = torch.randn((n, wl.batch, wl.num_kv_heads, wl.head_dim), generator=gen, device="cuda").to(torch.bfloat16)
    va = torch.randn((n, wl.batch, wl.num_kv_heads, wl.head_dim), generator=gen, device="cuda").to(torch.bfloat16)
    cache.append(0, qa, ka, va)
    second = cache.decode_attention(0, q)
    torch.cuda.synchronize()
    assert cache.layer_state(0)["fill"] == 300
    _check(wl, cache, 0, q_bits, second, 300)
    assert not torch.equal(first, second)


def test_decode_full_size_qwen3_8b_layer_sampled_units():
    wl = W.WORKLOADS["qwen3_8b_k4096"]
    cache = _cache(wl, 1)
    st = W.layer_state(wl, 41, 0, 0, "gapped")
    PU.upload_layer(cache, 0, st, 0)
    cache.evict(0)
    q_bits, q = _queries(wl, 42)
    out = cache.decode_attention(0, q)
    torch.cuda.synchronize()
    _check(wl, cache, 0, q_bits, out, wl.budget_k, units=[(0, 0), (17, 3), (31, 7)])


@pytest.mark.parametrize("heads", [(1, 1), (4, 1)])
def test_decode_at_the_largest_supported_fill(heads):
    """K + B = 16640 slots in one unit (260 chunks of 64, 520 of 32): both kernels, every output checked."""
    Hq, Hkv = heads
    wl = W.shrink(SMALL, budget_k=16384, buffer_b=256, window=8, num_q_heads=Hq, num_kv_heads=Hkv, batch=1,
                  num_layers=1)
    cache = _cache(wl, 1)
    st = W.layer_state(wl, 51, 0, 0, "dense")
    PU.upload_layer(cache, 0, st, 0)
    q_bits, q = _queries(wl, 52)
    out = cache.decode_attention(0, q)
    torch.cuda.synchronize()
    _check(wl, cache, 0, q_bits, out, wl.slots)
