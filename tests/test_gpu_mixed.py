"""GPU parity of the mixed-precision values: the per-token b-bit quantizer of Sec. 4.4 with
the reserved cache of Sec. 6 (R_V and R_B keep bf16), and the decode attention that reads the other values
from their codes, against the fp64 oracle.

Codes, (s, z) and the reserved masks are integer or exactly reproducible decisions taken in fp32 on both
sides: bit-exact.  The decode output: |o_gpu - o_ref| <= 1e-4 * sum_i alpha_i |v'_i| + 1e-7, as for the bf16
decode (the dequantization v' = Q s + z is one fp32 FMA on the GPU)."""

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


def _evicted(wl, seed, **kw):
    from paper_2606_03928_gb300.vase import VaseCache
    cache = VaseCache(PU.geometry_of(wl, 1), **kw)
    st = W.layer_state(wl, seed, 0, 2, "gapped")
    PU.upload_layer(cache, 0, st, 2)
    assert cache.evict(0) == 0
    return cache


def _unpack(codes_row, bits):
    """Lane-packed codes of one row -> [d] codes: lane l holds dims 4l .. 4l+3 in 4*bits bits."""
    raw = np.asarray(codes_row, dtype=np.uint8)
    nb = bits // 2
    out = np.empty(128, dtype=np.uint8)
    for lane in range(32):
        word = int.from_bytes(raw[lane * nb:(lane + 1) * nb].tobytes(), "little")
        for e in range(4):
            out[4 * lane + e] = (word >> (e * bits)) & ((1 << bits) - 1)
    return out


def _n_v(wl):
    return wl.budget_k // 4


@pytest.mark.parametrize("bits", [2, 4, 8])
def test_quantize_matches_oracle_bit_exact(bits):
    wl = W.shrink(SMALL, budget_k=200, buffer_b=40, window=16, num_q_heads=16, num_kv_heads=8, batch=2,
                  num_layers=1)
    cache = _evicted(wl, 3)
    mb, t = cache.mixed_buffers(bits)
    cache.quantize_values(0, bits, mb)
    torch.cuda.synchronize()
    K, B = wl.budget_k, wl.buffer_b
    Kp = (K + 1) & ~1
    words = (K + 31) // 32
    row = 128 * bits // 8
    codes = t["codes"].cpu().numpy().reshape(wl.batch * wl.num_kv_heads, K, row)
    qp = t["qparams"].cpu().numpy().reshape(wl.batch * wl.num_kv_heads, Kp, 2)
    masks = t["rmask"].cpu().numpy().view(np.uint32).reshape(wl.batch * wl.num_kv_heads, words)
    v_bits = cache.v_cache[0].view(torch.int16).cpu().numpy().view(np.uint16)
    for s in range(wl.batch):
        for h in range(wl.num_kv_heads):
            u = s * wl.num_kv_heads + h
            v = O.bf16_bits_to_f64(v_bits[s, h, :K])
            reserved = O.reserved_after_eviction(O.value_magnitude(v), K, B, _n_v(wl))
            got_mask = np.array([(masks[u, j // 32] >> (j % 32)) & 1 for j in range(K)], dtype=bool)
            assert np.array_equal(got_mask, reserved), f"unit {u}: reserved mask"
            assert not np.any(masks[u, K // 32] >> np.uint32(K % 32)) if K % 32 else True
            ref_codes, ref_s, ref_z = O.quantize_values(v, bits)
            for j in np.flatnonzero(~reserved):
                assert np.array_equal(_unpack(codes[u, j], bits), ref_codes[j]), f"unit {u} slot {j}: codes"
                assert qp[u, j, 0] == ref_s[j] and qp[u, j, 1] == ref_z[j], f"unit {u} slot {j}: (s, z)"


@pytest.mark.parametrize("bits", [2, 4, 8])
@pytest.mark.parametrize("heads", [(16, 8), (32, 8)])
def test_mixed_decode_matches_oracle(bits, heads):
    Hq, Hkv = heads
    wl = W.shrink(SMALL, budget_k=256, buffer_b=64, window=16, num_q_heads=Hq, num_kv_heads=Hkv, batch=2,
                  num_layers=1)
    cache = _evicted(wl, 5)
    mb, t = cache.mixed_buffers(bits)
    cache.quantize_values(0, bits, mb)
    # pairs appended after the quantization are read in bf16
    gen = torch.Generator(device="cuda")
    gen.manual_seed(6)
    n = 37
    shape = lambda H: (n, wl.batch, H, wl.head_dim)
    cache.append(0, torch.randn(shape(Hq), generator=gen, device="cuda").to(torch.bfloat16),
                 torch.randn(shape(Hkv), generator=gen, device="cuda").to(torch.bfloat16),
                 torch.randn(shape(Hkv), generator=gen, device="cuda").to(torch.bfloat16))
    fill = wl.budget_k + n
    rng = np.random.default_rng(7)
    q_bits = W.f32_to_bf16_bits(rng.standard_normal((wl.batch, Hq, wl.head_dim)).astype(np.float32))
    out = cache.decode_attention_mixed(0, bits, mb, PU.bits_to_bf16_tensor(q_bits, "cuda"))
    torch.cuda.synchronize()
    got = out.cpu().numpy().astype(np.float64)
    k_bits = cache.k_cache[0].view(torch.int16).cpu().numpy().view(np.uint16)
    v_bits = cache.v_cache[0].view(torch.int16).cpu().numpy().view(np.uint16)
    K, B, G = wl.budget_k, wl.buffer_b, wl.group
    for s in range(wl.batch):
        for h in range(wl.num_kv_heads):
            v = O.bf16_bits_to_f64(v_bits[s, h, :fill])
            reserved = np.ones(fill, dtype=bool)
            reserved[:K] = O.reserved_after_eviction(O.value_magnitude(v[:K]), K, B, _n_v(wl))
            ref, bound = O.decode_attention_mixed(O.bf16_bits_to_f64(q_bits[s, h * G:(h + 1) * G]),
                                                  O.bf16_bits_to_f64(k_bits[s, h, :fill]), v, reserved, bits)
            g = got[s, h * G:(h + 1) * G]
            bad = np.abs(g - ref) > DEC_RTOL * bound + DEC_ATOL
            assert not bad.any(), f"unit ({s}, {h}): {bad.sum()} outputs off, worst {np.abs(g - ref).max():.3e}"


def test_mixed_decode_full_size_layer_sampled_units():
    wl = W.WORKLOADS["qwen3_1p7b_k2048"]
    cache = _evicted(wl, 9)
    mb, _ = cache.mixed_buffers(4)
    cache.quantize_values(0, 4, mb)
    rng = np.random.default_rng(10)
    q_bits = W.f32_to_bf16_bits(rng.standard_normal((wl.batch, wl.num_q_heads, wl.head_dim)).astype(np.float32))
    out = cache.decode_attention_mixed(0, 4, mb, PU.bits_to_bf16_tensor(q_bits, "cuda"))
    torch.cuda.synchronize()
    got = out.cpu().numpy().astype(np.float64)
    k_bits = cache.k_cache[0].view(torch.int16).cpu().numpy().view(np.uint16)
    v_bits = cache.v_cache[0].view(torch.int16).cpu().numpy().view(np.uint16)
    K, B, G = wl.budget_k, wl.buffer_b, wl.group
    for s, h in [(0, 0), (4, 3), (7, 7)]:
        v = O.bf16_bits_to_f64(v_bits[s, h, :K])
        reserved = O.reserved_after_eviction(O.value_magnitude(v), K, B, _n_v(wl))
        ref, bound = O.decode_attention_mixed(O.bf16_bits_to_f64(q_bits[s, h * G:(h + 1) * G]),
                                              O.bf16_bits_to_f64(k_bits[s, h, :K]), v, reserved, 4)
        assert not (np.abs(got[s, h * G:(h + 1) * G] - ref) > DEC_RTOL * bound + DEC_ATOL).any()


def test_mixed_values_status_checks():
    from paper_2606_03928_gb300.vase import VaseCache, VaseError
    wl = W.shrink(SMALL, budget_k=128, buffer_b=32, window=8, batch=1, num_layers=1)
    cache = VaseCache(PU.geometry_of(wl, 1))
    mb, _ = cache.mixed_buffers(4)
    with pytest.raises(VaseError):        # no eviction yet
        cache.quantize_values(0, 4, mb)
    st = W.layer_state(wl, 1, 0, 0, "gapped")
    PU.upload_layer(cache, 0, st, 0)
    assert cache.evict(0) == 0
    with pytest.raises(VaseError):        # bits must be 2, 4 or 8
        cache.quantize_values(0, 3, mb)
    q = torch.zeros((wl.batch, wl.num_q_heads, wl.head_dim), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(VaseError):        # no codes for this round
        cache.decode_attention_mixed(0, 4, mb, q)
    cache.quantize_values(0, 4, mb)
    cache.decode_attention_mixed(0, 4, mb, q)
    with pytest.raises(VaseError):        # codes of another bit width
        cache.decode_attention_mixed(0, 8, mb, q)
    rnd = VaseCache(PU.geometry_of(wl, 1), reserve="random")
    PU.upload_layer(rnd, 0, st, 0)
    assert rnd.evict(0) == 0
    mb2, t2 = rnd.mixed_buffers(4)
    with pytest.raises(VaseError):        # a random R_V cannot be recovered from the kept values
        rnd.quantize_values(0, 4, mb2)


def test_mixed_decode_at_the_largest_budget():
    """K = 16384: 512 mask words per unit, the most the mixed decode holds."""
    wl = W.shrink(SMALL, budget_k=16384, buffer_b=256, window=8, num_q_heads=2, num_kv_heads=1, batch=1,
                  num_layers=1)
    cache = _evicted(wl, 61)
    mb, _ = cache.mixed_buffers(4)
    cache.quantize_values(0, 4, mb)
    rng = np.random.default_rng(62)
    q_bits = W.f32_to_bf16_bits(rng.standard_normal((1, 2, wl.head_dim)).astype(np.float32))
    out = cache.decode_attention_mixed(0, 4, mb, PU.bits_to_bf16_tensor(q_bits, "cuda"))
    torch.cuda.synchronize()
    K, B = wl.budget_k, wl.buffer_b
    k_bits = cache.k_cache[0].view(torch.int16).cpu().numpy().view(np.uint16)
    v_bits = cache.v_cache[0].view(torch.int16).cpu().numpy().view(np.uint16)
    v = O.bf16_bits_to_f64(v_bits[0, 0, :K])
    reserved = O.reserved_after_eviction(O.value_magnitude(v), K, B, K // 4)
    ref, bound = O.decode_attention_mixed(O.bf16_bits_to_f64(q_bits[0]), O.bf16_bits_to_f64(k_bits[0, 0, :K]), v,
                                          reserved, 4)
    assert not (np.abs(out.cpu().numpy()[0].astype(np.float64) - ref) > DEC_RTOL * bound + DEC_ATOL).any()
