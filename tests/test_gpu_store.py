"""GPU parity of the compressed value store (value_bits = 2, 4, 8), the mixed-precision value cache of Sec. 6
built on the quantizer of Sec. 4.4: a reserved bf16 ring of N_v + 2B rows that spills its earliest value when an
append finds it full, evictions that quantize the kept values leaving R_V u R_B, and the decode attention that
reads the store.  Checked against the oracle's store model, driven by the same appends and by the GPU's own kept
lists (the selection has its own parity tests; here R_V comes from the oracle's ranking of the exact value
magnitudes, ties to the lower slot, as on the GPU).

Bit-exact: the ring rows at their positions, the bf16 mask, the ring (head, count), the codes and (s, z) of every
coded slot (integers and fp32 values decided in fp32 on both sides), the kept keys and positions.  The decode
output: within 1e-4 * sum_i alpha_i tau_i + 1e-7, tau_i = |v_i| for a bf16 value and |Q_i s_i| + |z_i| for a coded
one (the bound of the mixed decode's parity test)."""

import numpy as np
import pytest
import torch

from oracle import vase_oracle as O
from paper_2606_03928_gb300 import workloads as W
import parity_utils as PU

pytestmark = pytest.mark.gpu

DEC_RTOL = 1e-4
DEC_ATOL = 1e-7


def _unpack(rows, bits):
    """Lane-packed code rows [n, 16 b] -> codes [n, 128]: dim i at bits (i mod 4) * b of lane i // 4's field,
    the fields little-endian in byte order, so the codes follow each other in bit order."""
    raw = np.ascontiguousarray(rows, dtype=np.uint8)
    b = np.unpackbits(raw, axis=1, bitorder="little").reshape(raw.shape[0], 128, bits).astype(np.uint32)
    return (b << np.arange(bits, dtype=np.uint32)).sum(axis=2).astype(np.uint8)


class Model:
    """Host copy of one layer: each unit's slot contents (k, v bits and positions) and the oracle's store."""

    def __init__(self, geo, n_v):
        self.N = geo.budget_k + geo.buffer_b
        self.units = geo.batch * geo.num_kv_heads
        self.k = np.zeros((self.units, self.N, 128), np.uint16)
        self.v = np.zeros((self.units, self.N, 128), np.uint16)
        self.pos = np.full((self.units, self.N), -1, np.int64)
        self.vm = np.zeros((self.units, self.N))   # value magnitudes (Range) of the slots' values
        H = O.store_capacity(geo.budget_k, geo.buffer_b, n_v)
        self.store = [O.store_new(H) for _ in range(self.units)]
        self.fill = 0
        self.next_pos = 0
        self.n_v = n_v
        self.geo = geo

    def append(self, k, v):
        n = k.shape[0]
        Hkv = self.geo.num_kv_heads
        for u in range(self.units):
            s, h = divmod(u, Hkv)
            self.k[u, self.fill:self.fill + n] = k[:, s, h]
            self.v[u, self.fill:self.fill + n] = v[:, s, h]
            self.pos[u, self.fill:self.fill + n] = np.arange(self.next_pos, self.next_pos + n)
            self.vm[u, self.fill:self.fill + n] = O.value_magnitude(O.bf16_bits_to_f64(v[:, s, h]))
            O.store_append(self.store[u], self.fill, n, self.vm[u], self.geo.budget_k, self.n_v)
        self.fill += n
        self.next_pos += n

    def evict(self, src_all):
        K = self.geo.budget_k
        for u in range(self.units):
            src = src_all[u].astype(np.int64)
            r_v = O.top_k_slots(self.vm[u, :K], self.n_v)
            resnew = (src >= K) | np.isin(src, r_v)
            O.store_evict(self.store[u], src, resnew)
            for arr in (self.k, self.v, self.vm):
                arr[u, :K] = arr[u, src]
            self.pos[u, :K] = self.pos[u, src]
            self.pos[u, K:] = -1
        self.fill = K


def _check_store(cache, layer, model, bits, after_evict=False):
    torch.cuda.synchronize()
    vs = cache.value_store(layer)
    codes = vs["codes"].cpu().numpy()
    sz = vs["sz"].cpu().numpy()
    mask = vs["mask"].cpu().numpy().view(np.uint32)
    ring = vs["ring"].view(torch.int16).cpu().numpy().view(np.uint16)
    state = vs["state"].cpu().numpy()
    H = vs["ring_rows"]
    fill = model.fill
    assert vs["fill"] == fill
    for u in range(model.units):
        st = model.store[u]
        assert state[u, 0] == st["head"] and state[u, 1] == len(st["slots"]), f"unit {u}: ring state"
        bf = O.store_reserved_mask(st, model.N)
        if after_evict:  # R_V and R_B are all bf16 (the first fill kept the large-Range values)
            assert bf[:model.fill].sum() == model.n_v + model.geo.buffer_b, f"unit {u}: reserved count"
        got = np.array([(mask[u, j >> 5] >> np.uint32(j & 31)) & 1 for j in range(model.N)], dtype=bool)
        assert np.array_equal(got, bf), f"unit {u}: bf16 mask"
        for s, p in O.store_ring_positions(st).items():
            assert np.array_equal(ring[u, p], model.v[u, s]), f"unit {u}: ring row of slot {s}"
        coded = np.flatnonzero(~bf[:fill])
        if coded.size:
            ref_c, ref_s, ref_z = O.quantize_values(O.bf16_bits_to_f64(model.v[u, coded]), bits)
            assert np.array_equal(_unpack(codes[u, coded], bits), ref_c), f"unit {u}: codes"
            assert np.array_equal(sz[u, coded, 0], ref_s) and np.array_equal(sz[u, coded, 1], ref_z), \
                f"unit {u}: (s, z)"


def _check_keys(cache, layer, model):
    torch.cuda.synchronize()
    k = cache.k_cache[layer].view(torch.int16).cpu().numpy().view(np.uint16)
    pos = cache.positions[layer].cpu().numpy()
    Hkv = model.geo.num_kv_heads
    for u in range(model.units):
        s, h = divmod(u, Hkv)
        assert np.array_equal(k[s, h, :model.fill], model.k[u, :model.fill]), f"unit {u}: keys"
        assert np.array_equal(pos[s, h, :model.fill], model.pos[u, :model.fill]), f"unit {u}: positions"


def _check_decode(cache, layer, model, bits, rng):
    geo = model.geo
    G = geo.num_q_heads // geo.num_kv_heads
    q_bits = W.f32_to_bf16_bits(rng.standard_normal((geo.batch, geo.num_q_heads, 128)).astype(np.float32))
    out = cache.decode_attention(layer, PU.bits_to_bf16_tensor(q_bits, cache.device)).cpu().numpy()
    for u in range(model.units):
        s, h = divmod(u, geo.num_kv_heads)
        q = O.bf16_bits_to_f64(q_bits[s, h * G:(h + 1) * G])
        keys = O.bf16_bits_to_f64(model.k[u, :model.fill])
        vals = O.bf16_bits_to_f64(model.v[u, :model.fill])
        bf = O.store_reserved_mask(model.store[u], model.N)[:model.fill]
        ref, scale = O.decode_attention_mixed(q, keys, vals, bf, bits)
        err = np.abs(out[s, h * G:(h + 1) * G] - ref)
        assert np.all(err <= DEC_RTOL * scale + DEC_ATOL), f"unit {u}: decode error {err.max()}"


def _stream(rng, n, geo, layers):
    """n decode steps of every layer: q [L, n, b, Hq, d], k / v [L, n, b, Hkv, d] bf16 bits; keys N(0, 1), values
    N(0, 1) with 2 % of rows scaled by 20 (large-Range outliers)."""
    L, b = layers, geo.batch
    q = rng.standard_normal((L, n, b, geo.num_q_heads, 128)).astype(np.float32)
    k = rng.standard_normal((L, n, b, geo.num_kv_heads, 128)).astype(np.float32)
    v = rng.standard_normal((L, n, b, geo.num_kv_heads, 128)).astype(np.float32)
    v[rng.random((L, n, b, geo.num_kv_heads)) < 0.02] *= 20
    return W.f32_to_bf16_bits(q), W.f32_to_bf16_bits(k), W.f32_to_bf16_bits(v)


def _append(cache, models, rng, n, layers):
    geo = models[0].geo
    q, k, v = _stream(rng, n, geo, layers)
    for l in range(layers):
        dev = cache.device
        cache.append(l, PU.bits_to_bf16_tensor(q[l], dev), PU.bits_to_bf16_tensor(k[l], dev),
                     PU.bits_to_bf16_tensor(v[l], dev))
        models[l].append(k[l], v[l])


def _run_rounds(geo, n_v, bits, prefill, rounds, seed, decode=True, evict_all=False):
    from paper_2606_03928_gb300.vase import VaseCache
    layers = geo.num_layers
    cache = VaseCache(geo, n_v=n_v, value_bits=bits, debug_outputs=True, seed=seed)
    models = [Model(geo, n_v) for _ in range(layers)]
    rng = np.random.default_rng(seed)
    for n in prefill:  # the first fill, in pieces: the ring overflows across and within calls
        _append(cache, models, rng, n, layers)
        for l in range(layers):
            _check_store(cache, l, models[l], bits)
    _check_keys(cache, 0, models[0])
    for r in range(rounds):
        if evict_all:
            assert cache.evict_all() == layers
        for l in range(layers):
            if not evict_all:
                assert cache.evict(l) == 0
                srcs = cache.debug_view(0)["src"].cpu().numpy()
            else:
                srcs = cache.debug_view(l)["src"].cpu().numpy()
            models[l].evict(srcs)
            _check_store(cache, l, models[l], bits, after_evict=True)
            _check_keys(cache, l, models[l])
        if decode:
            _check_decode(cache, 0, models[0], bits, rng)
        # the next round's B values: one step at a time, then the rest in one call
        steps = [1, 1, 1, geo.buffer_b - 3]
        for i, n in enumerate(steps):
            _append(cache, models, rng, n, layers)
            if i == 0 and decode and r == 0:  # a ragged last chunk, one slot past K
                _check_decode(cache, 0, models[0], bits, rng)
            if i == 1:
                for l in range(layers):
                    _check_store(cache, l, models[l], bits)
        if decode and r == 0:
            _check_decode(cache, 0, models[0], bits, rng)
    assert cache.check_device_error()[0] == 0
    return cache, models


@pytest.mark.parametrize("bits", [2, 4, 8])
def test_store_chained_rounds_match_oracle(bits):
    """K 256, B 64, W 32, 16/8 heads, two sequences, two layers, N_v 64 (H = 192 ring rows): a first fill of 320
    values in pieces of 250 (58 quantized inside the call, the large-Range ones kept), 1, 40 and 29, then four
    rounds of eviction and 64 appends."""
    from paper_2606_03928_gb300.vase import Geometry
    geo = Geometry(256, 64, 32, 16, 8, 2, 2)
    _run_rounds(geo, 64, bits, [250, 1, 40, 29], 4, seed=bits)


def test_store_batched_evictions_and_small_ring():
    """evict_all over three layers; N_v 0 (the ring holds R_B only, H = 2B) and a fill in single steps at first."""
    from paper_2606_03928_gb300.vase import Geometry
    geo = Geometry(128, 32, 16, 8, 8, 1, 3)
    _run_rounds(geo, 0, 4, [1] * 5 + [155], 3, seed=11, evict_all=True)


@pytest.mark.parametrize("bits", [2, 4, 8])
def test_store_grouped_query_heads_decode(bits):
    """G = 4 and G = 8 query heads per KV head read the store on the tensor cores (as G = 1 and 2 do in the tests
    above): bf16 rows from the ring and the other rows expanded from their codes into the V tile; a first fill of
    256 in one call (80 quantized in it), K 192 (three whole 64-slot chunks) and ragged fills."""
    from paper_2606_03928_gb300.vase import Geometry
    for hq, seed in ((32, 21), (64, 22)):
        geo = Geometry(192, 64, 16, hq, 8, 1, 1)
        _run_rounds(geo, 48, bits, [256], 2, seed=seed + bits)


def test_store_decode_sixteen_query_heads():
    """G = 16 (64 query heads over 4 KV heads): the 32-column form of the tensor-core decode over the store."""
    from paper_2606_03928_gb300.vase import Geometry
    geo = Geometry(128, 32, 16, 64, 4, 1, 1)
    _run_rounds(geo, 32, 4, [160], 2, seed=41)


def test_store_decode_qwen3_8b_geometry_sampled():
    """A larger unit on the tensor-core path: K 1024, B 128, 32/8 heads (G = 4), two sequences, 4 bits, the ring
    wrapped by several rounds; a decode step after every eviction."""
    from paper_2606_03928_gb300.vase import Geometry
    geo = Geometry(1024, 128, 32, 32, 8, 2, 1)
    _run_rounds(geo, 256, 4, [700, 452], 3, seed=31)


def test_store_refuses_a_state_it_did_not_write():
    """A ring head out of range (a store this library did not write): the append kernel records the error site
    and writes nothing, without touching the ring; the decode reads with head 0 and records it too."""
    from paper_2606_03928_gb300 import vase as V
    from paper_2606_03928_gb300.vase import Geometry, VaseCache
    geo = Geometry(128, 32, 16, 8, 8, 1, 1)
    cache = VaseCache(geo, n_v=16, value_bits=4, seed=3)
    models = [Model(geo, 16)]
    rng = np.random.default_rng(3)
    _append(cache, models, rng, 10, 1)
    assert cache.check_device_error()[0] == 0
    vs = cache.value_store(0)
    before = vs["ring"].clone()
    vs["state"][0, 0] = vs["ring_rows"] + 5
    _append(cache, models, rng, 1, 1)
    status, code = cache.check_device_error()
    assert status != 0 and code & 0x80000000 and (code & 0xFFFF) == V.VASE_SITE_STORE_STATE, (status, code)
    torch.cuda.synchronize()
    assert torch.equal(cache.value_store(0)["ring"][0], before[0])
    q = torch.zeros((1, 8, 128), dtype=torch.bfloat16, device=cache.device)
    cache.decode_attention(0, q)
    status, code = cache.check_device_error()
    assert status != 0 and code & 0x80000000, (status, code)  # the decode's own site; the context stays usable
    assert cache.check_device_error()[0] == 0



def test_store_qwen3_1p7b_geometry_batched_sampled_units():
    """The bench's store configuration at full unit size: Qwen3-1.7B geometry (K 2048, B 128, W 32, 16/8 heads,
    batch 8: 64 units per layer), two layers, 4 bits, appended and evicted through the batched all-layer calls
    the bench times (vase_append_all, vase_evict_all).  The first fill of 2176 values in two pieces overflows the
    768-row ring; then three rounds.  Eight sampled units of each layer are checked bit-exactly against the
    oracle's store model after every eviction, and decoded."""
    from paper_2606_03928_gb300.vase import Geometry, VaseCache
    geo = Geometry(2048, 128, 32, 16, 8, 2, 8)
    nv, bits, L = 512, 4, 2
    cache = VaseCache(geo, n_v=nv, value_bits=bits, debug_outputs=True, seed=5)
    rng = np.random.default_rng(55)
    sample = sorted(rng.choice(64, 8, replace=False).tolist())
    models = [Model(geo, nv) for _ in range(L)]
    dev = cache.device

    def append_all(n):
        q, k, v = _stream(rng, n, geo, L)
        cache.append_all(PU.bits_to_bf16_tensor(q, dev), PU.bits_to_bf16_tensor(k, dev),
                         PU.bits_to_bf16_tensor(v, dev))
        for l in range(L):
            models[l].append(k[l], v[l])

    def check_sampled(l, after_evict):
        torch.cuda.synchronize()
        vs = cache.value_store(l)
        codes, sz = vs["codes"].cpu().numpy(), vs["sz"].cpu().numpy()
        mask = vs["mask"].cpu().numpy().view(np.uint32)
        ring = vs["ring"].view(torch.int16).cpu().numpy().view(np.uint16)
        state = vs["state"].cpu().numpy()
        m = models[l]
        for u in sample:
            st = m.store[u]
            assert state[u, 0] == st["head"] and state[u, 1] == len(st["slots"]), f"layer {l} unit {u}: ring state"
            bf = O.store_reserved_mask(st, m.N)
            if after_evict:
                assert bf[:m.fill].sum() == nv + geo.buffer_b
            got = np.unpackbits(mask[u].view(np.uint8), bitorder="little")[:m.N].astype(bool)
            assert np.array_equal(got, bf), f"layer {l} unit {u}: mask"
            pos = O.store_ring_positions(st)
            slots = np.array(st["slots"], dtype=np.int64)
            assert np.array_equal(ring[u, [pos[s] for s in st["slots"]]], m.v[u, slots]), f"layer {l} unit {u}: ring"
            coded = np.flatnonzero(~bf[:m.fill])
            rc, rs, rz = O.quantize_values(O.bf16_bits_to_f64(m.v[u, coded]), bits)
            assert np.array_equal(_unpack(codes[u, coded], bits), rc), f"layer {l} unit {u}: codes"
            assert np.array_equal(sz[u, coded, 0], rs) and np.array_equal(sz[u, coded, 1], rz)

    append_all(1500)
    append_all(676)
    for l in range(L):
        check_sampled(l, False)
    for r in range(3):
        assert cache.evict_all() == L
        for l in range(L):
            models[l].evict(cache.debug_view(l)["src"].cpu().numpy())
            check_sampled(l, True)
        # decode of layer 1 on the sampled units
        G = geo.num_q_heads // geo.num_kv_heads
        q_bits = W.f32_to_bf16_bits(rng.standard_normal((geo.batch, geo.num_q_heads, 128)).astype(np.float32))
        out = cache.decode_attention(1, PU.bits_to_bf16_tensor(q_bits, dev)).cpu().numpy()
        m = models[1]
        for u in sample:
            s, h = divmod(u, geo.num_kv_heads)
            ref, scale = O.decode_attention_mixed(O.bf16_bits_to_f64(q_bits[s, h * G:(h + 1) * G]),
                                                  O.bf16_bits_to_f64(m.k[u, :m.fill]), O.bf16_bits_to_f64(m.v[u, :m.fill]),
                                                  O.store_reserved_mask(m.store[u], m.N)[:m.fill], bits)
            assert np.all(np.abs(out[s, h * G:(h + 1) * G] - ref) <= DEC_RTOL * scale + DEC_ATOL), f"unit {u}: decode"
        append_all(geo.buffer_b)
    assert cache.check_device_error()[0] == 0


def test_store_refuses_the_bf16_cache_calls():
    """With the store, the calls that need bf16 value rows -- the magnitude refresh, the read path's quantizer
    and its mixed decode -- return VASE_ERR_UNSUPPORTED and launch nothing; the view reports no V rows."""
    from paper_2606_03928_gb300 import vase as V
    from paper_2606_03928_gb300.vase import Geometry, VaseCache
    cache = VaseCache(Geometry(128, 32, 16, 8, 8, 1, 1), n_v=16, value_bits=2, seed=1)
    n0 = cache.launch_count()
    for call in (lambda: cache.refresh_value_scores(0),
                 lambda: cache.quantize_values(0, 2, cache.mixed_buffers(2)[0])):
        with pytest.raises(V.VaseError) as exc:
            call()
        assert exc.value.status == V.VASE_ERR_UNSUPPORTED
    mb, _ = cache.mixed_buffers(2)
    q = torch.zeros((1, 8, 128), dtype=torch.bfloat16, device=cache.device)
    with pytest.raises(V.VaseError) as exc:
        cache.decode_attention_mixed(0, 2, mb, q)
    assert exc.value.status == V.VASE_ERR_UNSUPPORTED
    assert cache.launch_count() == n0
    import ctypes
    kv = V.vase_kv_view()
    assert V.load().vase_kv_view_get(cache.ctx, 0, ctypes.byref(kv)) == 0
    assert kv.k and not kv.v
