"""GPU parity of the VaSE eviction step (C ABI -> CUDA kernels) against the fp64 oracle.

Inputs are the seeded synthetic workloads; every expected value comes from
the oracle or from the definition of a pure data movement.
"""

import itertools

import numpy as np
import pytest
import torch

from oracle import vase_oracle as O
from paper_2606_03928_gb300 import workloads as W
import parity_utils as PU

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_03928_gb300 import build
    build.build()
    from paper_2606_03928_gb300 import vase as V
    V.load()


def _cache(wl, num_layers, variant="attnv", debug=True, **kw):
    from paper_2606_03928_gb300.vase import VaseCache
    return VaseCache(PU.geometry_of(wl, num_layers), variant=variant, debug_outputs=debug, **kw)


def _run_layer(wl, *, variant="attnv", layer=1, num_layers=2, round_index=3, seed=0, data_seed=0, units=None,
               debug=True, positions="gapped", cache_kw=None, oracle_kw=None, state_round=None, cache=None,
               edit=None):
    """Uploads one layer, evicts it through the C ABI and checks `units` (default all) against the oracle.

    round_index is the eviction counter (it keys the noise); state_round (default round_index) draws the data.
    """
    cache_kw = dict(cache_kw or {})
    oracle_kw = dict(oracle_kw or {})
    if cache is None:
        cache = _cache(wl, num_layers, variant=variant, debug=debug, seed=seed, **cache_kw)
    st = W.layer_state(wl, data_seed, layer, round_index if state_round is None else state_round, positions)
    if edit is not None:
        edit(st)
    PU.upload_layer(cache, layer, st, round_index)
    other = None
    if num_layers > 1:
        other_layer = 0 if layer != 0 else 1
        other = W.layer_state(wl, data_seed + 1, other_layer, 0, "dense")
        PU.upload_layer(cache, other_layer, other, 0)
    assert cache.evict(layer) == 0
    status, code = cache.check_device_error()
    assert status == 0, f"device error word {code:#x}"
    got = PU.download(cache, layer)
    if other is not None:
        rest = PU.download(cache, other_layer)
        assert np.array_equal(rest["k_bits"], other["k_bits"]), "another layer was modified"
    st_after = cache.layer_state(layer)
    assert st_after["fill"] == wl.budget_k and st_after["round"] == round_index + 1
    nv = oracle_kw.get("n_v", -1)
    nv = wl.budget_k // 4 if nv is None or nv < 0 else nv
    if variant == "dkv":
        nv = 0
    flips = 0
    todo = units if units is not None else [(s, h) for s in range(wl.batch) for h in range(wl.num_kv_heads)]
    for (s, h) in todo:
        ref = PU.oracle_unit(wl, st, s, h, variant=variant, round_index=round_index, seed=seed, layer=layer,
                             **oracle_kw)
        gu = PU.unit_slice(got, s, h, wl.num_kv_heads)
        if not debug:
            gu["pooled"] = None
            gu["key"] = None
            if variant == "attnv":  # written to the workspace only with debug outputs (DKV always writes it)
                gu["value_score"] = None
        flips += PU.check_unit(wl, ref, gu, st["k_bits"][s, h], st["v_bits"][s, h], st["positions"][s, h],
                               variant=variant, n_v=nv, value_kind=cache_kw.get("value_score", O.VALUE_RANGE))
    # properties that hold at any size, checked on every unit
    K, B = wl.budget_k, wl.buffer_b
    for s in range(wl.batch):
        for h in range(wl.num_kv_heads):
            u = s * wl.num_kv_heads + h
            src = got["src"][u]
            assert len(set(src.tolist())) == K and set(range(K, K + B)) <= set(src.tolist())
    return cache, st, got, flips


# ----------------------------------------------------------------------------- small configurations

SMALL = W.WORKLOADS["single_layer_k256"]


def test_single_layer_k256_all_units_match_oracle():
    _, _, _, flips = _run_layer(SMALL, layer=0, num_layers=1, round_index=0, positions="dense")
    assert flips <= 2


# Launch-bound single-layer evictions of small units run the fused kernel (score held in TMEM, selection and
# gather in the same launch).  Its edges: 128 window rows (a whole 128-column TMEM block per tile), a ragged last
# tile, four tiles of 128 rows (all 512 TMEM columns, and K rows of K and V filling most of shared memory), debug
# outputs off, GQA max-aggregation and noise off.
@pytest.mark.parametrize("K,B,Wn,Hq,Hkv,kw", [
    (256, 64, 32, 32, 8, {}),                      # G*W = 128
    (200, 40, 16, 16, 8, {}),                      # N = 240: a ragged last tile
    (320, 192, 32, 32, 8, {}),                     # N = 512, G*W = 128: 512 TMEM columns
    (256, 64, 32, 16, 8, {"debug": False}),
    (256, 64, 16, 32, 8, {"gqa": "max"}),
    (256, 64, 32, 16, 8, {"stochastic": False}),
])
def test_fused_small_unit_eviction_matches_oracle(K, B, Wn, Hq, Hkv, kw):
    kw = dict(kw)
    debug = kw.pop("debug", True)
    wl = W.shrink(SMALL, budget_k=K, buffer_b=B, window=Wn, num_q_heads=Hq, num_kv_heads=Hkv, batch=2, num_layers=2)
    _, _, _, flips = _run_layer(wl, debug=debug, cache_kw=kw, oracle_kw=kw)
    assert flips <= 4


def test_layer_offset_and_gapped_positions():
    _run_layer(SMALL, layer=1, num_layers=2, round_index=5)


@pytest.mark.parametrize("value_score", [O.VALUE_L2, O.VALUE_VAR])
def test_value_score_variants(value_score):
    _run_layer(SMALL, cache_kw={"value_score": value_score}, oracle_kw={"value_score": value_score})


def test_deterministic_top_k_and_no_pooling():
    _run_layer(SMALL, cache_kw={"stochastic": False, "pool_kernel": 1},
               oracle_kw={"stochastic": False, "pool_kernel": 1})


def test_no_value_reservation():
    _run_layer(SMALL, cache_kw={"n_v": 0}, oracle_kw={"n_v": 0})


@pytest.mark.parametrize("K,B,Wn,Hq,Hkv", [(100, 27, 5, 6, 3), (130, 1, 1, 2, 2), (8, 2, 3, 4, 1),
                                          (384, 128, 64, 8, 2), (200, 50, 20, 24, 8)])
def test_ragged_geometries(K, B, Wn, Hq, Hkv):
    wl = W.shrink(SMALL, budget_k=K, buffer_b=B, window=Wn, num_q_heads=Hq, num_kv_heads=Hkv, batch=2,
                  num_layers=2)
    _run_layer(wl, cache_kw={"n_v": K // 5}, oracle_kw={"n_v": K // 5})


def test_seed_changes_selection():
    a = _run_layer(SMALL, seed=1)[2]["src"]
    b = _run_layer(SMALL, seed=2)[2]["src"]
    assert not np.array_equal(a, b)


def test_dkv_small_all_units():
    _run_layer(SMALL, variant="dkv", layer=0, num_layers=1, oracle_kw={"dkv_rank": 20})


@pytest.mark.parametrize("r", [1, 7, 32])
def test_dkv_ranks(r):
    _run_layer(SMALL, variant="dkv", cache_kw={"dkv_rank": r}, oracle_kw={"dkv_rank": r})


def test_dkv_fixed_g_is_round_independent():
    a = _run_layer(SMALL, variant="dkv", round_index=2, state_round=2, cache_kw={"dkv_fixed_g": True},
                   oracle_kw={"dkv_fixed_g": True})[2]
    b = _run_layer(SMALL, variant="dkv", round_index=9, state_round=2, cache_kw={"dkv_fixed_g": True},
                   oracle_kw={"dkv_fixed_g": True})[2]
    c = _run_layer(SMALL, variant="dkv", round_index=9, state_round=2)[2]
    assert np.array_equal(a["src"], b["src"])
    assert not np.array_equal(b["src"], c["src"])


# ----------------------------------------------------------------------------- append path

def test_append_writes_cache_ring_and_positions():
    wl = W.shrink(SMALL, budget_k=64, buffer_b=16, window=8, batch=2, num_layers=2)
    cache = _cache(wl, 2)
    N = wl.slots
    chunk = W.stream_chunk(wl, 3, 1, 0, N)
    dev = cache.device
    q = PU.bits_to_bf16_tensor(chunk["q_bits"], dev)
    k = PU.bits_to_bf16_tensor(chunk["k_bits"], dev)
    v = PU.bits_to_bf16_tensor(chunk["v_bits"], dev)
    assert cache.append(1, q[:50], k[:50], v[:50]) == 0
    assert cache.append(1, q[50:], k[50:], v[50:]) == 1  # full: eviction due
    torch.cuda.synchronize()
    kb = cache.k_cache[1].view(torch.int16).cpu().numpy().view(np.uint16)
    vb = cache.v_cache[1].view(torch.int16).cpu().numpy().view(np.uint16)
    qb = cache.q_window[1].view(torch.int16).cpu().numpy().view(np.uint16)
    pos = cache.positions[1].cpu().numpy()
    assert np.array_equal(kb, chunk["k_bits"].transpose(1, 2, 0, 3))
    assert np.array_equal(vb, chunk["v_bits"].transpose(1, 2, 0, 3))
    assert np.array_equal(pos, np.broadcast_to(np.arange(N), pos.shape))
    # ring slot (t mod W) holds the query of step t for the last W steps
    for t in range(N - wl.window, N):
        assert np.array_equal(qb[:, :, t % wl.window], chunk["q_bits"][t])
    with pytest.raises(Exception):
        cache.append(1, q[:1], k[:1], v[:1])  # full
    st = cache.layer_state(1)
    assert st["fill"] == N and st["next_position"] == N and st["queries_seen"] == N


@pytest.mark.parametrize("pinned", [True, False])
def test_host_append_and_read_positions_match_device_append(pinned):
    """Host appends equal device appends: page-locked inputs are read by the kernel in place, pageable ones
    go through the staging copies (only the query rows of the last W steps are copied)."""
    wl = W.shrink(SMALL, budget_k=64, buffer_b=16, window=8, batch=2, num_layers=1)
    a = _cache(wl, 1)
    b = _cache(wl, 1)
    chunk = W.stream_chunk(wl, 5, 0, 0, wl.slots)
    tq = torch.from_numpy(chunk["q_bits"].view(np.int16)).view(torch.bfloat16)
    tk = torch.from_numpy(chunk["k_bits"].view(np.int16)).view(torch.bfloat16)
    tv = torch.from_numpy(chunk["v_bits"].view(np.int16)).view(torch.bfloat16)
    for s in range(0, wl.slots, wl.buffer_b):
        e = min(wl.slots, s + wl.buffer_b)
        a.append(0, tq[s:e].cuda().contiguous(), tk[s:e].cuda().contiguous(), tv[s:e].cuda().contiguous())
        host = [x[s:e].contiguous() for x in (tq, tk, tv)]
        if pinned:
            host = [x.pin_memory() for x in host]
        b.append_host(0, *host)
        torch.cuda.synchronize()  # the pageable inputs are reused by the next iteration
    torch.cuda.synchronize()
    assert torch.equal(a.q_window, b.q_window)
    assert torch.equal(a.value_scores, b.value_scores)
    a.evict(0)
    b.evict(0)
    torch.cuda.synchronize()
    assert torch.equal(a.k_cache, b.k_cache) and torch.equal(a.v_cache, b.v_cache)
    out = torch.empty((wl.batch, wl.num_kv_heads, wl.budget_k), dtype=torch.int32).pin_memory()
    b.read_positions(0, out)
    torch.cuda.synchronize()
    assert torch.equal(out, b.positions[0, :, :, :wl.budget_k].cpu())


def test_status_codes():
    from paper_2606_03928_gb300 import vase as V
    wl = W.shrink(SMALL, budget_k=64, buffer_b=16, window=8, batch=1, num_layers=1)
    c = _cache(wl, 1)
    with pytest.raises(V.VaseError) as ei:
        c.evict(0)
    assert ei.value.status == V.VASE_ERR_NOT_FULL
    with pytest.raises(V.VaseError) as ei:
        c.evict(3)
    assert ei.value.status == V.VASE_ERR_INVALID
    q = torch.zeros((1, 1, wl.num_q_heads, 128), dtype=torch.bfloat16, device="cuda")
    k = torch.zeros((1, 1, wl.num_kv_heads, 128), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(V.VaseError) as ei:
        V.vase_append(c.ctx, 0, q.data_ptr() + 2, k.data_ptr(), k.data_ptr(), 1)
    assert ei.value.status == V.VASE_ERR_ALIGN
    assert c.check_device_error()[0] == 0


# ----------------------------------------------------------------------------- chained rounds

def test_chained_rounds_follow_the_oracle_until_a_threshold_tie():
    """Appends B new tokens and evicts, 6 rounds in a row; the oracle chains its own state."""
    wl = W.shrink(SMALL, budget_k=256, buffer_b=64, window=32, batch=1, num_layers=1)
    cache = _cache(wl, 1)
    N, K, B = wl.slots, wl.budget_k, wl.buffer_b
    dev = cache.device
    first = W.stream_chunk(wl, 11, 0, 0, N)
    cache.append(0, *(PU.bits_to_bf16_tensor(first[x], dev) for x in ("q_bits", "k_bits", "v_bits")))
    G = wl.group
    state_k = first["k_bits"].transpose(1, 2, 0, 3).copy()
    state_v = first["v_bits"].transpose(1, 2, 0, 3).copy()
    pos = np.broadcast_to(np.arange(N), (wl.batch, wl.num_kv_heads, N)).copy()
    qhist = [first["q_bits"][t] for t in range(N)]
    compared = 0
    for rnd in range(6):
        cache.evict(0)
        got = PU.download(cache, 0)
        qwin = np.stack(qhist[-wl.window:], axis=2)  # [b, Hq, W, d]
        same = True
        for h in range(wl.num_kv_heads):
            ref = O.evict_unit_bits(qwin[0, h * G:(h + 1) * G].reshape(-1, 128), state_k[0, h], state_v[0, h],
                                    pos[0, h], budget_k=K, buffer_b=B, seed=0, layer=0, seq=0, head=h,
                                    num_kv_heads=wl.num_kv_heads, rnd=rnd)
            gu = PU.unit_slice(got, 0, h, wl.num_kv_heads)
            PU.check_unit(wl, ref, gu, state_k[0, h], state_v[0, h], pos[0, h], variant="attnv", n_v=K // 4)
            same &= np.array_equal(gu["src"], ref["src"])
            state_k[0, h, :K] = ref["k_bits_new"]
            state_v[0, h, :K] = ref["v_bits_new"]
            pos[0, h, :K] = ref["positions_new"]
        compared += 1
        if not same:
            break
        nxt = W.stream_chunk(wl, 11, 0, N + rnd * B, B)
        cache.append(0, *(PU.bits_to_bf16_tensor(nxt[x], dev) for x in ("q_bits", "k_bits", "v_bits")))
        state_k[:, :, K:] = nxt["k_bits"].transpose(1, 2, 0, 3)
        state_v[:, :, K:] = nxt["v_bits"].transpose(1, 2, 0, 3)
        pos[:, :, K:] = np.arange(N + rnd * B, N + (rnd + 1) * B)
        qhist.extend(nxt["q_bits"][t] for t in range(B))
    assert compared >= 1


# ----------------------------------------------------------------------------- sampling law on the GPU path

def _inclusion(w, m):
    n = len(w)
    pi = np.zeros(n)
    for seq in itertools.permutations(range(n), m):
        p, rest = 1.0, float(np.sum(w))
        for i in seq:
            p *= w[i] / rest
            rest -= w[i]
        for i in seq:
            pi[i] += p
    return pi


def test_gpu_keep_frequencies_match_successive_sampling():
    """64 sequences with identical content draw independent noise; 64 rounds give 4096 samples."""
    from paper_2606_03928_gb300.vase import VaseCache, Geometry
    K, B, nv, Wn = 7, 2, 1, 2
    N = K + B
    cache = VaseCache(Geometry(K, B, Wn, 1, 1, 1, 64), n_v=nv, pool_kernel=1, debug_outputs=True, seed=123)
    rng = np.random.default_rng(8)
    q = W.f32_to_bf16_bits(rng.standard_normal((Wn, 128)) * 0.15)
    k = W.f32_to_bf16_bits(rng.standard_normal((N, 128)) * 1.0)
    v = W.f32_to_bf16_bits(rng.standard_normal((N, 128)))
    pos = np.arange(N)
    ref = O.evict_unit_bits(q, k, v, pos, budget_k=K, buffer_b=B, n_v=nv, pool_kernel=1)
    rv = set(ref["reserved_v"].tolist())
    cand = [i for i in range(K) if i not in rv]
    m = K - nv - B
    pi = _inclusion(ref["pooled"][cand], m)
    dev = cache.device
    kt = PU.bits_to_bf16_tensor(np.broadcast_to(k, (64, 1, N, 128)).copy(), dev)
    vt = PU.bits_to_bf16_tensor(np.broadcast_to(v, (64, 1, N, 128)).copy(), dev)
    qt = PU.bits_to_bf16_tensor(np.broadcast_to(q, (64, 1, Wn, 128)).copy(), dev)
    pt = torch.from_numpy(np.broadcast_to(pos, (64, 1, N)).astype(np.int32).copy()).to(dev)
    counts = np.zeros(N)
    R = 64
    for t in range(R):
        cache.k_cache[0].copy_(kt)
        cache.v_cache[0].copy_(vt)
        cache.q_window[0].copy_(qt)
        cache.positions[0].copy_(pt)
        cache.set_layer_state(0, N, t, N, 10 ** 6)
        cache.refresh_value_scores(0)
        cache.evict(0)
        src = cache.debug_view()["src"].cpu().numpy()
        for u in range(64):
            counts[src[u]] += 1
    assert cache.check_device_error()[0] == 0
    S = 64 * R
    freq = counts[cand] / S
    sigma = np.sqrt(pi * (1 - pi) / S)
    assert np.all(np.abs(freq - pi) <= 4.5 * sigma + 1e-9), (freq, pi)
    assert np.all(counts[list(rv)] == S) and np.all(counts[K:] == S)
    w = ref["pooled"][cand]
    assert np.all(freq >= 1 - (1 - w / w.sum()) ** m - 4.5 * sigma)


# ----------------------------------------------------------------------------- full-size configurations

def test_qwen3_1p7b_k2048_full_layer_in_bench_launch_configuration():
    """All 64 units of one layer at full size, with the bench's launch configuration (no debug outputs)."""
    wl = W.WORKLOADS["qwen3_1p7b_k2048"]
    _run_layer(wl, layer=27, num_layers=28, round_index=40, debug=False)


def test_qwen3_8b_k4096_attnv_sampled_units():
    wl = W.WORKLOADS["qwen3_8b_k4096"]
    units = [(0, 0), (5, 3), (17, 7), (31, 6)]
    _run_layer(wl, layer=35, num_layers=36, round_index=90, units=units, debug=False)


def test_qwen3_8b_k4096_dkv_sampled_units():
    wl = W.WORKLOADS["qwen3_8b_k4096"]
    units = [(0, 0), (9, 2), (31, 7)]
    _run_layer(wl, variant="dkv", layer=2, num_layers=4, round_index=77, units=units, debug=False)


@pytest.mark.parametrize("K,B,b,rate,units", [
    (16384, 512, 1, 0.005, [(0, 0), (0, 5)]),             # the sweep's largest unit: N = 16896, unstaged selection
    (1024, 32, 128, 0.02, [(0, 0), (77, 3), (127, 7)]),   # smallest budget and buffer, largest batch, most outliers
    (2048, 128, 8, 0.0, [(0, 2), (7, 7)]),                 # no value outliers: the reservation takes ordinary rows
])
def test_qwen3_8b_sweep_points_sampled_units(K, B, b, rate, units):
    """Points of the Qwen3-8B-geometry sweep (32/8 heads, W = 32) at its extremes, sampled units against the oracle."""
    wl = W.sweep_point(K, B, b, rate)
    _run_layer(wl, layer=0, num_layers=1, round_index=5, units=units, debug=False)


def test_qwen3_32b_k8192_sampled_units():
    wl = W.WORKLOADS["qwen3_32b_k8192"]
    units = [(0, 0), (7, 5), (15, 7)]
    _run_layer(wl, layer=1, num_layers=2, round_index=95, units=units, debug=True)


# ----------------------------------------------------------------------------- batched layers

def test_evict_all_equals_per_layer_evictions_and_matches_oracle():
    """vase_evict_all covers every full layer in one launch per kernel; results equal per-layer calls."""
    wl = W.shrink(SMALL, budget_k=192, buffer_b=64, window=16, batch=2, num_layers=3)
    a = _cache(wl, 3)
    b = _cache(wl, 3)
    states = [W.layer_state(wl, 4, layer, 2 + layer, "gapped") for layer in range(3)]
    for layer, st in enumerate(states):
        PU.upload_layer(a, layer, st, 2 + layer)
        PU.upload_layer(b, layer, st, 2 + layer)
    for layer in range(3):
        a.evict(layer)
    assert b.evict_all() == 3
    torch.cuda.synchronize()
    assert torch.equal(a.k_cache, b.k_cache) and torch.equal(a.v_cache, b.v_cache)
    assert torch.equal(a.positions, b.positions)
    assert b.check_device_error()[0] == 0
    for z in range(3):
        dv = {k: (v.cpu().numpy() if k != "layer" else v) for k, v in b.debug_view(z).items()}
        layer = dv["layer"]
        assert layer == z
        st = states[layer]
        got = PU.download(b, layer)
        got.update({k: v for k, v in dv.items() if k != "layer"})
        for s in range(wl.batch):
            for h in range(wl.num_kv_heads):
                ref = PU.oracle_unit(wl, st, s, h, variant="attnv", round_index=2 + layer, seed=0, layer=layer)
                PU.check_unit(wl, ref, PU.unit_slice(got, s, h, wl.num_kv_heads), st["k_bits"][s, h],
                              st["v_bits"][s, h], st["positions"][s, h], variant="attnv", n_v=wl.budget_k // 4)
        assert b.layer_state(layer)["round"] == 3 + layer


def test_append_all_equals_per_layer_appends():
    wl = W.shrink(SMALL, budget_k=64, buffer_b=16, window=8, batch=2, num_layers=3)
    a = _cache(wl, 3)
    b = _cache(wl, 3)
    dev = a.device
    chunks = [W.stream_chunk(wl, 9, layer, 0, 40) for layer in range(3)]
    qs = [PU.bits_to_bf16_tensor(c["q_bits"], dev) for c in chunks]
    ks = [PU.bits_to_bf16_tensor(c["k_bits"], dev) for c in chunks]
    vs = [PU.bits_to_bf16_tensor(c["v_bits"], dev) for c in chunks]
    for layer in range(3):
        a.append(layer, qs[layer], ks[layer], vs[layer])
    b.append_all(torch.stack(qs), torch.stack(ks), torch.stack(vs))
    torch.cuda.synchronize()
    # only the first 40 slots were written (the rest of both caches is uninitialised memory)
    assert torch.equal(a.k_cache[:, :, :, :40], b.k_cache[:, :, :, :40])
    assert torch.equal(a.v_cache[:, :, :, :40], b.v_cache[:, :, :, :40])
    assert torch.equal(a.q_window, b.q_window) and torch.equal(a.positions, b.positions)
    for layer in range(3):
        assert a.layer_state(layer) == b.layer_state(layer)


def test_append_all_strided_from_one_staging_block_equals_packed_append_all():
    """vase_append_all_strided over a staging buffer that holds, per layer, only [last W query rows | k | v]
    (q pointers W rows before each tail, one block between layers) writes exactly what vase_append_all writes
    from packed [L][n] inputs: the rows before each layer's query tail belong to the previous block and are
    never read."""
    from paper_2606_03928_gb300 import vase as V
    L, n = 3, 40
    wl = W.shrink(SMALL, budget_k=64, buffer_b=16, window=8, batch=2, num_layers=L)
    a, b = _cache(wl, L), _cache(wl, L)
    dev = a.device
    chunks = [W.stream_chunk(wl, 9, layer, 0, n) for layer in range(L)]
    qs = [PU.bits_to_bf16_tensor(c["q_bits"], dev) for c in chunks]
    ks = [PU.bits_to_bf16_tensor(c["k_bits"], dev) for c in chunks]
    vs = [PU.bits_to_bf16_tensor(c["v_bits"], dev) for c in chunks]
    a.append_all(torch.stack(qs), torch.stack(ks), torch.stack(vs))
    Wq = wl.window
    q_row = qs[0][0].numel()
    kv_el = ks[0].numel()
    pad = (n - Wq) * q_row
    blk = Wq * q_row + 2 * kv_el
    flat = torch.full((pad + L * blk,), float("nan"), dtype=torch.bfloat16, device=dev)
    for layer in range(L):
        o = pad + layer * blk
        flat[o:o + Wq * q_row] = qs[layer][n - Wq:].reshape(-1)
        flat[o + Wq * q_row:o + Wq * q_row + kv_el] = ks[layer].reshape(-1)
        flat[o + Wq * q_row + kv_el:o + blk] = vs[layer].reshape(-1)
    base = flat.data_ptr()
    with pytest.raises(V.VaseError):  # a stride that is not a multiple of 16 bytes: nothing is written
        V.vase_append_all_strided(b.ctx, base, base + 2 * (pad + Wq * q_row), base + 2 * (pad + Wq * q_row + kv_el),
                                  n, 2 * blk + 2, 2 * blk)
    V.vase_append_all_strided(b.ctx, base, base + 2 * (pad + Wq * q_row), base + 2 * (pad + Wq * q_row + kv_el),
                              n, 2 * blk, 2 * blk)
    torch.cuda.synchronize()
    assert torch.equal(a.k_cache[:, :, :, :n], b.k_cache[:, :, :, :n])
    assert torch.equal(a.v_cache[:, :, :, :n], b.v_cache[:, :, :, :n])
    assert torch.equal(a.q_window, b.q_window) and torch.equal(a.positions, b.positions)
    assert torch.equal(a.value_scores[..., :n], b.value_scores[..., :n])
    for layer in range(L):
        assert a.layer_state(layer) == b.layer_state(layer)


# ----------------------------------------------------------------------------- interleaved (persistent) schedule

@pytest.mark.parametrize("K,B,Wn,Hq,Hkv", [(192, 64, 16, 16, 8), (200, 40, 16, 16, 8), (256, 64, 32, 32, 8),
                                          (160, 96, 32, 64, 8), (160, 64, 64, 64, 8)])
def test_evict_all_with_several_units_per_cta_matches_oracle(K, B, Wn, Hq, Hkv):
    """Eight layers of 64 units: more than two items per SM, so one CTA per SM takes a strided list of units and
    interleaves the pass-B sweep of each with the pass-A sweep of the next.  Every unit of every layer is checked."""
    wl = W.shrink(SMALL, budget_k=K, buffer_b=B, window=Wn, num_q_heads=Hq, num_kv_heads=Hkv, batch=64 // Hkv,
                  num_layers=8)
    cache = _cache(wl, 8)
    states = [W.layer_state(wl, 11, layer, 3 + layer, "gapped") for layer in range(8)]
    for layer, st in enumerate(states):
        PU.upload_layer(cache, layer, st, 3 + layer)
    assert cache.evict_all() == 8
    status, code = cache.check_device_error()
    assert status == 0, f"device error word {code:#x}"
    for z in range(8):
        dv = {k: (v.cpu().numpy() if k != "layer" else v) for k, v in cache.debug_view(z).items()}
        layer = dv["layer"]
        st = states[layer]
        got = PU.download(cache, layer)
        got.update({k: v for k, v in dv.items() if k != "layer"})
        for s in range(wl.batch):
            for h in range(wl.num_kv_heads):
                ref = PU.oracle_unit(wl, st, s, h, variant="attnv", round_index=3 + layer, seed=0, layer=layer)
                PU.check_unit(wl, ref, PU.unit_slice(got, s, h, wl.num_kv_heads), st["k_bits"][s, h],
                              st["v_bits"][s, h], st["positions"][s, h], variant="attnv", n_v=wl.budget_k // 4)


def test_sixteen_layers_of_512_window_rows_match_oracle():
    """G*W = 512 window rows (the Qwen3-32B group and window) on sixteen layers in one batched launch, one CTA
    per unit whose four consumer groups each score one 128-row block in both passes: every layer's workspace
    slot, kept set and compacted rows are checked on sampled units, and every layer's counters advance."""
    wl = W.shrink(W.WORKLOADS["qwen3_32b_k8192"], budget_k=192, buffer_b=64, batch=2, num_layers=16)
    L = wl.num_layers
    cache = _cache(wl, L)
    states = [W.layer_state(wl, 17, layer, 5 + layer, "gapped") for layer in range(L)]
    for layer, st in enumerate(states):
        PU.upload_layer(cache, layer, st, 5 + layer)
    assert cache.evict_all() == L
    status, code = cache.check_device_error()
    assert status == 0, f"device error word {code:#x}"
    seen = set()
    for z in range(L):
        dv = {k: (v.cpu().numpy() if k != "layer" else v) for k, v in cache.debug_view(z).items()}
        layer = dv["layer"]
        seen.add(layer)
        st = states[layer]
        got = PU.download(cache, layer)
        got.update({k: v for k, v in dv.items() if k != "layer"})
        for (s_, h) in ((0, 0), (1, 7), (z % 2, z % 8)):
            ref = PU.oracle_unit(wl, st, s_, h, variant="attnv", round_index=5 + layer, seed=0, layer=layer)
            PU.check_unit(wl, ref, PU.unit_slice(got, s_, h, wl.num_kv_heads), st["k_bits"][s_, h],
                          st["v_bits"][s_, h], st["positions"][s_, h], variant="attnv", n_v=wl.budget_k // 4)
        assert cache.layer_state(layer)["fill"] == wl.budget_k and cache.layer_state(layer)["round"] == 6 + layer
    assert seen == set(range(L))


def test_qwen3_1p7b_k2048_all_layers_in_one_launch():
    """The bench's launch: all 28 layers of the 1.7B geometry in one launch per kernel, no debug outputs.
    Three layers are checked unit by unit against the oracle; every unit of every layer keeps K distinct slots
    including the buffer."""
    wl = W.WORKLOADS["qwen3_1p7b_k2048"]
    L = wl.num_layers
    cache = _cache(wl, L, debug=False)
    base = [W.layer_state(wl, 21, i, 40 + i, "gapped") for i in range(3)]
    for layer in range(L):
        PU.upload_layer(cache, layer, base[layer % 3], 40 + layer)
    assert cache.evict_all() == L
    status, code = cache.check_device_error()
    assert status == 0, f"device error word {code:#x}"
    K, B = wl.budget_k, wl.buffer_b
    for layer in range(L):
        pos = cache.positions[layer].cpu().numpy()
        st = base[layer % 3]
        for s in range(wl.batch):
            for h in range(wl.num_kv_heads):
                kept = pos[s, h, :K]
                assert len(set(kept.tolist())) == K
                assert set(st["positions"][s, h, K:K + B].tolist()) <= set(kept.tolist())
    for layer in (0, 13, L - 1):
        st = base[layer % 3]
        got = PU.download(cache, layer)
        for s in range(wl.batch):
            for h in range(wl.num_kv_heads):
                ref = PU.oracle_unit(wl, st, s, h, variant="attnv", round_index=40 + layer, seed=0, layer=layer)
                gu = {"k_bits": got["k_bits"][s, h], "v_bits": got["v_bits"][s, h],
                      "positions": got["positions"][s, h], "vmag": got["vmag"][s, h]}
                # the kept list is the compacted positions mapped back to slots of the uploaded state
                slot_of = {int(p_): i for i, p_ in enumerate(st["positions"][s, h])}
                gu["src"] = np.array([slot_of[int(p_)] for p_ in gu["positions"][:K]], dtype=np.int64)
                gu["attn"] = gu["pooled"] = gu["key"] = gu["value_score"] = None
                PU.check_unit(wl, ref, gu, st["k_bits"][s, h], st["v_bits"][s, h], st["positions"][s, h],
                              variant="attnv", n_v=wl.budget_k // 4, check_scores=False)


def _unit_state_from_stream(wl, ch, t0, t1, s, h):
    """[t0, t1) of a host stream chunk as one unit's rows: keys and values [n, d], and the query rows of its G
    heads over the last W steps of the range, head-major [G*W, d]."""
    G, Wn = wl.group, wl.window
    q = ch["q_bits"][t1 - Wn:t1, s, h * G:(h + 1) * G]            # [W, G, d]
    return (ch["k_bits"][t0:t1, s, h], ch["v_bits"][t0:t1, s, h],
            np.ascontiguousarray(q.transpose(1, 0, 2)).reshape(G * Wn, wl.head_dim))


def test_qwen3_1p7b_k2048_appended_stream_two_rounds_in_the_bench_launch():
    """The bench's launch (all 28 layers per kernel launch, debug outputs on), driven as the bench drives it:
    every layer's stream enters through the library's append (K + B tokens each, then B more for every layer in
    one vase_append_all_strided launch from [last W query rows | k | v] blocks), and every layer is evicted twice.
    The value magnitudes the appends computed are compared with the oracle's for every unit of three layers; after
    each eviction, sampled units of those layers are compared with the oracle on the chained state (window
    scores, pooled scores, keys, kept sets, compacted rows), the second round on the oracle's own compaction of
    the first.  Layer l runs host stream l % 2."""
    from paper_2606_03928_gb300 import vase as V
    wl = W.WORKLOADS["qwen3_1p7b_k2048"]
    L, K, B, N, Wn, G = wl.num_layers, wl.budget_k, wl.buffer_b, wl.slots, wl.window, wl.group
    b, Hq, Hkv, d = wl.batch, wl.num_q_heads, wl.num_kv_heads, wl.head_dim
    cache = _cache(wl, L, debug=True)
    dev = cache.device
    streams = [W.stream_chunk(wl, 23, i, 0, N + B) for i in range(2)]
    dstreams = [{x: PU.bits_to_bf16_tensor(c[x], dev) for x in ("q_bits", "k_bits", "v_bits")} for c in streams]
    for layer in range(L):  # the first K + B tokens of each layer, appended through the library
        ds = dstreams[layer % 2]
        cache.append(layer, ds["q_bits"][:N], ds["k_bits"][:N], ds["v_bits"][:N])
    layers, units = (0, 13, L - 1), [(0, 0), (3, 5), (b - 1, Hkv - 1)]
    torch.cuda.synchronize()
    for layer in layers:  # magnitudes computed by the append kernel, every unit
        ch = streams[layer % 2]
        vref = O.value_magnitude(O.bf16_bits_to_f64(ch["v_bits"][:N].transpose(1, 2, 0, 3)).reshape(-1, d))
        PU.assert_close_scores(cache.value_scores[layer].cpu().numpy().reshape(-1), vref, "append magnitudes")
    # round 0
    assert cache.evict_all() == L
    assert cache.check_device_error()[0] == 0
    chained = {}
    z_of = {}
    for z in range(L):
        z_of[cache.debug_view(z)["layer"]] = z
    for layer in layers:
        ch = streams[layer % 2]
        dv = {k: (v.cpu().numpy() if k != "layer" else v) for k, v in cache.debug_view(z_of[layer]).items()}
        got = PU.download(cache, layer)
        got.update({k: v for k, v in dv.items() if k != "layer"})
        for (s_, h) in units:
            k0, v0, q0 = _unit_state_from_stream(wl, ch, 0, N, s_, h)
            pos0 = np.arange(N)
            ref = O.evict_unit_bits(q0, k0, v0, pos0, budget_k=K, buffer_b=B, seed=0, layer=layer, seq=s_, head=h,
                                    num_kv_heads=Hkv, rnd=0, group=G)
            gu = PU.unit_slice(got, s_, h, Hkv)
            PU.check_unit(wl, ref, gu, k0, v0, pos0, variant="attnv", n_v=K // 4)
            if np.array_equal(gu["src"], ref["src"]):  # chain only from a state both sides agree on
                chained[(layer, s_, h)] = ref
    # round 1: B new tokens for every layer in one strided launch from per-layer [W query rows | k | v] blocks
    qtail = [dstreams[i]["q_bits"][N + B - Wn:N + B] for i in range(2)]
    blk = Wn * b * Hq * d + 2 * B * b * Hkv * d
    flat = torch.empty((L * blk,), dtype=torch.bfloat16, device=dev)
    for layer in range(L):
        ds, o = dstreams[layer % 2], layer * blk
        flat[o:o + Wn * b * Hq * d] = qtail[layer % 2].reshape(-1)
        flat[o + Wn * b * Hq * d:o + Wn * b * Hq * d + B * b * Hkv * d] = ds["k_bits"][N:N + B].reshape(-1)
        flat[o + Wn * b * Hq * d + B * b * Hkv * d:o + blk] = ds["v_bits"][N:N + B].reshape(-1)
    base = flat.data_ptr()
    q_ptr = base - (B - Wn) * b * Hq * d * 2  # the append reads only the last W query rows of each layer
    k_ptr = base + Wn * b * Hq * d * 2
    v_ptr = k_ptr + B * b * Hkv * d * 2
    assert V.vase_append_all_strided(cache.ctx, q_ptr, k_ptr, v_ptr, B, blk * 2, blk * 2) == V.VASE_EVICT_DUE
    torch.cuda.synchronize()
    for layer in layers:  # the appended slots' magnitudes, every unit
        ch = streams[layer % 2]
        vref = O.value_magnitude(O.bf16_bits_to_f64(ch["v_bits"][N:N + B].transpose(1, 2, 0, 3)).reshape(-1, d))
        PU.assert_close_scores(cache.value_scores[layer][..., K:].cpu().numpy().reshape(-1), vref,
                               "append magnitudes, second round")
    assert cache.evict_all() == L
    assert cache.check_device_error()[0] == 0
    for z in range(L):
        z_of[cache.debug_view(z)["layer"]] = z
    compared = 0
    for layer in layers:
        ch = streams[layer % 2]
        dv = {k: (v.cpu().numpy() if k != "layer" else v) for k, v in cache.debug_view(z_of[layer]).items()}
        got = PU.download(cache, layer)
        got.update({k: v for k, v in dv.items() if k != "layer"})
        for (s_, h) in units:
            prev = chained.get((layer, s_, h))
            if prev is None:
                continue
            k1 = np.concatenate([prev["k_bits_new"], ch["k_bits"][N:N + B, s_, h]])
            v1 = np.concatenate([prev["v_bits_new"], ch["v_bits"][N:N + B, s_, h]])
            pos1 = np.concatenate([prev["positions_new"], np.arange(N, N + B)])
            _, _, q1 = _unit_state_from_stream(wl, ch, N, N + B, s_, h)
            ref = O.evict_unit_bits(q1, k1, v1, pos1, budget_k=K, buffer_b=B, seed=0, layer=layer, seq=s_, head=h,
                                    num_kv_heads=Hkv, rnd=1, group=G)
            PU.check_unit(wl, ref, PU.unit_slice(got, s_, h, Hkv), k1, v1, pos1, variant="attnv", n_v=K // 4)
            compared += 1
    assert compared >= len(layers) * len(units) - 2  # a first-round threshold tie may end a unit's chain


# ----------------------------------------------------------------------------- variants: GQA max-aggregation, shared-G DKV, random reservation

def _reserved_slots(key_row, K):
    """R_V of a unit from the debug keys: the candidates' keys are >= 0, the reserved slots carry -1."""
    return np.flatnonzero(np.asarray(key_row[:K]) < 0)


@pytest.mark.parametrize("stochastic", [True, False])
def test_random_reservation_matches_oracle_exactly(stochastic):
    kw = {"reserve": "random", "stochastic": stochastic}
    cache, st, got, _ = _run_layer(SMALL, cache_kw=kw, oracle_kw=kw)
    K = SMALL.budget_k
    for s in range(SMALL.batch):
        for h in range(SMALL.num_kv_heads):
            ref = PU.oracle_unit(SMALL, st, s, h, variant="attnv", round_index=3, seed=0, layer=1, **kw)
            gu = PU.unit_slice(got, s, h, SMALL.num_kv_heads)
            # an integer decision on the same 23-bit uniforms on both sides: identical reserved sets
            assert np.array_equal(_reserved_slots(gu["key"], K), ref["reserved_v"])


def test_random_reservation_differs_from_value_reservation():
    a = _run_layer(SMALL)[2]["key"]
    b = _run_layer(SMALL, cache_kw={"reserve": "random"}, oracle_kw={"reserve": "random"})[2]["key"]
    assert not np.array_equal(a < 0, b < 0)


# (K, B, W, Hq, Hkv): heads of 16 rows four to a 64-column chunk; 12-row heads that straddle chunks and a
# padded tail; G*W = 512 in four 128-row blocks (parts combined by max); G*W = 512 with 256-row heads, two
# 256-row blocks; one query head per KV head
@pytest.mark.parametrize("K,B,Wn,Hq,Hkv", [(256, 64, 16, 32, 8), (200, 40, 12, 24, 8), (256, 64, 64, 32, 4),
                                          (512, 128, 256, 16, 8), (192, 64, 32, 8, 8)])
def test_gqa_max_aggregation_matches_oracle(K, B, Wn, Hq, Hkv):
    wl = W.shrink(SMALL, budget_k=K, buffer_b=B, window=Wn, num_q_heads=Hq, num_kv_heads=Hkv, batch=2,
                  num_layers=2)
    _run_layer(wl, cache_kw={"gqa": "max"}, oracle_kw={"gqa": "max"})


def test_gqa_max_in_the_persistent_schedule():
    """Eight layers of 64 units (one CTA per SM takes a strided list of units), max over the query heads."""
    wl = W.shrink(SMALL, budget_k=192, buffer_b=64, window=16, num_q_heads=32, num_kv_heads=8, batch=8,
                  num_layers=8)
    cache = _cache(wl, 8, gqa="max")
    states = [W.layer_state(wl, 12, layer, 2 + layer, "gapped") for layer in range(8)]
    for layer, st in enumerate(states):
        PU.upload_layer(cache, layer, st, 2 + layer)
    assert cache.evict_all() == 8
    status, code = cache.check_device_error()
    assert status == 0, f"device error word {code:#x}"
    for z in range(8):
        dv = {k: (v.cpu().numpy() if k != "layer" else v) for k, v in cache.debug_view(z).items()}
        layer = dv["layer"]
        st = states[layer]
        got = PU.download(cache, layer)
        got.update({k: v for k, v in dv.items() if k != "layer"})
        for s in range(wl.batch):
            for h in range(wl.num_kv_heads):
                ref = PU.oracle_unit(wl, st, s, h, variant="attnv", round_index=2 + layer, seed=0, layer=layer,
                                     gqa="max")
                PU.check_unit(wl, ref, PU.unit_slice(got, s, h, wl.num_kv_heads), st["k_bits"][s, h],
                              st["v_bits"][s, h], st["positions"][s, h], variant="attnv", n_v=wl.budget_k // 4)


def test_gqa_max_rejects_windows_that_split_a_row_block():
    from paper_2606_03928_gb300.vase import VaseError
    wl = W.shrink(SMALL, budget_k=256, buffer_b=64, window=48, num_q_heads=64, num_kv_heads=8, batch=1,
                  num_layers=1)   # G*W = 384 > 256 and 48 does not divide 256
    with pytest.raises(VaseError):
        _cache(wl, 1, gqa="max")
    wl2 = W.shrink(SMALL, budget_k=256, buffer_b=64, window=6, num_q_heads=16, num_kv_heads=8, batch=1,
                   num_layers=1)  # W % 4 != 0
    with pytest.raises(VaseError):
        _cache(wl2, 1, gqa="max")


def test_dkv_shared_g_matches_oracle_and_is_shared():
    kw = {"dkv_shared_g": True}
    _run_layer(SMALL, variant="dkv", cache_kw=kw, oracle_kw=kw)
    # one projection for every unit of a round: two units holding identical rows score identically
    wl = W.shrink(SMALL, batch=2, num_layers=1)
    cache = _cache(wl, 1, variant="dkv", dkv_shared_g=True)
    st = W.layer_state(wl, 3, 0, 0, "gapped")
    for key in ("q_bits", "k_bits", "v_bits", "positions"):
        st[key][1] = st[key][0]
    PU.upload_layer(cache, 0, st, 0)
    assert cache.evict(0) == 0
    scores = cache.debug_view(0)["value_score"].cpu().numpy().reshape(wl.batch, wl.num_kv_heads, -1)
    assert np.array_equal(scores[0], scores[1])
    cache2 = _cache(wl, 1, variant="dkv")
    PU.upload_layer(cache2, 0, st, 0)
    assert cache2.evict(0) == 0
    scores2 = cache2.debug_view(0)["value_score"].cpu().numpy().reshape(wl.batch, wl.num_kv_heads, -1)
    assert not np.array_equal(scores2[0], scores2[1])


# ----------------------------------------------------------------------------- maximum sizes and degenerate cases

def _lift_keys(wl, st, units, alphas=(4.0, 5.0, 8.0)):
    """Plants key rows far above the rest of a window row's logits: key = alpha * q_r for one window query r
    of the unit, so that q_r . k / sqrt(d) in log2 units sits about 60 (alpha 4), 80 (5) and 130 (8) above
    the other keys of that row.  They sit in later tiles than the first, among the candidates."""
    N, G, Wn = wl.slots, wl.group, wl.window
    for n, (s, h) in enumerate(units):
        for i, a in enumerate(alphas):
            r = (n * 7 + i * 5) % (G * Wn)
            g, w = divmod(r, Wn)
            q = O.bf16_bits_to_f64(st["q_bits"][s, h * G + g, w])
            j = 130 + (70 + i * 397 + n * 131) % (wl.budget_k - 130)  # past the first 128-token tile
            st["k_bits"][s, h, j] = W.f32_to_bf16_bits(a * q)


# The window score sums each row's exponentials against the maximum of the row's first chunk and raises that
# reference only for a chunk whose sum against it passes 2^64.  Keys planted far above the first chunk make some
# rows take that path (sums of about 2^60, 2^80 and an overflow to inf); every score, kept set and moved row still
# follows the oracle.  Geometries: the persistent schedule with replicated 64-row windows, cluster mode with 128
# rows, and 512 window rows (two 256-column pass-B accumulators).
@pytest.mark.parametrize("K,B,Wn,Hq,Hkv,batch", [(256, 64, 32, 16, 8, 20), (1024, 128, 32, 32, 8, 2),
                                                 (1024, 256, 64, 64, 8, 1)])
def test_window_score_with_keys_far_above_the_first_chunk(K, B, Wn, Hq, Hkv, batch):
    wl = W.shrink(SMALL, budget_k=K, buffer_b=B, window=Wn, num_q_heads=Hq, num_kv_heads=Hkv, batch=batch,
                  num_layers=2)
    units = [(0, 0), (0, Hkv - 1), (batch - 1, 3)]
    _, _, _, flips = _run_layer(wl, units=units, edit=lambda st: _lift_keys(wl, st, units))
    assert flips <= 2

def test_largest_supported_unit_matches_oracle():
    """K = 16384, B = 256 (N = 16640, inputs read unstaged by the single-CTA selection), one unit, the score
    kernel in cluster mode; every slot checked against the oracle (the sweep test samples N = 16896)."""
    wl = W.shrink(SMALL, budget_k=16384, buffer_b=256, window=16, num_q_heads=4, num_kv_heads=1, batch=1,
                  num_layers=1)
    _run_layer(wl, layer=0, num_layers=1, round_index=4)


def test_budget_equal_to_buffer_keeps_only_the_buffer():
    """K == B (so N_v = 0 and m = 0): every candidate is evicted and the B newest pairs move down."""
    wl = W.shrink(SMALL, budget_k=96, buffer_b=96, window=8, batch=2, num_layers=1)
    cache, st, got, _ = _run_layer(wl, layer=0, num_layers=1, cache_kw={"n_v": 0}, oracle_kw={"n_v": 0})
    for u in range(wl.batch * wl.num_kv_heads):
        assert np.array_equal(got["src"][u], np.arange(96, 192))


def test_value_reservation_filling_every_kept_candidate():
    """N_v = K - B: R_V takes every kept candidate (m = 0), so the kept set is R_V plus the buffer."""
    K, B = 160, 32
    wl = W.shrink(SMALL, budget_k=K, buffer_b=B, window=8, batch=2, num_layers=1)
    _run_layer(wl, layer=0, num_layers=1, cache_kw={"n_v": K - B}, oracle_kw={"n_v": K - B})


def test_append_reads_only_the_last_window_query_rows():
    """vase_append's contract: query rows before the last min(W, n) are never read (NaN there changes nothing)."""
    wl = W.shrink(SMALL, budget_k=128, buffer_b=64, window=8, batch=2, num_layers=1)
    gen = torch.Generator(device="cuda")
    gen.manual_seed(71)
    n = 40
    q = torch.randn((n, wl.batch, wl.num_q_heads, wl.head_dim), generator=gen, device="cuda").to(torch.bfloat16)
    k = torch.randn((n, wl.batch, wl.num_kv_heads, wl.head_dim), generator=gen, device="cuda").to(torch.bfloat16)
    v = torch.randn((n, wl.batch, wl.num_kv_heads, wl.head_dim), generator=gen, device="cuda").to(torch.bfloat16)
    q_nan = q.clone()
    q_nan[:n - wl.window] = float("nan")
    a, b = _cache(wl, 1, debug=False), _cache(wl, 1, debug=False)
    a.append(0, q, k, v)
    b.append(0, q_nan, k, v)
    torch.cuda.synchronize()
    assert torch.equal(a.q_window, b.q_window)  # the ring is full (n >= W)
    # slots past the fill hold whatever the allocation held: compare the n written ones
    assert torch.equal(a.k_cache[..., :n, :], b.k_cache[..., :n, :])
    assert torch.equal(a.v_cache[..., :n, :], b.v_cache[..., :n, :])
    assert torch.equal(a.positions[..., :n], b.positions[..., :n])


# ----------------------------------------------------------------------------- failure detection

def test_bounded_wait_runs_out_and_the_host_reads_its_site():
    """A kernel whose mbarrier wait nothing completes: the wait gives up at its limit (about two seconds), the
    site lands in the device error word, the host reads and clears it, and the same context then evicts a
    layer that matches the oracle (no fault, nothing left stuck)."""
    from paper_2606_03928_gb300 import vase as V
    cache = _cache(SMALL, 2)
    V.vase_self_test_wait_timeout(cache.ctx)
    status, code = cache.check_device_error()
    assert status == V.VASE_ERR_DEVICE
    assert code & 0x80000000 and (code & 0xFFFF) == V.VASE_SITE_SELF_TEST
    assert cache.check_device_error() == (0, 0)  # read and cleared
    _run_layer(SMALL, cache=cache)


# Ties in the selection go to the lower slot: R_V over equal value magnitudes, the sampled set (noise off) over
# equal keys.  Value rows are drawn from three distinct rows and three quarters of the key rows are one row, so
# both thresholds fall inside runs of bit-identical scores.  The kept set must be exactly the rule applied to the
# GPU's own scores (its debug outputs): on the fused small-unit kernel (rank count), the selection kernel's rank
# count (K = 256) and its radix select (K = 1024).
@pytest.mark.parametrize("K,B,batch", [(256, 64, 2), (256, 64, 24), (1024, 64, 24)])
def test_selection_ties_go_to_the_lower_slot(K, B, batch):
    wl = W.shrink(SMALL, budget_k=K, buffer_b=B, window=16, num_q_heads=16, num_kv_heads=8, batch=batch,
                  num_layers=1)
    N = K + B
    st = W.layer_state(wl, 3, 0, 0, "dense")
    rng = np.random.default_rng(11)
    for s in range(batch):
        for h in range(wl.num_kv_heads):
            rows = st["v_bits"][s, h, rng.integers(0, N, size=3)].copy()
            st["v_bits"][s, h] = rows[rng.integers(0, 3, size=N)]
            st["k_bits"][s, h, : 3 * N // 4] = st["k_bits"][s, h, 0]
    cache = _cache(wl, 1, stochastic=False)
    PU.upload_layer(cache, 0, st, 0)
    assert cache.evict(0) == 0
    status, code = cache.check_device_error()
    assert status == 0, f"device error word {code:#x}"
    got = PU.download(cache, 0)
    n_v = K // 4
    m = K - n_v - B
    tied_v = tied_k = 0
    for u in range(batch * wl.num_kv_heads):
        vm = np.asarray(got["value_score"][u][:K], dtype=np.float32)  # the magnitudes the kernel ranked
        order = sorted(range(K), key=lambda i: (-vm[i], i))
        r_v = set(order[:n_v])
        key = np.asarray(got["key"][u][:K], dtype=np.float32)
        cand = [i for i in range(K) if i not in r_v]
        korder = sorted(cand, key=lambda i: (-key[i], i))
        kept = sorted(r_v | set(korder[:m]) | set(range(K, N)))
        assert got["src"][u].tolist() == kept, f"unit {u}: kept set differs from the lower-slot tie rule"
        tied_v += int(np.sum(vm == vm[order[n_v - 1]]) > 1)
        tied_k += int(np.sum(key[cand] == key[korder[m - 1]]) > 1)
    assert tied_v > 0 and tied_k > 0, (tied_v, tied_k)


# ----------------------------------------------------------------------------- the fused step (append + eviction)

# vase_append_evict_all is vase_append_all_strided then vase_evict_all: bit-identical caches, positions, value
# magnitudes, window rings and layer states over chained steps, in one launch per step where every unit of every
# layer fits one wave of the fused kernel, and as the two calls where it does not (384 units).
@pytest.mark.parametrize("L,K,B,Wn,Hq,Hkv,batch,kw,fused", [
    (1, 256, 64, 32, 16, 8, 1, {}, True),                     # the single-layer geometry
    (2, 200, 40, 16, 32, 8, 2, {"gqa": "max"}, True),         # G = 4, a ragged last tile, GQA max
    (2, 256, 64, 16, 16, 8, 2, {"reserve": "random"}, True),  # random reservation (keys from positions)
    (3, 192, 64, 16, 16, 8, 16, {}, False),                   # 384 units: the two calls
])
def test_append_evict_all_equals_append_all_then_evict_all(L, K, B, Wn, Hq, Hkv, batch, kw, fused):
    from paper_2606_03928_gb300 import vase as V
    wl = W.shrink(SMALL, budget_k=K, buffer_b=B, window=Wn, num_q_heads=Hq, num_kv_heads=Hkv, batch=batch,
                  num_layers=L)
    a, b = _cache(wl, L, **kw), _cache(wl, L, **kw)
    dev = a.device

    def inputs(first, n):
        chunks = [W.stream_chunk(wl, 21, layer, first, n) for layer in range(L)]
        return [torch.stack([PU.bits_to_bf16_tensor(c[key], dev) for c in chunks])
                for key in ("q_bits", "k_bits", "v_bits")]

    q, k, v = inputs(0, K)
    for c in (a, b):
        c.append_all(q, k, v)
    for step in range(3):
        q, k, v = inputs(K + step * B, B)
        before = a.launch_count()
        assert a.append_evict_all(q, k, v) == L
        assert a.launch_count() - before == (1 if fused else 3)
        b.append_all(q, k, v)
        assert b.evict_all() == L
        torch.cuda.synchronize()
        for c in (a, b):
            status, code = c.check_device_error()
            assert status == 0, f"device error word {code:#x}"
        assert torch.equal(a.k_cache, b.k_cache) and torch.equal(a.v_cache, b.v_cache)
        assert torch.equal(a.positions, b.positions) and torch.equal(a.q_window, b.q_window)
        assert torch.equal(a.value_scores[..., :K], b.value_scores[..., :K])
        for layer in range(L):
            assert a.layer_state(layer) == b.layer_state(layer)
            assert a.layer_state(layer)["fill"] == K
