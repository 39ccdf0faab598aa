"""Helpers of the GPU parity tests: load synthetic unit states into a VaSE
context, run one eviction through the C ABI and compare with the fp64 oracle.

Tolerances (written here once, used by every parity test):
  * per-token scores within 1e-3 relative of the oracle, with an absolute
    floor of 1e-30 for weights that fp32 cannot represent;
  * kept-slot sets identical except for slots whose oracle selection key lies
    within 1e-4 relative of the K-th threshold of its ranking;
  * compacted K/V rows and positions bit-exact for the kept set.
"""

from __future__ import annotations

import numpy as np
import torch

from oracle import vase_oracle as O
from paper_2606_03928_gb300 import workloads as W

SCORE_RTOL = 1e-3
SCORE_ATOL = 1e-30
THRESH_RTOL = 1e-4


def bits_to_bf16_tensor(bits: np.ndarray, device) -> torch.Tensor:
    t = torch.from_numpy(np.ascontiguousarray(bits).view(np.int16))
    return t.view(torch.bfloat16).to(device)


def geometry_of(wl: W.Workload, num_layers=None):
    from paper_2606_03928_gb300.vase import Geometry
    return Geometry(wl.budget_k, wl.buffer_b, wl.window, wl.num_q_heads, wl.num_kv_heads,
                    num_layers if num_layers is not None else wl.num_layers, wl.batch)


def upload_layer(cache, layer: int, st: dict, round_index: int):
    """Writes a pre-eviction layer state (workloads.layer_state) into the context's buffers."""
    dev = cache.device
    cache.k_cache[layer].copy_(bits_to_bf16_tensor(st["k_bits"], dev))
    cache.v_cache[layer].copy_(bits_to_bf16_tensor(st["v_bits"], dev))
    cache.q_window[layer].copy_(bits_to_bf16_tensor(st["q_bits"], dev))
    cache.positions[layer].copy_(torch.from_numpy(st["positions"].astype(np.int32)).to(dev))
    N = cache.slots
    next_pos = int(st["positions"].max()) + 1
    cache.set_layer_state(layer, N, round_index, next_pos, 10 ** 6)
    cache.refresh_value_scores(layer)


def download(cache, layer):
    torch.cuda.synchronize()
    out = {
        "k_bits": cache.k_cache[layer].view(torch.int16).cpu().numpy().view(np.uint16),
        "v_bits": cache.v_cache[layer].view(torch.int16).cpu().numpy().view(np.uint16),
        "positions": cache.positions[layer].cpu().numpy(),
        "vmag": cache.value_scores[layer].cpu().numpy(),
    }
    dv = cache.debug_view()
    for k, v in dv.items():
        if k != "layer":
            out[k] = v.cpu().numpy()
    return out


def oracle_unit(wl, st, s, h, *, variant, round_index, seed, layer, **kw):
    G = wl.group
    q = st["q_bits"][s, h * G:(h + 1) * G].reshape(-1, wl.head_dim)
    return O.evict_unit_bits(q, st["k_bits"][s, h], st["v_bits"][s, h], st["positions"][s, h],
                             budget_k=wl.budget_k, buffer_b=wl.buffer_b, variant=variant, seed=seed, layer=layer,
                             seq=s, head=h, num_kv_heads=wl.num_kv_heads, rnd=round_index, group=G, **kw)


def assert_close_scores(gpu, ref, what, rtol=SCORE_RTOL, atol=SCORE_ATOL):
    gpu = np.asarray(gpu, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    err = np.abs(gpu - ref)
    bad = err > rtol * np.abs(ref) + atol
    if bad.any():
        i = np.flatnonzero(bad)[:5]
        raise AssertionError(f"{what}: {bad.sum()} of {bad.size} outside {rtol} rel; e.g. idx {i} gpu {gpu[i]} ref {ref[i]}")


def _near(values, thr, rtol=THRESH_RTOL):
    return np.abs(values - thr) <= rtol * abs(thr)


def check_unit(wl, ref, got_unit, orig_k, orig_v, orig_pos, *, variant, n_v, check_scores=True,
               value_kind=O.VALUE_RANGE):
    """Compares one unit of a GPU eviction with the oracle's result `ref`."""
    K, B = wl.budget_k, wl.buffer_b
    N = K + B
    src_g = got_unit["src"].astype(np.int64)
    # --- the compaction itself is a bit-exact stable gather of the GPU's own kept list
    assert src_g.shape == (K,)
    assert np.all(np.diff(src_g) > 0), "kept slots must be ascending (stable order)"
    assert src_g[0] >= 0 and src_g[-1] < N
    assert np.array_equal(got_unit["k_bits"][:K], orig_k[src_g]), "compacted keys differ from the kept rows"
    assert np.array_equal(got_unit["v_bits"][:K], orig_v[src_g]), "compacted values differ from the kept rows"
    assert np.array_equal(got_unit["positions"][:K], orig_pos[src_g]), "compacted positions differ"
    assert np.all(got_unit["positions"][K:] == -1)
    assert set(range(K, N)) <= set(src_g.tolist()), "the buffer R_B is always kept"
    # --- the per-slot value magnitudes moved with their rows (oracle magnitudes of the kept rows)
    if got_unit.get("vmag") is not None:
        vm_ref = O.value_magnitude(O.bf16_bits_to_f64(orig_v[src_g]), value_kind)
        assert_close_scores(got_unit["vmag"][:K], vm_ref, "compacted value magnitudes")
    # --- scores
    if check_scores:
        if variant == "attnv":
            assert_close_scores(got_unit["attn"], ref["attn"], "window attention score")
            if got_unit.get("value_score") is not None:
                assert_close_scores(got_unit["value_score"][:K], ref["value_score"], "value magnitude")
            if got_unit.get("pooled") is not None:
                assert_close_scores(got_unit["pooled"], ref["pooled"], "pooled score")
            if got_unit.get("key") is not None:
                kref = ref["key"][:K]
                cand = kref >= 0
                assert_close_scores(got_unit["key"][:K][cand], kref[cand], "selection key")
        else:
            assert_close_scores(got_unit["value_score"][:K], ref["value_score"], "leverage product")
    # --- kept set: identical up to near-threshold slots
    src_o = ref["src"]
    diff = set(src_g.tolist()) ^ set(src_o.tolist())
    if diff:
        allowed = set()
        if variant == "attnv":
            vref = ref["value_score"]
            if n_v > 0:
                thr_v = np.sort(vref)[::-1][n_v - 1]
                allowed |= set(np.flatnonzero(_near(vref, thr_v)).tolist())
            kref = ref["key"][:K]
            cand = np.flatnonzero(kref >= 0)
            m = K - n_v - B
            if m > 0:
                thr = np.sort(kref[cand])[::-1][m - 1]
                allowed |= set(cand[_near(kref[cand], thr)].tolist())
        else:
            s = ref["value_score"]
            thr = np.sort(s)[::-1][K - B - 1]
            allowed |= set(np.flatnonzero(_near(s, thr)).tolist())
        extra = diff - allowed
        assert not extra, f"kept sets differ away from the threshold at slots {sorted(extra)[:10]}"
    else:
        assert np.array_equal(got_unit["k_bits"][:K], ref["k_bits_new"])
        assert np.array_equal(got_unit["v_bits"][:K], ref["v_bits_new"])
    return len(diff)


def unit_slice(got, s, h, Hkv):
    u = s * Hkv + h
    return {
        "k_bits": got["k_bits"][s, h], "v_bits": got["v_bits"][s, h], "positions": got["positions"][s, h],
        "src": got["src"][u], "attn": got["attn"][u], "pooled": got["pooled"][u], "vmag": got["vmag"][s, h],
        "value_score": got["value_score"][u], "key": got["key"][u],
    }
