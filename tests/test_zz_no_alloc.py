"""The eviction entry point for callers that cannot allocate device memory.

Such callers (a plugin whose host process owns all device memory, a runtime that
forbids allocation after start-up) hand the library their caches but no workspace;
vase_evict_static_scratch then keeps its scratch in a static device array.  This
file checks, through the C ABI, that two such calls in a row give what vase_evict
gives on an identical copy of the caches -- for both scoring variants, and for a
window of more than 256 rows, whose score comes in four parts -- and that a layer
needing more scratch than the array holds is refused before anything runs.  It is
collected last on purpose.
"""

import numpy as np
import pytest
import torch

from paper_2606_03928_gb300 import workloads as W
import parity_utils as PU

pytestmark = pytest.mark.gpu


def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_03928_gb300 import build
    build.build()
    from paper_2606_03928_gb300 import vase as V
    return V


CASES = {
    # (workload, shrink arguments, variant)
    "attnv_k256": ("single_layer_k256", dict(num_layers=2, batch=2), "attnv"),
    "dkv_k256": ("single_layer_k256", dict(num_layers=2, batch=2), "dkv"),
    # G*W = 8 * 64 = 512 window rows: the window score is written as four parts that the selection adds
    "attnv_four_parts": ("qwen3_32b_k8192", dict(num_layers=2, batch=1, budget_k=256, buffer_b=64), "attnv"),
}


@pytest.mark.parametrize("case", sorted(CASES))
def test_static_scratch_eviction_matches_vase_evict_on_two_calls(case):
    V = _lib()
    name, shrink, variant = CASES[case]
    wl = W.shrink(W.WORKLOADS[name], **shrink)
    geometry = PU.geometry_of(wl, 2)
    ref = V.VaseCache(geometry, seed=5, variant=variant)  # evicted with vase_evict
    dut = V.VaseCache(geometry, seed=5, variant=variant)  # its caches go to the static-scratch entry point
    rounds = [3, 4]
    for layer in range(2):
        st = W.layer_state(wl, 7, layer, rounds[layer])
        PU.upload_layer(ref, layer, st, rounds[layer])
        PU.upload_layer(dut, layer, st, rounds[layer])
    torch.cuda.synchronize()
    # no workspace: the caller has none to give
    bufs = V.vase_buffers(dut.k_cache.data_ptr(), dut.v_cache.data_ptr(), dut.q_window.data_ptr(),
                          dut.positions.data_ptr(), dut.value_scores.data_ptr(), None)
    for layer in (1, 0):  # two calls in a row, sharing the one static scratch array
        ref.evict(layer)
        word = V.vase_evict_static_scratch(dut.cfg, bufs, layer, wl.slots, rounds[layer])
        assert word == 0, f"device error word {word:#x}"
    torch.cuda.synchronize()
    assert ref.check_device_error()[0] == 0
    assert torch.equal(ref.k_cache, dut.k_cache)
    assert torch.equal(ref.v_cache, dut.v_cache)
    assert torch.equal(ref.positions, dut.positions)
    PU.assert_close_scores(dut.value_scores.cpu().numpy().ravel(), ref.value_scores.cpu().numpy().ravel(),
                           "value magnitudes")
    # the kept set really changed the caches (K of K+B slots per unit, stable order)
    pos = dut.positions.cpu().numpy()
    assert np.all(pos[..., wl.budget_k:] == -1)
    assert np.all(np.diff(pos[..., :wl.budget_k], axis=-1) > 0)


def test_static_scratch_refuses_a_layer_larger_than_the_array():
    """The Qwen3-32B geometry at batch 16 needs about 17 MB of scratch per layer, more than the 16 MiB
    array: the call returns VASE_ERR_UNSUPPORTED from the configuration alone (no buffer is given, so
    nothing could have been launched)."""
    V = _lib()
    wl = W.shrink(W.WORKLOADS["qwen3_32b_k8192"], num_layers=1)
    cfg = V.vase_config_default(budget_k=wl.budget_k, buffer_b=wl.buffer_b, window=wl.window,
                                num_q_heads=wl.num_q_heads, num_kv_heads=wl.num_kv_heads, head_dim=128,
                                num_layers=1, batch=wl.batch)
    bufs = V.vase_buffers(None, None, None, None, None, None)
    with pytest.raises(V.VaseError) as exc:
        V.vase_evict_static_scratch(cfg, bufs, 0, wl.slots, 0)
    assert exc.value.status == V.VASE_ERR_UNSUPPORTED
    assert "VASE_STATIC_SCRATCH_BYTES" in str(exc.value)


def test_static_scratch_refuses_the_compressed_value_store():
    """The static-scratch eviction works on the bf16 value cache: with value_bits set it returns
    VASE_ERR_UNSUPPORTED from the configuration alone."""
    V = _lib()
    cfg = V.vase_config_default(budget_k=256, buffer_b=64, window=32, num_q_heads=16, num_kv_heads=8, head_dim=128,
                                num_layers=1, batch=1, value_bits=4)
    bufs = V.vase_buffers(None, None, None, None, None, None)
    with pytest.raises(V.VaseError) as exc:
        V.vase_evict_static_scratch(cfg, bufs, 0, 320, 0)
    assert exc.value.status == V.VASE_ERR_UNSUPPORTED
