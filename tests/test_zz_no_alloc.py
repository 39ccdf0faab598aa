"""The eviction entry point for callers that cannot allocate device memory.

Such callers (a plugin whose host process owns all device memory, a runtime that
forbids allocation after start-up) hand the library their caches but no workspace;
vase_evict_static_scratch then keeps its scratch in a static device array.  This
file checks, through the C ABI, that two such calls in a row give what vase_evict
gives on an identical copy of the caches.  It is collected last on purpose.
"""

import numpy as np
import pytest
import torch

from paper_2606_03928_gb300 import workloads as W
import parity_utils as PU

pytestmark = pytest.mark.gpu


def test_static_scratch_eviction_matches_vase_evict_on_two_calls():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_03928_gb300 import build
    build.build()
    from paper_2606_03928_gb300 import vase as V

    wl = W.shrink(W.WORKLOADS["single_layer_k256"], num_layers=2, batch=2)
    geometry = PU.geometry_of(wl, 2)
    ref = V.VaseCache(geometry, seed=5)        # evicted with vase_evict
    dut = V.VaseCache(geometry, seed=5)        # its caches go to the static-scratch entry point
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
