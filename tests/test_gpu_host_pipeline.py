"""The host-buffer pipeline of the C ABI (vase_stage_host_inputs, vase_append_all_staged,
vase_read_positions_all): a decode loop whose inputs and kept positions live in host memory.

Several eviction rounds staged from pinned host tensors, with each round's copies issued before
the previous round is appended (so both staging halves and the waits between the two streams are
exercised), must leave exactly the caches, window rings, value magnitudes and counters that the
same rounds leave when appended from device tensors; the positions read back to the host must equal
the device's after every round.
"""

import numpy as np
import pytest
import torch

from paper_2606_03928_gb300 import workloads as W
import parity_utils as PU

pytestmark = pytest.mark.gpu


def _tensors(wl, L, r, n, dev=None):
    chunks = [W.stream_chunk(wl, 31, layer, wl.budget_k + r * n, n) for layer in range(L)]
    out = []
    for key in ("q_bits", "k_bits", "v_bits"):
        t = torch.stack([torch.from_numpy(np.ascontiguousarray(c[key]).view(np.int16)).view(torch.bfloat16)
                         for c in chunks])
        out.append(t.to(dev) if dev is not None else t.pin_memory())
    return out


@pytest.mark.parametrize("variant,value_bits", [("attnv", 0), ("dkv", 0), ("attnv", 4)])
def test_staged_host_rounds_equal_device_appends(variant, value_bits):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_03928_gb300 import build
    build.build()
    from paper_2606_03928_gb300 import vase as V
    L = 3
    wl = W.shrink(W.WORKLOADS["single_layer_k256"], num_layers=L, batch=2, budget_k=128, buffer_b=32, window=16)
    K, B = wl.budget_k, wl.buffer_b
    ref = V.VaseCache(PU.geometry_of(wl, L), variant=variant, seed=11, value_bits=value_bits)
    dut = V.VaseCache(PU.geometry_of(wl, L), variant=variant, seed=11, value_bits=value_bits)
    # the same prefill of K tokens per layer in both
    pre = [W.stream_chunk(wl, 31, layer, 0, K) for layer in range(L)]
    for layer in range(L):
        args = [PU.bits_to_bf16_tensor(pre[layer][key], ref.device) for key in ("q_bits", "k_bits", "v_bits")]
        ref.append(layer, *args)
        dut.append(layer, *args)
    torch.cuda.synchronize()
    rounds = 5
    host = [_tensors(wl, L, r, B) for r in range(rounds)]
    dev = [_tensors(wl, L, r, B, ref.device) for r in range(rounds)]
    staging = dut.host_staging(B)
    copy_stream = torch.cuda.Stream()
    pos_host = [torch.empty((L, wl.batch, wl.num_kv_heads, K), dtype=torch.int32).pin_memory() for _ in range(rounds)]
    dut.stage_host_inputs(*host[0], staging, copy_stream)
    for r in range(rounds):
        if r + 1 < rounds:  # the next round's copies go out before this round's kernels
            dut.stage_host_inputs(*host[r + 1], staging, copy_stream)
        assert dut.append_all_staged() == V.VASE_EVICT_DUE
        assert dut.evict_all() == L
        dut.read_positions_all(pos_host[r], copy_stream)
        ref.append_all(*dev[r])
        ref.evict_all()
    torch.cuda.current_stream().wait_stream(copy_stream)
    torch.cuda.synchronize()
    assert ref.check_device_error()[0] == 0 and dut.check_device_error()[0] == 0
    assert torch.equal(ref.k_cache, dut.k_cache) and torch.equal(ref.v_cache, dut.v_cache)
    assert torch.equal(ref.q_window, dut.q_window) and torch.equal(ref.positions, dut.positions)
    assert torch.equal(ref.value_scores, dut.value_scores)
    for layer in range(L):
        assert ref.layer_state(layer) == dut.layer_state(layer)
    # the last read-back holds the final kept positions; every round's read-back is a stable kept set
    assert torch.equal(pos_host[-1], ref.positions[..., :K].cpu())
    for r in range(rounds):
        p = pos_host[r].numpy()
        assert np.all(np.diff(p, axis=-1) > 0)
        assert np.all(p[..., -B:] == (K + r * B + np.arange(B)))  # R_B: the round's B new tokens, kept


def test_staging_errors_leave_the_context_unchanged():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_03928_gb300 import build
    build.build()
    from paper_2606_03928_gb300 import vase as V
    L = 2
    wl = W.shrink(W.WORKLOADS["single_layer_k256"], num_layers=L, batch=1, budget_k=64, buffer_b=16, window=8)
    c = V.VaseCache(PU.geometry_of(wl, L), seed=1)
    q, k, v = _tensors(wl, L, 0, 16)
    staging = c.host_staging(16)
    cs = torch.cuda.Stream()
    with pytest.raises(V.VaseError):  # nothing staged yet
        c.append_all_staged()
    with pytest.raises(V.VaseError):  # a staging buffer for one step only
        c.stage_host_inputs(q, k, v, staging[: staging.numel() // 2], cs)
    c.stage_host_inputs(q, k, v, staging, cs)
    c.stage_host_inputs(q, k, v, staging, cs)
    with pytest.raises(V.VaseError) as exc:  # a third staged step before any append
        c.stage_host_inputs(q, k, v, staging, cs)
    assert exc.value.status == V.VASE_ERR_FULL
    for layer in range(L):
        assert c.layer_state(layer)["fill"] == 0
    assert c.append_all_staged() == V.VASE_OK
    torch.cuda.synchronize()
    assert c.layer_state(0)["fill"] == 16
