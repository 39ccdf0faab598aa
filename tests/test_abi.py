"""CPU checks of the C ABI: the library builds and loads, exports every symbol
include/vase.h declares, its struct layouts agree with the ctypes mirrors, and
configuration validation works without a GPU."""

import os
import re
import subprocess
import tempfile

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "vase.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2606_03928_gb300 import build
    build.build()
    from paper_2606_03928_gb300 import vase as V
    return V.load()


def _declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"^\s*[A-Za-z_][\w\s\*]*?\b(vase_\w+)\s*\(", text, flags=re.M)))


def test_header_declares_the_boundary():
    names = _declared_functions()
    for required in ("vase_create", "vase_append", "vase_evict", "vase_destroy"):
        assert required in names


def test_every_declared_symbol_is_exported(lib):
    from paper_2606_03928_gb300 import vase as V
    names = _declared_functions()
    assert sorted(V.EXPORTED) == names
    for n in names:
        assert hasattr(lib, n), n


def test_struct_layouts_match_ctypes(lib):
    from paper_2606_03928_gb300 import vase as V
    import ctypes
    structs = {
        "vase_config": V.vase_config, "vase_buffer_sizes": V.vase_buffer_sizes, "vase_buffers": V.vase_buffers,
        "vase_layer_state": V.vase_layer_state, "vase_kv_view": V.vase_kv_view, "vase_debug_view": V.vase_debug_view,
        "vase_mixed_buffers": V.vase_mixed_buffers, "vase_value_store": V.vase_value_store,
    }
    lines = ['#include <stdio.h>', '#include <stddef.h>', '#include "vase.h"', "int main(void) {"]
    for name, cls in structs.items():
        lines.append(f'printf("{name} %zu\\n", sizeof({name}));')
        for f, _ in cls._fields_:
            lines.append(f'printf("{name}.{f} %zu\\n", offsetof({name}, {f}));')
    lines.append("return 0; }")
    with tempfile.TemporaryDirectory() as d:
        src = os.path.join(d, "t.c")
        exe = os.path.join(d, "t")
        open(src, "w").write("\n".join(lines))
        subprocess.run(["gcc", "-I", os.path.join(ROOT, "include"), src, "-o", exe], check=True)
        out = subprocess.run([exe], capture_output=True, text=True, check=True).stdout.split("\n")
    got = dict(line.split() for line in out if line.strip())
    for name, cls in structs.items():
        assert int(got[name]) == ctypes.sizeof(cls), name
        for f, _ in cls._fields_:
            assert int(got[f"{name}.{f}"]) == getattr(cls, f).offset, f"{name}.{f}"


def test_config_validation_without_a_gpu(lib):
    from paper_2606_03928_gb300 import vase as V
    good = dict(budget_k=2048, buffer_b=128, window=32, num_q_heads=16, num_kv_heads=8, num_layers=28, batch=8)
    s = V.vase_get_buffer_sizes(V.vase_config_default(**good))
    assert s.k_cache == 28 * 8 * 8 * 2176 * 256 and s.positions == 28 * 8 * 8 * 2176 * 4
    assert s.q_window == 28 * 8 * 16 * 32 * 256
    for bad in (dict(head_dim=64), dict(num_q_heads=12, num_kv_heads=8), dict(pool_kernel=4), dict(buffer_b=4096),
                dict(n_v=2000), dict(window=64, num_q_heads=128), dict(dkv_rank=33), dict(variant=7),
                dict(budget_k=16384, buffer_b=16384)):
        cfg = V.vase_config_default(**{**good, **bad})
        with pytest.raises(V.VaseError):
            V.vase_get_buffer_sizes(cfg)


def test_value_store_configuration_without_a_gpu(lib):
    """The compressed value store: bit widths 2, 4, 8 only, AttnV only; its V buffer is the layout of codes,
    (s, z), masks, ring (N_v + 2B rows) and ring state per unit, smaller than the bf16 cache it replaces
    (Qwen3-1.7B geometry, one layer, K 2048, B 128, N_v 512)."""
    from oracle import vase_oracle as O
    from paper_2606_03928_gb300 import vase as V
    base = dict(budget_k=2048, buffer_b=128, window=32, num_q_heads=16, num_kv_heads=8, num_layers=1, batch=8)
    bf = V.vase_get_buffer_sizes(V.vase_config_default(**base)).v_cache
    units, N, words = 64, 2176, 68
    for bits in (2, 4, 8):
        st = V.vase_get_buffer_sizes(V.vase_config_default(value_bits=bits, **base)).v_cache
        per_unit, bf_unit = O.store_bytes(N, O.store_capacity(2048, 128, 512), 128, bits)
        assert bf == units * bf_unit
        exact = units * (per_unit + 4 * words + 16)   # + the mask words and the ring state
        assert exact <= st < exact + 5 * 256 and st < bf
    for bad in (dict(value_bits=3), dict(value_bits=16), dict(value_bits=4, variant=V.VASE_VARIANT_DKV)):
        with pytest.raises(V.VaseError):
            V.vase_get_buffer_sizes(V.vase_config_default(**{**base, **bad}))


def test_paper_defaults(lib):
    from paper_2606_03928_gb300 import vase as V
    c = V.vase_config_default()
    assert (c.n_v, c.dkv_rank, c.pool_kernel, c.stochastic, c.dkv_fixed_g, c.head_dim) == (-1, 20, 7, 1, 0, 128)


def test_status_strings(lib):
    assert lib.vase_status_string(-3) == b"cache not full"
    assert lib.vase_abi_version() == 3
