"""Python binding of the VaSE C ABI (include/vase.h): argument marshalling only.

Every step of the eviction path runs in the CUDA kernels of libvase.so; this
module only converts arguments, and uses PyTorch for device memory and
streams.  It raises if the compiled library is missing: there is no CPU
fallback.
"""

from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "_lib", "libvase.so")

VASE_OK = 0
VASE_EVICT_DUE = 1
VASE_ERR_INVALID = -1
VASE_ERR_FULL = -2
VASE_ERR_NOT_FULL = -3
VASE_ERR_CUDA = -4
VASE_ERR_UNSUPPORTED = -5
VASE_ERR_ALIGN = -6
VASE_ERR_DEVICE = -7
VASE_SITE_SELF_TEST = 127  # error-word site of vase_self_test_wait_timeout
VASE_SITE_STORE_OVERFLOW, VASE_SITE_STORE_STATE = 80, 81  # error-word sites of the compressed value store

VASE_VARIANT_ATTNV = 0
VASE_VARIANT_DKV = 1
VASE_VALUE_RANGE, VASE_VALUE_L2, VASE_VALUE_VAR = 0, 1, 2
VASE_RESERVE_VALUE, VASE_RESERVE_RANDOM = 0, 1
VASE_GQA_MEAN, VASE_GQA_MAX = 0, 1

EXPORTED = [
    "vase_config_default", "vase_get_buffer_sizes", "vase_create", "vase_destroy", "vase_append",
    "vase_append_host", "vase_evict", "vase_read_positions", "vase_get_layer_state", "vase_set_layer_state",
    "vase_kv_view_get", "vase_debug_view_get", "vase_check_device_error", "vase_launch_count",
    "vase_status_string", "vase_last_error", "vase_abi_version", "vase_profile_enable", "vase_profile_collect",
    "vase_append_all", "vase_append_all_strided", "vase_evict_all", "vase_self_test_wait_timeout", "vase_refresh_value_scores", "vase_evict_static_scratch",
    "vase_decode_attention", "vase_mixed_buffer_sizes", "vase_quantize_values", "vase_decode_attention_mixed",
    "vase_host_staging_bytes", "vase_stage_host_inputs", "vase_append_all_staged", "vase_read_positions_all",
    "vase_value_store_get", "vase_append_evict_all",
]
KERNEL_NAMES = ["append", "score_attn", "value_score", "dkv_score", "select_compact", "evict_small", "store_append",
                "store_evict"]


class vase_config(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "budget_k", "buffer_b", "window", "num_q_heads", "num_kv_heads", "head_dim", "num_layers", "batch",
        "variant", "n_v", "value_score", "pool_kernel", "dkv_rank", "stochastic", "dkv_fixed_g", "debug_outputs")] + [
        ("seed", ctypes.c_uint64)] + [(n, ctypes.c_int32) for n in ("reserve_kind", "gqa_reduce", "dkv_shared_g",
                                                                     "value_bits")]


class vase_buffer_sizes(ctypes.Structure):
    _fields_ = [(n, ctypes.c_size_t) for n in ("k_cache", "v_cache", "q_window", "positions", "value_scores",
                                               "workspace")]


class vase_buffers(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in ("k_cache", "v_cache", "q_window", "positions", "value_scores",
                                               "workspace")]


class vase_layer_state(ctypes.Structure):
    _fields_ = [("fill", ctypes.c_int32), ("round", ctypes.c_int32), ("next_position", ctypes.c_int64),
                ("queries_seen", ctypes.c_int64)]


class vase_kv_view(ctypes.Structure):
    _fields_ = [("k", ctypes.c_void_p), ("v", ctypes.c_void_p), ("positions", ctypes.c_void_p),
                ("value_scores", ctypes.c_void_p), ("unit_stride", ctypes.c_int64), ("slots", ctypes.c_int32),
                ("fill", ctypes.c_int32)]


class vase_mixed_buffers(ctypes.Structure):
    _fields_ = [("codes", ctypes.c_void_p), ("qparams", ctypes.c_void_p), ("rmask", ctypes.c_void_p),
                ("hp_rows", ctypes.c_void_p)]


class vase_value_store(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in ("codes", "sz", "mask", "ring", "state")] + [
        (n, ctypes.c_int32) for n in ("bits", "code_row", "slots", "sz_stride", "mask_stride", "ring_rows", "units",
                                      "fill")]


class vase_debug_view(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in ("attn", "pooled", "value_score", "key", "keep", "src")] + [
        ("units", ctypes.c_int32), ("slots", ctypes.c_int32), ("layer", ctypes.c_int32)]


_lib = None


def load(path: str = LIB_PATH):
    """Loads libvase.so (built by paper_2606_03928_gb300.build); raises if it is missing."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"VaSE CUDA library not built ({path}); run `python -m paper_2606_03928_gb300.build`")
    lib = ctypes.CDLL(path)
    P, I32, I64, U32 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_uint32
    sig = {
        "vase_config_default": (None, [ctypes.POINTER(vase_config)]),
        "vase_get_buffer_sizes": (ctypes.c_int, [ctypes.POINTER(vase_config), ctypes.POINTER(vase_buffer_sizes)]),
        "vase_create": (ctypes.c_int, [ctypes.POINTER(vase_config), ctypes.POINTER(vase_buffers),
                                       ctypes.POINTER(P)]),
        "vase_destroy": (None, [P]),
        "vase_append": (ctypes.c_int, [P, I32, P, P, P, I32, P]),
        "vase_append_host": (ctypes.c_int, [P, I32, P, P, P, I32, P]),
        "vase_append_all": (ctypes.c_int, [P, P, P, P, I32, P]),
        "vase_append_all_strided": (ctypes.c_int, [P, P, P, P, I32, I64, I64, P]),
        "vase_self_test_wait_timeout": (ctypes.c_int, [P, P]),
        "vase_evict": (ctypes.c_int, [P, I32, P]),
        "vase_evict_all": (ctypes.c_int, [P, P]),
        "vase_append_evict_all": (ctypes.c_int, [P, P, P, P, I32, I64, I64, P]),
        "vase_refresh_value_scores": (ctypes.c_int, [P, I32, P]),
        "vase_evict_static_scratch": (ctypes.c_int, [ctypes.POINTER(vase_config), ctypes.POINTER(vase_buffers), I32,
                                                     ctypes.POINTER(vase_layer_state), ctypes.POINTER(U32), P]),
        "vase_read_positions": (ctypes.c_int, [P, I32, P, P]),
        "vase_host_staging_bytes": (ctypes.c_size_t, [ctypes.POINTER(vase_config), I32]),
        "vase_stage_host_inputs": (ctypes.c_int, [P, P, P, P, I32, I64, I64, P, ctypes.c_size_t, P]),
        "vase_append_all_staged": (ctypes.c_int, [P, P]),
        "vase_read_positions_all": (ctypes.c_int, [P, P, P, P]),
        "vase_decode_attention": (ctypes.c_int, [P, I32, P, P, P]),
        "vase_mixed_buffer_sizes": (ctypes.c_int, [ctypes.POINTER(vase_config), I32] +
                                    [ctypes.POINTER(ctypes.c_size_t)] * 4),
        "vase_quantize_values": (ctypes.c_int, [P, I32, I32, ctypes.POINTER(vase_mixed_buffers), P]),
        "vase_decode_attention_mixed": (ctypes.c_int, [P, I32, I32, ctypes.POINTER(vase_mixed_buffers), P, P, P]),
        "vase_get_layer_state": (ctypes.c_int, [P, I32, ctypes.POINTER(vase_layer_state)]),
        "vase_set_layer_state": (ctypes.c_int, [P, I32, ctypes.POINTER(vase_layer_state)]),
        "vase_kv_view_get": (ctypes.c_int, [P, I32, ctypes.POINTER(vase_kv_view)]),
        "vase_debug_view_get": (ctypes.c_int, [P, I32, ctypes.POINTER(vase_debug_view)]),
        "vase_value_store_get": (ctypes.c_int, [P, I32, ctypes.POINTER(vase_value_store)]),
        "vase_check_device_error": (ctypes.c_int, [P, P, ctypes.POINTER(U32)]),
        "vase_launch_count": (I64, [P]),
        "vase_status_string": (ctypes.c_char_p, [ctypes.c_int]),
        "vase_last_error": (ctypes.c_char_p, [P]),
        "vase_abi_version": (ctypes.c_int, []),
        "vase_profile_enable": (ctypes.c_int, [P, ctypes.c_int]),
        "vase_profile_collect": (ctypes.c_int, [P, ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_int64)]),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    _lib = lib
    return lib


class VaseError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__(f"{msg} (status {status})")
        self.status = status


# ---------------------------------------------------------------------------- C-ABI mirrors

def vase_config_default(**fields) -> vase_config:
    cfg = vase_config()
    load().vase_config_default(ctypes.byref(cfg))
    for k, v in fields.items():
        setattr(cfg, k, v)
    return cfg


def vase_get_buffer_sizes(cfg: vase_config) -> vase_buffer_sizes:
    out = vase_buffer_sizes()
    st = load().vase_get_buffer_sizes(ctypes.byref(cfg), ctypes.byref(out))
    if st != VASE_OK:
        raise VaseError(st, "invalid VaSE configuration: " + load().vase_last_error(None).decode())
    return out


def vase_create(cfg: vase_config, bufs: vase_buffers) -> int:
    h = ctypes.c_void_p()
    st = load().vase_create(ctypes.byref(cfg), ctypes.byref(bufs), ctypes.byref(h))
    if st != VASE_OK:
        raise VaseError(st, "vase_create failed: " + load().vase_last_error(None).decode())
    return h.value


def vase_destroy(ctx: int) -> None:
    load().vase_destroy(ctx)


def _stream_ptr(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _check(ctx, st, what):
    if st < 0:
        raise VaseError(st, f"{what}: {load().vase_last_error(ctx).decode()}")
    return st


def vase_append(ctx, layer, q_ptr, k_ptr, v_ptr, n_tokens, stream=None):
    return _check(ctx, load().vase_append(ctx, layer, q_ptr, k_ptr, v_ptr, n_tokens, _stream_ptr(stream)),
                  "vase_append")


def vase_append_host(ctx, layer, q_ptr, k_ptr, v_ptr, n_tokens, stream=None):
    return _check(ctx, load().vase_append_host(ctx, layer, q_ptr, k_ptr, v_ptr, n_tokens, _stream_ptr(stream)),
                  "vase_append_host")


def vase_append_all(ctx, q_ptr, k_ptr, v_ptr, n_tokens, stream=None):
    return _check(ctx, load().vase_append_all(ctx, q_ptr, k_ptr, v_ptr, n_tokens, _stream_ptr(stream)),
                  "vase_append_all")


def vase_append_all_strided(ctx, q_ptr, k_ptr, v_ptr, n_tokens, q_layer_stride, kv_layer_stride, stream=None):
    return _check(ctx, load().vase_append_all_strided(ctx, q_ptr, k_ptr, v_ptr, n_tokens, q_layer_stride,
                                                      kv_layer_stride, _stream_ptr(stream)),
                  "vase_append_all_strided")


def vase_self_test_wait_timeout(ctx, stream=None):
    return _check(ctx, load().vase_self_test_wait_timeout(ctx, _stream_ptr(stream)), "vase_self_test_wait_timeout")


def vase_evict(ctx, layer, stream=None):
    return _check(ctx, load().vase_evict(ctx, layer, _stream_ptr(stream)), "vase_evict")


def vase_evict_all(ctx, stream=None):
    return _check(ctx, load().vase_evict_all(ctx, _stream_ptr(stream)), "vase_evict_all")


def vase_append_evict_all(ctx, q_ptr, k_ptr, v_ptr, n_tokens, q_layer_stride, kv_layer_stride, stream=None):
    return _check(ctx, load().vase_append_evict_all(ctx, q_ptr, k_ptr, v_ptr, n_tokens, q_layer_stride,
                                                    kv_layer_stride, _stream_ptr(stream)),
                  "vase_append_evict_all")


def vase_refresh_value_scores(ctx, layer, stream=None):
    return _check(ctx, load().vase_refresh_value_scores(ctx, layer, _stream_ptr(stream)), "vase_refresh_value_scores")


def vase_evict_static_scratch(cfg: vase_config, bufs: vase_buffers, layer, fill, round_, stream=None,
                              check_error=True):
    """One eviction of one layer with the library's static device scratch instead of a workspace.

    For callers that cannot allocate device memory (they pass the caches only; bufs.workspace may be
    None).  Returns the device error word when check_error is set (the call then waits for the stream).
    The caller keeps the layer counters: afterwards fill is K and the round has advanced by one."""
    st = vase_layer_state(fill, round_, 0, 0)
    word = ctypes.c_uint32(0)
    status = load().vase_evict_static_scratch(ctypes.byref(cfg), ctypes.byref(bufs), layer, ctypes.byref(st),
                                              ctypes.byref(word) if check_error else None, _stream_ptr(stream))
    if status < 0:
        raise VaseError(status, "vase_evict_static_scratch: " + load().vase_last_error(None).decode())
    return word.value


def vase_decode_attention(ctx, layer, q_ptr, out_ptr, stream=None):
    return _check(ctx, load().vase_decode_attention(ctx, layer, q_ptr, out_ptr, _stream_ptr(stream)),
                  "vase_decode_attention")


def vase_mixed_buffer_sizes(cfg: vase_config, bits):
    sizes = [ctypes.c_size_t(), ctypes.c_size_t(), ctypes.c_size_t(), ctypes.c_size_t()]
    st = load().vase_mixed_buffer_sizes(ctypes.byref(cfg), bits, *(ctypes.byref(x) for x in sizes))
    if st != VASE_OK:
        raise VaseError(st, "vase_mixed_buffer_sizes: " + load().vase_last_error(None).decode())
    return tuple(x.value for x in sizes)


def vase_quantize_values(ctx, layer, bits, mb: vase_mixed_buffers, stream=None):
    return _check(ctx, load().vase_quantize_values(ctx, layer, bits, ctypes.byref(mb), _stream_ptr(stream)),
                  "vase_quantize_values")


def vase_decode_attention_mixed(ctx, layer, bits, mb: vase_mixed_buffers, q_ptr, out_ptr, stream=None):
    return _check(ctx, load().vase_decode_attention_mixed(ctx, layer, bits, ctypes.byref(mb), q_ptr, out_ptr,
                                                          _stream_ptr(stream)), "vase_decode_attention_mixed")


def vase_read_positions(ctx, layer, host_ptr, stream=None):
    return _check(ctx, load().vase_read_positions(ctx, layer, host_ptr, _stream_ptr(stream)), "vase_read_positions")


def vase_host_staging_bytes(cfg: vase_config, n_tokens) -> int:
    return int(load().vase_host_staging_bytes(ctypes.byref(cfg), n_tokens))


def vase_stage_host_inputs(ctx, q_ptr, k_ptr, v_ptr, n_tokens, q_layer_stride, kv_layer_stride, staging_ptr,
                           staging_bytes, copy_stream):
    return _check(ctx, load().vase_stage_host_inputs(ctx, q_ptr, k_ptr, v_ptr, n_tokens, q_layer_stride,
                                                     kv_layer_stride, staging_ptr, staging_bytes,
                                                     _stream_ptr(copy_stream)), "vase_stage_host_inputs")


def vase_append_all_staged(ctx, stream=None):
    return _check(ctx, load().vase_append_all_staged(ctx, _stream_ptr(stream)), "vase_append_all_staged")


def vase_read_positions_all(ctx, host_ptr, copy_stream, stream=None):
    return _check(ctx, load().vase_read_positions_all(ctx, host_ptr, _stream_ptr(copy_stream), _stream_ptr(stream)),
                  "vase_read_positions_all")


def vase_get_layer_state(ctx, layer) -> vase_layer_state:
    st = vase_layer_state()
    _check(ctx, load().vase_get_layer_state(ctx, layer, ctypes.byref(st)), "vase_get_layer_state")
    return st


def vase_set_layer_state(ctx, layer, fill, round_, next_position, queries_seen):
    st = vase_layer_state(fill, round_, next_position, queries_seen)
    return _check(ctx, load().vase_set_layer_state(ctx, layer, ctypes.byref(st)), "vase_set_layer_state")


def vase_check_device_error(ctx, stream=None):
    code = ctypes.c_uint32(0)
    st = load().vase_check_device_error(ctx, _stream_ptr(stream), ctypes.byref(code))
    return st, code.value


def vase_launch_count(ctx) -> int:
    return int(load().vase_launch_count(ctx))


def vase_profile_enable(ctx, enable: bool):
    return _check(ctx, load().vase_profile_enable(ctx, int(enable)), "vase_profile_enable")


def vase_profile_collect(ctx):
    """{kernel name: (summed device ms, launches)} since profiling was enabled or last collected."""
    ms = (ctypes.c_double * len(KERNEL_NAMES))()
    n = (ctypes.c_int64 * len(KERNEL_NAMES))()
    _check(ctx, load().vase_profile_collect(ctx, ms, n), "vase_profile_collect")
    return {name: (ms[i], int(n[i])) for i, name in enumerate(KERNEL_NAMES)}


# ---------------------------------------------------------------------------- convenience owner

@dataclass
class Geometry:
    budget_k: int
    buffer_b: int
    window: int
    num_q_heads: int
    num_kv_heads: int
    num_layers: int
    batch: int
    head_dim: int = 128


class VaseCache:
    """A VaSE context plus its device buffers, allocated with PyTorch on the current device."""

    def __init__(self, geometry: Geometry, *, variant="attnv", n_v=-1, value_score=VASE_VALUE_RANGE,
                 pool_kernel=7, dkv_rank=20, stochastic=True, dkv_fixed_g=False, debug_outputs=False, seed=0,
                 reserve="value", gqa="mean", dkv_shared_g=False, value_bits=0, device=None):
        g = geometry
        self.geometry = g
        self.cfg = vase_config_default(
            budget_k=g.budget_k, buffer_b=g.buffer_b, window=g.window, num_q_heads=g.num_q_heads,
            num_kv_heads=g.num_kv_heads, head_dim=g.head_dim, num_layers=g.num_layers, batch=g.batch,
            variant=VASE_VARIANT_ATTNV if variant == "attnv" else VASE_VARIANT_DKV, n_v=n_v,
            value_score=value_score, pool_kernel=pool_kernel, dkv_rank=dkv_rank, stochastic=int(stochastic),
            dkv_fixed_g=int(dkv_fixed_g), debug_outputs=int(debug_outputs), seed=seed,
            reserve_kind={"value": VASE_RESERVE_VALUE, "random": VASE_RESERVE_RANDOM}[reserve],
            gqa_reduce={"mean": VASE_GQA_MEAN, "max": VASE_GQA_MAX}[gqa], dkv_shared_g=int(dkv_shared_g),
            value_bits=int(value_bits))
        sizes = vase_get_buffer_sizes(self.cfg)
        dev = torch.device(device) if device is not None else torch.device("cuda", torch.cuda.current_device())
        self.device = dev
        N = g.budget_k + g.buffer_b
        self.slots = N
        self.k_cache = torch.empty((g.num_layers, g.batch, g.num_kv_heads, N, g.head_dim), dtype=torch.bfloat16,
                                   device=dev)
        # the bf16 value cache, or (value_bits > 0) the compressed value store the library lays out itself (zeroed,
        # so that the bytes the library never writes -- padding, unused ring rows -- compare equal across caches)
        self.v_cache = (torch.zeros(sizes.v_cache, dtype=torch.uint8, device=dev) if value_bits
                        else torch.empty_like(self.k_cache))
        self.value_bits = int(value_bits)
        self.q_window = torch.empty((g.num_layers, g.batch, g.num_q_heads, g.window, g.head_dim),
                                    dtype=torch.bfloat16, device=dev)
        self.positions = torch.full((g.num_layers, g.batch, g.num_kv_heads, N), -1, dtype=torch.int32, device=dev)
        self.value_scores = torch.zeros((g.num_layers, g.batch, g.num_kv_heads, N), dtype=torch.float32, device=dev)
        self.workspace = torch.zeros(sizes.workspace, dtype=torch.uint8, device=dev)
        assert self.k_cache.numel() * 2 == sizes.k_cache and self.positions.numel() * 4 == sizes.positions
        assert self.value_scores.numel() * 4 == sizes.value_scores
        bufs = vase_buffers(self.k_cache.data_ptr(), self.v_cache.data_ptr(), self.q_window.data_ptr(),
                            self.positions.data_ptr(), self.value_scores.data_ptr(), self.workspace.data_ptr())
        with torch.cuda.device(dev):
            self.ctx = vase_create(self.cfg, bufs)

    def close(self):
        if getattr(self, "ctx", None):
            vase_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # --- stream-ordered calls
    def append(self, layer, q, k, v, stream=None):
        """q [n, b, Hq, d], k/v [n, b, Hkv, d] bf16 CUDA tensors (contiguous)."""
        for t in (q, k, v):
            assert t.is_cuda and t.dtype == torch.bfloat16 and t.is_contiguous()
        return vase_append(self.ctx, layer, q.data_ptr(), k.data_ptr(), v.data_ptr(), q.shape[0], stream)

    def append_host(self, layer, q, k, v, stream=None):
        """Same as append with CPU tensors (pinned for asynchronous copies)."""
        for t in (q, k, v):
            assert (not t.is_cuda) and t.dtype == torch.bfloat16 and t.is_contiguous()
        return vase_append_host(self.ctx, layer, q.data_ptr(), k.data_ptr(), v.data_ptr(), q.shape[0], stream)

    def append_all(self, q, k, v, stream=None):
        """q [L, n, b, Hq, d], k/v [L, n, b, Hkv, d] bf16 CUDA tensors: n tokens for every layer, one launch."""
        for t in (q, k, v):
            assert t.is_cuda and t.dtype == torch.bfloat16 and t.is_contiguous()
        return vase_append_all(self.ctx, q.data_ptr(), k.data_ptr(), v.data_ptr(), q.shape[1], stream)

    def evict(self, layer, stream=None):
        return vase_evict(self.ctx, layer, stream)

    def refresh_value_scores(self, layer, stream=None):
        """Recomputes the per-slot value magnitudes of one layer after its V rows were written directly."""
        return vase_refresh_value_scores(self.ctx, layer, stream)

    def evict_all(self, stream=None):
        """Evicts every full layer in batched launches; returns how many layers were evicted."""
        return vase_evict_all(self.ctx, stream)

    def append_evict_all(self, q, k, v, stream=None):
        """One step: q [L, n, b, Hq, d], k/v [L, n, b, Hkv, d] bf16 CUDA tensors appended to every layer, then every
        full layer evicted (one fused launch where that applies); returns how many layers were evicted."""
        for t in (q, k, v):
            assert t.is_cuda and t.dtype == torch.bfloat16 and t.is_contiguous()
        return vase_append_evict_all(self.ctx, q.data_ptr(), k.data_ptr(), v.data_ptr(), q.shape[1],
                                     q[0].numel() * 2, k[0].numel() * 2, stream)

    def decode_attention(self, layer, q: torch.Tensor, out: torch.Tensor = None, stream=None):
        """Attention output of one decode step over the layer's cached pairs: q [b, Hq, d] bf16 CUDA tensor,
        returns (or fills) out [b, Hq, d] fp32."""
        assert q.is_cuda and q.dtype == torch.bfloat16 and q.is_contiguous()
        if out is None:
            out = torch.empty(q.shape, dtype=torch.float32, device=q.device)
        assert out.is_cuda and out.dtype == torch.float32 and out.is_contiguous()
        vase_decode_attention(self.ctx, layer, q.data_ptr(), out.data_ptr(), stream)
        return out

    def mixed_buffers(self, bits):
        """Device buffers of one layer's mixed-precision values (codes, (s, z), reserved mask, reserved rows) as
        torch tensors, plus the vase_mixed_buffers struct that points at them."""
        n_codes, n_qp, n_mask, n_hp = vase_mixed_buffer_sizes(self.cfg, bits)
        t = {"codes": torch.zeros(n_codes, dtype=torch.uint8, device=self.device),
             "qparams": torch.zeros(n_qp // 4, dtype=torch.float32, device=self.device),
             "rmask": torch.zeros(n_mask // 4, dtype=torch.int32, device=self.device),
             "hp_rows": torch.zeros(n_hp // 2, dtype=torch.bfloat16, device=self.device)}
        mb = vase_mixed_buffers(t["codes"].data_ptr(), t["qparams"].data_ptr(), t["rmask"].data_ptr(),
                                t["hp_rows"].data_ptr())
        return mb, t

    def quantize_values(self, layer, bits, mb, stream=None):
        """Codes of the layer's unreserved kept values, right after its eviction."""
        return vase_quantize_values(self.ctx, layer, bits, mb, stream)

    def decode_attention_mixed(self, layer, bits, mb, q: torch.Tensor, out: torch.Tensor = None, stream=None):
        """decode_attention with the unreserved values read from the codes of the layer's current round."""
        assert q.is_cuda and q.dtype == torch.bfloat16 and q.is_contiguous()
        if out is None:
            out = torch.empty(q.shape, dtype=torch.float32, device=q.device)
        assert out.is_cuda and out.dtype == torch.float32 and out.is_contiguous()
        vase_decode_attention_mixed(self.ctx, layer, bits, mb, q.data_ptr(), out.data_ptr(), stream)
        return out

    def host_staging(self, n_tokens):
        """A device staging buffer for vase_stage_host_inputs (two steps of n_tokens per layer)."""
        nbytes = 2 * vase_host_staging_bytes(self.cfg, n_tokens)
        return torch.empty(nbytes, dtype=torch.uint8, device=self.device)

    def stage_host_inputs(self, q, k, v, staging, copy_stream):
        """q [L, n, b, Hq, d], k/v [L, n, b, Hkv, d] bf16 CPU tensors (pinned for asynchronous copies):
        one step's inputs of every layer, copied on copy_stream into the next half of `staging`."""
        for t in (q, k, v):
            assert (not t.is_cuda) and t.dtype == torch.bfloat16 and t.is_contiguous()
        n = q.shape[1]
        return vase_stage_host_inputs(self.ctx, q.data_ptr(), k.data_ptr(), v.data_ptr(), n,
                                      q[0].numel() * 2, k[0].numel() * 2, staging.data_ptr(), staging.numel(),
                                      copy_stream)

    def append_all_staged(self, stream=None):
        return vase_append_all_staged(self.ctx, stream)

    def read_positions_all(self, out: torch.Tensor, copy_stream, stream=None):
        """Every layer's K kept positions into a CPU int32 tensor [L, b, Hkv, K] (pinned), on copy_stream."""
        assert (not out.is_cuda) and out.dtype == torch.int32 and out.is_contiguous()
        return vase_read_positions_all(self.ctx, out.data_ptr(), copy_stream, stream)

    def read_positions(self, layer, out: torch.Tensor, stream=None):
        """Copies the K kept positions of every unit into a CPU int32 tensor [b, Hkv, K]."""
        assert (not out.is_cuda) and out.dtype == torch.int32 and out.is_contiguous()
        return vase_read_positions(self.ctx, layer, out.data_ptr(), stream)

    def layer_state(self, layer):
        s = vase_get_layer_state(self.ctx, layer)
        return {"fill": s.fill, "round": s.round, "next_position": s.next_position, "queries_seen": s.queries_seen}

    def set_layer_state(self, layer, fill, round_, next_position, queries_seen):
        return vase_set_layer_state(self.ctx, layer, fill, round_, next_position, queries_seen)

    def check_device_error(self, stream=None):
        return vase_check_device_error(self.ctx, stream)

    def launch_count(self):
        return vase_launch_count(self.ctx)

    def profile_enable(self, enable=True):
        return vase_profile_enable(self.ctx, enable)

    def profile_collect(self):
        return vase_profile_collect(self.ctx)

    def value_store(self, layer):
        """One layer's compressed value store as torch views: codes [units, N, code_row] uint8, sz [units, Np, 2]
        fp32, mask [units, mask_stride] int32, ring [units, H, d] bf16, state [units, 4] int32 (ring head, count)."""
        vs = vase_value_store()
        _check(self.ctx, load().vase_value_store_get(self.ctx, layer, ctypes.byref(vs)), "vase_value_store_get")
        base = self.v_cache.data_ptr()
        U = vs.units

        def sl(ptr, nbytes, dtype):
            off = ptr - base
            return self.v_cache[off:off + nbytes].view(dtype)

        d = self.geometry.head_dim
        return {
            "codes": sl(vs.codes, U * vs.slots * vs.code_row, torch.uint8).view(U, vs.slots, vs.code_row),
            "sz": sl(vs.sz, U * vs.sz_stride * 8, torch.float32).view(U, vs.sz_stride, 2),
            "mask": sl(vs.mask, U * vs.mask_stride * 4, torch.int32).view(U, vs.mask_stride),
            "ring": sl(vs.ring, U * vs.ring_rows * d * 2, torch.bfloat16).view(U, vs.ring_rows, d),
            "state": sl(vs.state, U * 16, torch.int32).view(U, 4),
            "bits": vs.bits, "ring_rows": vs.ring_rows, "fill": vs.fill,
        }

    def debug_view(self, slot=0):
        """Workspace results of the latest eviction call for its slot-th layer: attn, pooled, value_score, key
        [units, N], keep, src [units, K], and the layer they belong to."""
        dv = vase_debug_view()
        _check(self.ctx, load().vase_debug_view_get(self.ctx, slot, ctypes.byref(dv)), "vase_debug_view_get")
        base = self.workspace.data_ptr()
        U, N, K = dv.units, dv.slots, self.geometry.budget_k

        def sl(ptr, nbytes, dtype):
            off = ptr - base
            return self.workspace[off:off + nbytes].view(dtype)

        return {
            "attn": sl(dv.attn, U * N * 4, torch.float32).view(U, N),
            "pooled": sl(dv.pooled, U * N * 4, torch.float32).view(U, N),
            "value_score": sl(dv.value_score, U * N * 4, torch.float32).view(U, N),
            "key": sl(dv.key, U * N * 4, torch.float32).view(U, N),
            "keep": sl(dv.keep, U * N, torch.uint8).view(U, N),
            "src": sl(dv.src, U * K * 4, torch.int32).view(U, K),
            "layer": dv.layer,
        }
