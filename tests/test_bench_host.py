"""Host logic of bench.py, no GPU: the sweep grid, the bytes of one layer-round that the step roofline divides
by, and the clock sampler's choice of the samples taken inside the timed region."""

import datetime
import tempfile
import time

import pytest

import bench
from paper_2606_03928_gb300 import workloads as W


def test_sweep_grid_covers_the_axes_and_the_full_grid():
    pts = bench.sweep_grid(False)
    assert len(pts) == len(set(pts)) == 20
    assert (4096, 128, 32, 0.005) in pts  # the point `value` reports
    Ks, Bs = (1024, 2048, 4096, 8192, 16384), (32, 128, 512)
    assert {(K, B) for K, B, b, r in pts if (b, r) == (32, 0.005)} == {(K, B) for K in Ks for B in Bs}
    assert {b for K, B, b, r in pts if (K, B, r) == (4096, 128, 0.005)} == {1, 8, 32, 128}
    assert {r for K, B, b, r in pts if (K, B, b) == (4096, 128, 32)} == {0.0, 0.005, 0.02}
    full = bench.sweep_grid(True)
    assert len(full) == len(set(full)) == 5 * 3 * 4 * 3 and set(pts) <= set(full)


@pytest.mark.parametrize("name,variant,mb", [("qwen3_1p7b_k2048", "attnv", 139.5), ("qwen3_8b_k4096", "attnv", 1099.0),
                                             ("qwen3_8b_k4096", "dkv", 1091.0), ("qwen3_32b_k8192", "attnv", 1107.0)])
def test_step_bytes_are_the_fused_step_per_layer_round(name, variant, mb):
    """4dN (read K and V of every slot) + 4dK (write the kept rows) + 2d*G*W (the window queries, AttnV only),
    times the units of a layer: the per-layer-round bytes of the configurations' roofline table."""
    wl = W.WORKLOADS[name]
    assert bench.step_bytes(wl, variant) / 1e6 == pytest.approx(mb, abs=0.5)


class _Stopped:
    def terminate(self):
        pass

    def wait(self, timeout=None):
        pass


def _sampler_with_rows(rows, t_begin):
    cs = bench.ClockSampler(0)
    f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
    f.write("\n".join(rows) + "\n")
    f.flush()
    cs.file, cs.proc, cs.t_begin = f, _Stopped(), t_begin
    return cs


def _stamp(t):
    return datetime.datetime.fromtimestamp(t).strftime("%Y/%m/%d %H:%M:%S.%f")[:-3]


def test_clock_sampler_keeps_only_the_samples_of_the_timed_region():
    now = time.time()  # the region began a second ago and ends now; idle samples before and after it
    rows = [f"{_stamp(now - 3)}, 0, 345, 2070, 100.0, 0x0, Not Active, Not Active, Not Active, Not Active",
            f"{_stamp(now - 0.5)}, 0, 2070, 2070, 900.0, 0x4, Not Active, Not Active, Not Active, Active",
            f"{_stamp(now + 60)}, 0, 900, 2070, 100.0, 0x0, Active, Not Active, Not Active, Not Active"]
    out = _sampler_with_rows(rows, now - 1).stop()
    assert out == {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"], "samples": 1}


def test_clock_sampler_keeps_every_sample_when_no_stamp_parses():
    rows = ["t0, 0, 2070, 2070, 900.0, 0x0, Not Active, Not Active, Not Active, Not Active",
            "t1, 0, 1980, 2070, 950.0, 0x0, Active, Not Active, Not Active, Not Active"]
    out = _sampler_with_rows(rows, time.time()).stop()
    assert out == {"sm_mhz": 2025.0, "sm_max_mhz": 2070.0, "reasons": ["hw_slowdown"], "samples": 2}


def test_clock_sampler_brackets_a_region_shorter_than_the_sampling_interval():
    """No sample inside the region: the last sample before it and the first after it stand for it."""
    now = time.time()
    rows = [f"{_stamp(now - 5)}, 0, 345, 2070, 100.0, 0x0, Not Active, Not Active, Not Active, Not Active",
            f"{_stamp(now - 0.2)}, 0, 2070, 2070, 900.0, 0x0, Not Active, Not Active, Not Active, Not Active",
            f"{_stamp(now + 0.5)}, 0, 2040, 2070, 950.0, 0x4, Not Active, Not Active, Not Active, Active",
            f"{_stamp(now + 9)}, 0, 300, 2070, 100.0, 0x0, Active, Not Active, Not Active, Not Active"]
    cs = _sampler_with_rows(rows, now - 0.1)
    out = cs.stop()
    assert out == {"sm_mhz": 2055.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"], "samples": 2,
                   "bracketing": True}


def test_score_roofline_bound_follows_the_algorithmic_ratio():
    """The window score is tensor-bound where its QK^T FLOPs at the bf16 peak outlast its bytes at the HBM
    peak (Qwen3-32B geometry, G*W = 512) and HBM-bound otherwise (Qwen3-1.7B geometry, G*W = 32)."""
    for name, bound in (("qwen3_32b_k8192", "tensor"), ("qwen3_1p7b_k2048", "hbm")):
        wl = W.WORKLOADS[name]
        tab = bench.kernel_table({"score_attn": (1.0, 1), "select_compact": (1.0, 1)}, wl, "attnv", 100.0, 8,
                                 6799.3, 1897.1)
        assert tab["score_attn"]["bound"] == bound
        roof = bench.roofline_of(tab, "score_attn", wl, "attnv", 100.0, 8, 6799.3, 1897.1, "measured", None)
        assert roof["bound"] == bound and roof["unit"] == ("TFLOP/s" if bound == "tensor" else "GB/s")
        assert roof["frac"] == pytest.approx(roof["achieved"] / roof["peak"], rel=1e-3)
