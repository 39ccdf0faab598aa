#!/usr/bin/env python
"""Throughput of the VaSE eviction step on one GB300 (or N, one process per GPU).

One step = one eviction round of every layer of the workload: for each layer
the B new decode tokens of the stream are appended (window ring + cache) and
the layer is evicted (score, value magnitude, selection, compaction), all
through the C ABI.  The default workload is the largest configuration, the
Qwen3-32B attention geometry (64 layers, 64/8 heads, d = 128, batch 16,
K = 8192, B = 256, W = 64; seeded synthetic decode tokens, a few distinct
rounds replayed cyclically); the same run also measures the other
configurations (the `configs` records).  Every step touches about 71 GB of
cache, far more than the 129 MB L2, so no L2 flush is needed between steps.

Metric: eviction-step KV token-heads per second = (layers * batch * Hkv * (K+B))
per step / step time.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
  python bench.py --workload qwen3_1p7b_k2048|qwen3_8b_k4096|sweep:K:B:batch:rate [--layers L] [--variant dkv]
  python bench.py --sweep [--sweep-full]     # the Qwen3-8B-geometry grid over K, B, batch, outlier rate
  python bench.py --decode [--mixed-bits b]  # decode attention over the kept cache

The step time of `value` is taken without per-launch events; each kernel's launch time comes from a
second, profiled pass of the same steps.  `e2e` runs the step from pinned host buffers with the
host-device copies inside the timed region.

Under torchrun (N > 1) every rank runs the same per-GPU workload on its own GPU
(units are independent: no collective on the data path); value is the
whole-job rate from the maximum step time over ranks.
"""

from __future__ import annotations

import argparse
import datetime
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "eviction-step KV tokens/sec and fraction of roofline (HBM GB/s, tensor util)"
UNIT = "token-heads/s"
FALLBACK_HBM_GBS = 6800.0


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="qwen3_32b_k8192")
    ap.add_argument("--variant", choices=["attnv", "dkv"], default="attnv")
    ap.add_argument("--reserve", choices=["value", "random"], default="value",
                    help="AttnV R_V: largest value magnitude (Sec. 3.1) or uniformly random (App. C ablation)")
    ap.add_argument("--gqa", choices=["mean", "max"], default="mean",
                    help="AttnV: combine the G query heads' window scores by mean or by max")
    ap.add_argument("--dkv-shared-g", action="store_true", help="DKV: one projection per round for every unit")
    ap.add_argument("--mixed-bits", type=int, default=0, choices=[0, 2, 4, 8],
                    help="with --decode: read the unreserved values from b-bit codes (Sec. 4.4 / Sec. 6)")
    ap.add_argument("--value-bits", type=int, default=0, choices=[0, 2, 4, 8],
                    help="AttnV: keep the values in the compressed value store (b-bit codes, bf16 reserved ring)")
    ap.add_argument("--layers", type=int, default=None, help="run only this many layers of the workload")
    ap.add_argument("--e2e-steps", type=int, default=None, help="steps of the host-buffer end-to-end pass")
    ap.add_argument("--cpu-seconds", type=float, default=15.0, help="budget of the oracle CPU baseline")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the records of the other configurations (single layer, Qwen3-1.7B, Qwen3-8B both "
                         "variants, the sweep's K 16384 point)")
    ap.add_argument("--sweep", action="store_true",
                    help="the Qwen3-8B-geometry sweep over K, B, batch and value-outlier rate (one JSON line, a point each)")
    ap.add_argument("--sweep-full", action="store_true", help="with --sweep: every point of the 5 x 3 x 4 x 3 grid")
    ap.add_argument("--sweep-gb", type=float, default=48.0,
                    help="with --sweep: cache bytes (GB) a point may hold; the layers beyond it are left out")
    ap.add_argument("--decode", action="store_true",
                    help="time the decode-step attention over every layer's kept cache instead of the eviction step")
    return ap.parse_args()


# ---------------------------------------------------------------------------------------------- helpers

def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), float(d.get("bf16_tflops", 1900.0)), "measured"
    return FALLBACK_HBM_GBS, 1900.0, "fallback"


class ClockSampler:
    """nvidia-smi clock / throttle-reason samples taken while the timed region runs."""

    FIELDS = ["timestamp", "index", "clocks.sm", "clocks.max.sm", "power.draw", "clocks_event_reasons.active",
              "clocks_event_reasons.hw_slowdown", "clocks_event_reasons.hw_thermal_slowdown",
              "clocks_event_reasons.sw_thermal_slowdown", "clocks_event_reasons.sw_power_cap"]

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.file = None
        self.t_begin = 0.0

    def _rows(self):
        with open(self.file.name) as f:
            return [r for r in f.read().splitlines() if r.strip()]

    def start(self):
        """Starts nvidia-smi and returns once its first sample is written (at most 5 s), so that its start-up
        falls before the timed region, which the caller begins next."""
        try:
            self.file = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", "--query-gpu=" + ",".join(self.FIELDS),
                 "--format=csv,noheader,nounits", "-lms", "20"], stdout=self.file, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
            return
        t0 = time.time()
        while time.time() - t0 < 5.0 and self.proc.poll() is None and not self._rows():
            time.sleep(0.01)
        self.t_begin = time.time()

    def stop(self):
        """Ends sampling (the caller has just ended the timed region); summarises the samples stamped inside it."""
        if self.proc is None:
            return None
        t_end = time.time()
        time.sleep(0.06)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.file.flush()
        self.file.seek(0)
        rows = [r.split(",") for r in self.file.read().strip().splitlines() if r.strip()]
        self.file.close()
        os.unlink(self.file.name)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        parsed = []  # (time stamp or None, fields)
        for r in rows:
            r = [x.strip() for x in r]
            if len(r) < 10:
                continue
            try:
                t = datetime.datetime.strptime(r[0], "%Y/%m/%d %H:%M:%S.%f").timestamp()
            except ValueError:
                t = None
            parsed.append((t, r))
        bracketed = False
        if any(t is not None for t, _ in parsed):  # else (an unknown stamp format) every sample is kept
            stamped = [(t, r) for t, r in parsed if t is not None]
            inside = [(t, r) for t, r in stamped if self.t_begin - 0.01 <= t <= t_end + 0.01]
            if not inside:
                # a region shorter than the sampling interval: the last sample before it and the first after it
                before = [x for x in stamped if x[0] < self.t_begin]
                after = [x for x in stamped if x[0] > t_end]
                inside = ([max(before, key=lambda x: x[0])] if before else []) + \
                         ([min(after, key=lambda x: x[0])] if after else [])
                bracketed = bool(inside)
            parsed = inside
        for _, r in parsed:
            try:
                sm.append(float(r[2]))
                mx.append(float(r[3]))
            except ValueError:
                continue
            for name, val in zip(names, r[6:10]):
                if val.lower() in ("active", "1"):
                    reasons.add(name)
        if not sm:
            return None
        out = {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons), "samples": len(sm)}
        if bracketed:
            out["bracketing"] = True
        return out


def max_over_ranks(ms, world, device):
    """The slowest rank's time: every rank's step time, reduced by MAX over the process group (any backend)."""
    if world <= 1:
        return ms
    import torch
    import torch.distributed as dist
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_rank, world, ms):
    """Units processed by all ranks (the same per-rank work: weak scaling) per second of the slowest rank."""
    return world * units_per_rank / (ms / 1e3)


def kernel_bytes(kind, wl, variant, moved_rows_per_unit, bits=0):
    """Algorithmic bytes of one kernel for one layer (a launch covers up to 64 layers); bits > 0: with the
    compressed value store, whose values move in the store kernels instead of the gather."""
    U = wl.batch * wl.num_kv_heads
    N, K, B, d = wl.slots, wl.budget_k, wl.buffer_b, wl.head_dim
    row = 2 * d
    if bits and kind == "select_compact":  # only the key rows move here
        return U * (N * 4 + K * 4 + K * 4 + K * 4 + K) + U * moved_rows_per_unit * (2 * row + 8)
    if kind == "store_append":  # the B value rows in and into the ring, the unit's masks and ring state
        return U * (2 * B * row + 2 * 4 * ((N + 31) // 32) + 16)
    if kind == "store_evict":
        # the kept list and flags, the masks; every kept slot's codes and (s, z) read and written; the reserved
        # rows (N_v + B after the eviction) read and written
        nv = K // 4  # the default N_v the bench runs with
        return U * (K * 5 + 2 * 4 * ((N + 31) // 32) + 2 * K * (d * bits // 8 + 8) + 2 * (nv + B) * row)
    if kind == "score_attn":
        return U * (N * row + wl.window_rows * row + N * 4)
    if kind == "value_score":
        return U * (K * row + K * 4)
    if kind == "dkv_score":
        return U * (2 * K * row + K * 4)
    if kind == "select_compact":
        # scores, magnitudes and positions in; kept list, positions, magnitudes and the moved K/V rows out
        return U * (N * 4 + K * 4 + K * 4 + K * 4) + U * moved_rows_per_unit * (2 * 2 * row + 8)
    if kind == "evict_small":  # window score, selection and gather of one unit in one launch
        return kernel_bytes("score_attn", wl, variant, moved_rows_per_unit) + \
            kernel_bytes("select_compact", wl, variant, moved_rows_per_unit)
    if kind == "append":
        # k and v rows of the B steps in and out, the query rows of the last W steps in and out (earlier
        # queries never reach the window ring), positions and value magnitudes out
        return 2 * (2 * B * U + min(wl.window, B) * wl.batch * wl.num_q_heads) * row + 2 * B * U * 4
    return 0


def step_bytes(wl, variant):
    """Algorithmic bytes of one layer-round of the whole step: read K and V (all N rows), write the K kept
    rows, read the window queries (AttnV)."""
    U = wl.batch * wl.num_kv_heads
    d = wl.head_dim
    q = 2 * d * wl.window_rows if variant == "attnv" else 0
    return U * (4 * d * wl.slots + 4 * d * wl.budget_k + q)


# ---------------------------------------------------------------------------------------------- oracle legs

_WORKER = {}


def _oracle_worker_init(name, variant, units, layer, rnd):
    """Pool initializer: draws the sampled unit states once, so the jobs time only the oracle."""
    from paper_2606_03928_gb300 import workloads as Wm
    wl = Wm.WORKLOADS[name]
    _WORKER.update(wl=wl, variant=variant, layer=layer, rnd=rnd, units=units,
                   states=[Wm.unit_state(wl, 0, layer, s, h, rnd) for (s, h) in units])


def _oracle_job(i):
    from oracle import vase_oracle as O
    wl, st = _WORKER["wl"], _WORKER["states"][i]
    s, h = _WORKER["units"][i]
    O.evict_unit_bits(st["q_bits"].reshape(-1, wl.head_dim), st["k_bits"], st["v_bits"], st["positions"],
                      budget_k=wl.budget_k, buffer_b=wl.buffer_b, variant=_WORKER["variant"], seed=0,
                      layer=_WORKER["layer"], seq=s, head=h, num_kv_heads=wl.num_kv_heads, rnd=_WORKER["rnd"])
    return wl.slots


def oracle_pool(wl, variant, max_units=64, layer=0, rnd=5):
    """A spawn pool with one single-threaded oracle worker per host core, each holding the sampled units."""
    import multiprocessing as mp
    for var in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        os.environ[var] = "1"
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    units = [(s, h) for s in range(wl.batch) for h in range(wl.num_kv_heads)][:max_units]
    pool = mp.get_context("spawn").Pool(cores, initializer=_oracle_worker_init,
                                        initargs=(wl.name, variant, units, layer, rnd))
    pool.map(_oracle_job, range(min(len(units), cores)))  # warm the workers
    return pool, cores, len(units)


def oracle_throughput(pool, n_units, wl, seconds):
    """Evicts the sampled units with the oracle on all host cores for about `seconds`; token-heads/s."""
    done = 0
    t0 = time.perf_counter()
    while True:
        done += len(pool.map(_oracle_job, range(n_units)))
        if time.perf_counter() - t0 >= seconds:
            break
    wall = time.perf_counter() - t0
    return done * wl.slots / wall, done, wall


# ---------------------------------------------------------------------------------------------- reference arm

def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    from paper_2606_03928_gb300 import workloads as Wm
    wl = Wm.WORKLOADS[args.workload]
    # one step = the oracle over one layer-round of the workload (all its units, at most 64)
    pool, cores, per_step = oracle_pool(wl, args.variant)
    units = wl.batch * wl.num_kv_heads

    def step(r):
        pool.map(_oracle_job, range(per_step))

    for r in range(args.warmup):
        step(r)
    t0 = time.perf_counter()
    for r in range(args.steps):
        step(r)
    wall = time.perf_counter() - t0
    pool.close()
    value = args.steps * per_step * wl.slots / wall
    sample = f"{per_step} of the {units} units of one layer-round per step (fp64 numpy oracle, spawn pool)"
    out = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * wall / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": wl.name, "variant": args.variant, "global_batch": wl.batch, "seq_len": wl.slots,
                   "parallelism": "host cores"},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(out))
    return 0


# ---------------------------------------------------------------------------------------------- our arm

def gen_stream(wl, n_tokens, gen, device, torch):
    """Seeded synthetic decode tokens of one layer: q [n, b, Hq, d], k/v [n, b, Hkv, d] in bf16.

    Keys and queries N(0, 1) (channel outliers x8 where the workload has them), values N(0, 1) with a
    fraction of rows scaled (x20, or log-uniform x10..x50)."""
    b, Hq, Hkv, d = wl.batch, wl.num_q_heads, wl.num_kv_heads, wl.head_dim
    q = torch.randn((n_tokens, b, Hq, d), generator=gen, device=device)
    k = torch.randn((n_tokens, b, Hkv, d), generator=gen, device=device)
    v = torch.randn((n_tokens, b, Hkv, d), generator=gen, device=device)
    if wl.key_channel_outliers or wl.query_channel_outliers:
        ch = torch.randperm(d, generator=torch.Generator().manual_seed(1234))[:wl.outlier_channels].to(device)
        if wl.key_channel_outliers:
            k[..., ch] *= wl.channel_scale
        if wl.query_channel_outliers:
            q[..., ch] *= wl.channel_scale
    rows = torch.rand((n_tokens, b, Hkv, 1), generator=gen, device=device) < wl.value_outlier_rate
    lo, hi = wl.value_outlier_scale
    if hi > lo:
        u = torch.rand((n_tokens, b, Hkv, 1), generator=gen, device=device)
        scale = torch.exp(u * (torch.log(torch.tensor(hi)) - torch.log(torch.tensor(lo))) + torch.log(torch.tensor(lo)))
    else:
        scale = torch.full((n_tokens, b, Hkv, 1), lo, device=device)
    v = torch.where(rows, v * scale, v)
    return q.to(torch.bfloat16), k.to(torch.bfloat16), v.to(torch.bfloat16)


class Rig:
    """One workload's context, its prefilled caches and a few distinct rounds of new decode tokens, resident
    in HBM.  A round holds, per layer, the B new key and value rows and the query rows of the last W steps
    (the only query rows the append reads: the window ring keeps no others)."""

    def __init__(self, wl, variant, device, seed, torch, V, n_distinct=4, **cache_kw):
        self.wl, self.torch, self.V = wl, torch, V
        L, K, Bf = wl.num_layers, wl.budget_k, wl.buffer_b
        self.cache = V.VaseCache(V.Geometry(K, Bf, wl.window, wl.num_q_heads, wl.num_kv_heads, L, wl.batch),
                                 variant=variant, seed=0, device=device, **cache_kw)
        gen = torch.Generator(device=device)
        gen.manual_seed(seed)
        for layer in range(L):  # prefill: K tokens per layer, in pieces of at most 1024 (bounded temporaries)
            for t0 in range(0, K, 1024):
                self.cache.append(layer, *gen_stream(wl, min(1024, K - t0), gen, device, torch))
        self.w_q = min(wl.window, Bf)
        self.rounds = []
        for _ in range(max(1, min(n_distinct, wl.rounds_per_layer))):
            qs, ks, vs = [], [], []
            for layer in range(L):
                q, k, v = gen_stream(wl, Bf, gen, device, torch)
                qs.append(q[Bf - self.w_q:].contiguous())
                ks.append(k)
                vs.append(v)
                del q
            self.rounds.append((torch.stack(qs), torch.stack(ks), torch.stack(vs)))
            del qs, ks, vs
        torch.cuda.synchronize()
        self.r = 0
        self.q_step = wl.batch * wl.num_q_heads * wl.head_dim * 2  # bytes of one step's query rows

    def step(self, stream):
        """One step: the next round's B tokens appended to every layer, then every layer evicted, through the
        library's one-step call (one launch for both where the fused small-unit kernel takes the eviction, else
        the append's launch and the eviction's).  Layer l's query pointer sits B - W steps before its tail,
        which the library never reads."""
        q, k, v = self.rounds[self.r % len(self.rounds)]
        self.r += 1
        Bf = self.wl.buffer_b
        return self.V.vase_append_evict_all(self.cache.ctx, q.data_ptr() - (Bf - self.w_q) * self.q_step,
                                            k.data_ptr(), v.data_ptr(), Bf, q[0].numel() * 2, k[0].numel() * 2,
                                            stream)

    def close(self):
        self.cache.close()
        del self.cache, self.rounds


def timed_steps(torch, step, steps, stream, barrier=lambda: None, sampler=None):
    """Mean ms per step of `steps` calls of step(), CUDA events on the launch stream, synchronised and
    bracketed by the barrier on both sides."""
    barrier()
    torch.cuda.synchronize()
    if sampler is not None:
        sampler.start()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(steps):
        step()
    e1.record(stream)
    torch.cuda.synchronize()
    barrier()
    clocks = sampler.stop() if sampler is not None else None
    return e0.elapsed_time(e1) / steps, clocks


def kernel_table(kernels, wl, variant, moved, layers_per_launch, hbm_peak, tflops_peak, bits=0):
    """Per kernel: launches, mean launch time, share of the kernel time, algorithmic GB/s; for the window
    score also its algorithmic QK^T TFLOP/s and the bound of its own roofline."""
    out = {}
    total = sum(v[0] for v in kernels.values()) or 1.0
    # the one-step call runs the append inside the fused small-unit kernel where that kernel takes the eviction
    fused_append = kernels.get("append", (0.0, 0))[1] == 0 and kernels.get("evict_small", (0.0, 0))[1] > 0
    for name, (kms, n) in kernels.items():
        if n == 0:
            continue
        per_launch = kms / n
        b = kernel_bytes(name, wl, variant, moved, bits) * layers_per_launch
        if name == "evict_small" and fused_append:
            b += kernel_bytes("append", wl, variant, moved, bits) * layers_per_launch
        rec = {"launches": n, "us_per_launch": round(1e3 * per_launch, 3), "share": round(kms / total, 4),
               "gbs": round(b / (per_launch / 1e3) / 1e9, 1)}
        if name == "score_attn":
            f = score_flops(wl) * layers_per_launch
            rec["qkt_tflops"] = round(f / (per_launch / 1e3) / 1e12, 1)
            rec["bound"] = "tensor" if f / (tflops_peak * 1e12) > b / (hbm_peak * 1e9) else "hbm"
        out[name] = rec
    return out


def score_flops(wl):
    """Algorithmic FLOPs of the window score of one layer: one QK^T over the unit's G*W window rows and its
    N keys, 2 * G*W * N * d per unit (the kernel's second, transposed product is not counted)."""
    return wl.batch * wl.num_kv_heads * 2 * wl.window_rows * wl.slots * wl.head_dim


def roofline_of(kernels_tab, dom, wl, variant, moved, layers_per_launch, hbm_peak, tflops_peak, peak_kind, traffic,
                bits=0):
    rec = kernels_tab[dom]
    if rec.get("bound") == "tensor":
        f = score_flops(wl) * layers_per_launch
        return {"bound": "tensor", "achieved": rec["qkt_tflops"], "peak": tflops_peak, "unit": "TFLOP/s",
                "frac": round(rec["qkt_tflops"] / tflops_peak, 4), "traffic": traffic, "kernel": dom,
                "algorithmic_flops_per_launch": f, "peak_source": peak_kind + " bf16 burst"}
    b = kernel_bytes(dom, wl, variant, moved, bits) * layers_per_launch
    return {"bound": "hbm", "achieved": rec["gbs"], "peak": hbm_peak, "unit": "GB/s",
            "frac": round(rec["gbs"] / hbm_peak, 4), "traffic": traffic, "kernel": dom,
            "algorithmic_bytes_per_launch": b, "peak_source": peak_kind}


def moved_rows(cache, torch):
    """Rows per unit whose slot changed in the last eviction (layer slot 0 of the last call)."""
    src = cache.debug_view(0)["src"].cpu()
    K = src.shape[-1]
    return float((src != torch.arange(K, dtype=torch.int32)).sum().item()) / src.shape[0]


def profiled_kernels(torch, rig, steps, stream):
    """The same steps again with a CUDA event pair around every launch (the library's profiling mode)."""
    rig.cache.profile_enable(True)
    ms, _ = timed_steps(torch, lambda: rig.step(stream), steps, stream)
    rig.cache.profile_enable(False)
    return rig.cache.profile_collect(), ms


def traffic_of(dom, wl, variant, L):
    """ncu DRAM bytes per launch of the dominant kernel, when a capture of these exact sources exists."""
    tpath = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(tpath):
        return None
    try:
        from paper_2606_03928_gb300.build import kernel_digest
        with open(tpath) as f:
            tr = json.load(f)
        ent = tr.get(f"{dom}:{wl.name}:{variant}:{L}")
        if ent and ent.get("kernel_digest") == kernel_digest(dom):
            return ent["bytes_per_launch"]
    except Exception:
        return None
    return None


def score_ncu(wl):
    """Tensor-pipe utilisation of the window-score kernel from its committed ncu capture at this workload, when
    that capture was taken on the current sources (profiles/score_ncu.json)."""
    path = os.path.join(ROOT, "profiles", "score_ncu.json")
    if not os.path.exists(path):
        return None
    try:
        from paper_2606_03928_gb300.build import kernel_digest
        with open(path) as f:
            d = json.load(f)
        ent = d.get(wl.name)
        if ent and ent.get("kernel_digest") == kernel_digest("score_attn"):
            return {k: v for k, v in ent.items() if k != "kernel_digest"}
    except Exception:
        return None
    return None


# the other configurations measured in the same run, each as a record of the JSON line: the single-layer case,
# the Qwen3-1.7B and Qwen3-8B geometries (both scoring variants) and the sweep's largest budget
EXTRA_CONFIGS = [("single_layer_k256", "attnv", None, {}), ("qwen3_1p7b_k2048", "attnv", None, {"decode": True}),
                 ("qwen3_1p7b_k2048", "attnv", None, {"value_bits": 4, "decode": True}),
                 ("qwen3_8b_k4096", "attnv", None, {}), ("qwen3_8b_k4096", "dkv", None, {}),
                 ("sweep:16384:128:32:0.005", "attnv", 21, {})]


def decode_step_ms(torch, V, cache, wl, device, steps, warmup):
    """ms of one decode step's attention over every layer's cache (vase_decode_attention per layer, captured in a
    CUDA graph and replayed, as a serving loop runs it)."""
    L = wl.num_layers
    gen = torch.Generator(device=device)
    gen.manual_seed(7)
    q = torch.randn((L, wl.batch, wl.num_q_heads, wl.head_dim), generator=gen, device=device).to(torch.bfloat16)
    out = torch.empty((L, wl.batch, wl.num_q_heads, wl.head_dim), dtype=torch.float32, device=device)
    ptrs = [(q[l].data_ptr(), out[l].data_ptr()) for l in range(L)]

    def step():
        sh = torch.cuda.current_stream()
        for l in range(L):
            V.vase_decode_attention(cache.ctx, l, ptrs[l][0], ptrs[l][1], sh)

    step()
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        step()
    for _ in range(warmup):
        graph.replay()
    stream = torch.cuda.current_stream()
    ms, _ = timed_steps(torch, graph.replay, steps, stream)
    st, code = cache.check_device_error()
    if st != 0:
        raise RuntimeError(f"device error in the decode steps: {code:#x}")
    return ms


def workload_by_name(Wm, name, layers=None):
    if name.startswith("sweep:"):
        _, K, Bf, b, rate = name.split(":")
        wl = Wm.sweep_point(int(K), int(Bf), int(b), float(rate))
    else:
        wl = Wm.WORKLOADS[name]
    if layers:
        wl = Wm.shrink(wl, num_layers=min(layers, wl.num_layers))
    return wl


def measure_config(torch, V, Wm, name, variant, layers, steps, warmup, device, hbm_peak, tflops_peak,
                   cache_kw=None):
    wl = workload_by_name(Wm, name, layers)
    cache_kw = dict(cache_kw or {})
    with_decode = cache_kw.pop("decode", False)
    bits = cache_kw.get("value_bits", 0)
    rig = Rig(wl, variant, device, 1000, torch, V, **cache_kw)
    stream = torch.cuda.current_stream()
    for _ in range(warmup):
        rig.step(stream)
    ms, clocks = timed_steps(torch, lambda: rig.step(stream), steps, stream, sampler=ClockSampler(0))
    kernels, _ = profiled_kernels(torch, rig, steps, stream)
    st, code = rig.cache.check_device_error()
    if st != 0:
        raise RuntimeError(f"device error in {name}: {code:#x}")
    L = wl.num_layers
    moved = moved_rows(rig.cache, torch)
    tab = kernel_table(kernels, wl, variant, moved, min(L, 64), hbm_peak, tflops_peak, bits)
    roof_ms = L * step_bytes(wl, variant) / (hbm_peak * 1e9) * 1e3
    extra = {}
    if bits:  # the compressed value store: its V buffer against the bf16 cache
        sizes = V.vase_get_buffer_sizes(rig.cache.cfg)
        bf_bytes = L * wl.batch * wl.num_kv_heads * wl.slots * 2 * wl.head_dim
        extra = {"value_bits": bits, "v_bytes": sizes.v_cache, "v_bytes_bf16": bf_bytes,
                 "v_bytes_ratio": round(sizes.v_cache / bf_bytes, 4)}
    if with_decode:  # the decode step that reads the cache the eviction leaves (the store, with value_bits)
        extra["decode_ms_per_step"] = round(decode_step_ms(torch, V, rig.cache, wl, device, steps, warmup), 4)
    rig.close()
    torch.cuda.empty_cache()
    return {"workload": wl.name, "variant": variant, **extra, "layers": L, "batch": wl.batch, "budget_k": wl.budget_k,
            "buffer_b": wl.buffer_b, "window": wl.window, "heads": f"{wl.num_q_heads}/{wl.num_kv_heads}",
            "steps": steps, "ms_per_step": round(ms, 4),
            "token_heads_per_s": L * wl.batch * wl.num_kv_heads * wl.slots / (ms / 1e3),
            "step_roofline_ms": round(roof_ms, 4), "step_roofline_frac": round(roof_ms / ms, 4),
            "kernels": tab, "clocks": clocks}


def run_ours(args):
    import torch
    import torch.distributed as dist

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    else:
        torch.cuda.set_device(0)
    device = torch.device("cuda", torch.cuda.current_device())

    # the oracle pool is started before the first CUDA work of this process
    from paper_2606_03928_gb300 import workloads as Wm
    wl = workload_by_name(Wm, args.workload, args.layers)
    pool = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        pool, cores, n_units = oracle_pool(wl, args.variant)

    from paper_2606_03928_gb300 import build as B
    B.build()
    from paper_2606_03928_gb300 import vase as V

    hbm_peak, tflops_peak, peak_kind = measured_peaks()
    L, K, Bf = wl.num_layers, wl.budget_k, wl.buffer_b
    rig = Rig(wl, args.variant, device, 1000 + rank, torch, V, reserve=args.reserve, gqa=args.gqa,
              dkv_shared_g=args.dkv_shared_g, value_bits=args.value_bits)
    cache = rig.cache
    stream = torch.cuda.current_stream()

    def barrier():
        if world > 1:
            dist.barrier()

    for _ in range(args.warmup):
        rig.step(stream)
    st, code = cache.check_device_error()
    if st != 0:
        raise RuntimeError(f"device error during warm-up: {code:#x}")

    launches0 = cache.launch_count()
    ms, clocks = timed_steps(torch, lambda: rig.step(stream), args.steps, stream, barrier,
                             ClockSampler(local if world > 1 else 0))
    launches = cache.launch_count() - launches0
    # each kernel's launch duration: the same K steps again with a CUDA event pair around every launch (the
    # library's profiling mode); the step time above is taken without those events
    kernels, profiled_ms = profiled_kernels(torch, rig, args.steps, stream)
    st, code = cache.check_device_error()
    if st != 0:
        raise RuntimeError(f"device error in the timed region: {code:#x}")
    ms = max_over_ranks(ms, world, device)
    token_heads = L * wl.batch * wl.num_kv_heads * wl.slots
    value = whole_job_rate(token_heads, world, ms)
    moved = moved_rows(cache, torch)

    # ---- end to end through the C ABI from host buffers: every step's inputs cross from pinned host memory
    # (vase_stage_host_inputs on a copy stream, the next step's copies issued before this step's kernels),
    # are appended from the staging buffer (vase_append_all_staged), and every layer's kept positions come
    # back to pinned host memory (vase_read_positions_all); all of it inside the timed region
    e2e_steps = args.e2e_steps if args.e2e_steps is not None else max(1, min(args.steps, 20))
    host_rounds = [tuple(t.cpu().pin_memory() for t in r) for r in rig.rounds]
    staging = cache.host_staging(Bf)
    copy_stream = torch.cuda.Stream(device=device)
    pos_host = torch.empty((L, wl.batch, wl.num_kv_heads, K), dtype=torch.int32).pin_memory()
    q0, k0, v0 = host_rounds[0]
    h2d = sum(t.numel() * t.element_size() for t in (q0, k0, v0))
    d2h = pos_host.numel() * pos_host.element_size()
    Wq, q_step = rig.w_q, rig.q_step

    def stage(r):
        q, k, v = host_rounds[r % len(host_rounds)]
        V.vase_stage_host_inputs(cache.ctx, q.data_ptr() - (Bf - Wq) * q_step, k.data_ptr(), v.data_ptr(), Bf,
                                 q[0].numel() * 2, k[0].numel() * 2, staging.data_ptr(), staging.numel(),
                                 copy_stream)

    def e2e_run(n):
        stage(0)
        for r in range(n):
            if r + 1 < n:
                stage(r + 1)
            cache.append_all_staged(stream)
            cache.evict_all(stream)
            cache.read_positions_all(pos_host, copy_stream, stream)
        stream.wait_stream(copy_stream)  # the last read-back ends inside the timed region

    e2e_run(2)  # warm-up of the host path
    e2e_total, _ = timed_steps(torch, lambda: e2e_run(e2e_steps), 1, stream, barrier)
    e2e_ms = max_over_ranks(e2e_total / e2e_steps, world, device)
    e2e_value = whole_job_rate(token_heads, world, e2e_ms)
    st, code = cache.check_device_error()
    if st != 0:
        raise RuntimeError(f"device error in the end-to-end steps: {code:#x}")

    # ---- roofline of the dominant kernel
    layers_per_launch = min(L, 64)
    tab = kernel_table(kernels, wl, args.variant, moved, layers_per_launch, hbm_peak, tflops_peak, args.value_bits)
    dom = max(tab, key=lambda k: tab[k]["share"])
    roofline = roofline_of(tab, dom, wl, args.variant, moved, layers_per_launch, hbm_peak, tflops_peak, peak_kind,
                           None if args.value_bits else traffic_of(dom, wl, args.variant, L), args.value_bits)
    step_roof_ms = L * step_bytes(wl, args.variant) / (hbm_peak * 1e9) * 1e3
    evict_ms = sum(kernels[k][0] for k in kernels if k != "append") / args.steps
    rig.close()
    del staging, host_rounds
    torch.cuda.empty_cache()

    out = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": wl.name, "variant": args.variant, **variant_options(args), "layers": L,
                   "global_batch": wl.batch * world,
                   "seq_len": wl.slots, "budget_k": K, "buffer_b": Bf, "window": wl.window,
                   "heads": f"{wl.num_q_heads}/{wl.num_kv_heads}", "parallelism": f"dp{world}",
                   "l2": f"inputs larger than L2 (about {L * step_bytes(wl, args.variant) / 1e9:.1f} GB touched per step)"},
        "roofline": roofline,
        "step_roofline": {"ms_per_step_at_hbm_peak": round(step_roof_ms, 4),
                          "frac": round(step_roof_ms / ms, 4),
                          "amortised_us_per_decode_token": round(1e3 * evict_ms / Bf, 3)},
        "kernels": tab,
        "score_kernel_ncu": score_ncu(wl) if args.variant == "attnv" else None,
        "kernels_pass_ms_per_step": round(profiled_ms, 4),
        "clocks": clocks,
        "gpu_launches": launches,
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "ms_per_step": e2e_ms, "steps": e2e_steps,
                "form": "C ABI: vase_stage_host_inputs (pinned host -> device on a copy stream, the next step's "
                        "copies issued before this step's kernels), vase_append_all_staged, vase_evict_all, "
                        "vase_read_positions_all (every layer's kept positions to pinned host memory)"},
    }
    if rank == 0 and world == 1 and not args.no_configs:
        out["configs"] = [measure_config(torch, V, Wm, name, variant, layers, args.steps, args.warmup, device,
                                         hbm_peak, tflops_peak, kw)
                          for (name, variant, layers, kw) in EXTRA_CONFIGS]
    if pool is not None:
        v, done, wall = oracle_throughput(pool, n_units, wl, args.cpu_seconds)
        pool.close()
        out["cpu_baseline"] = {"value": v, "unit": UNIT, "cores": cores, "kind": "oracle",
                               "sample": f"{done} units of one layer-round ({wall:.1f} s on {cores} host cores)"}
    if rank == 0:
        print(json.dumps(out))
    if world > 1:
        dist.destroy_process_group()
    return 0


def run_decode(args):
    """One decode step's attention (Eq. (1)) over the kept cache of every layer, after an eviction round:
    vase_decode_attention per layer, reading K and V of the K kept slots of every unit once."""
    import torch

    torch.cuda.set_device(0)
    device = torch.device("cuda", 0)
    from paper_2606_03928_gb300 import workloads as Wm
    wl = Wm.WORKLOADS[args.workload]
    if args.layers:
        wl = Wm.shrink(wl, num_layers=args.layers)
    from paper_2606_03928_gb300 import build as B
    B.build()
    from paper_2606_03928_gb300 import vase as V

    L, K, Bf = wl.num_layers, wl.budget_k, wl.buffer_b
    cache = V.VaseCache(V.Geometry(K, Bf, wl.window, wl.num_q_heads, wl.num_kv_heads, L, wl.batch),
                        variant=args.variant, seed=0, device=device, value_bits=args.value_bits)
    gen = torch.Generator(device=device)
    gen.manual_seed(1000)
    for layer in range(L):
        cache.append(layer, *gen_stream(wl, K + Bf, gen, device, torch))
    cache.evict_all()  # every layer now holds its K kept pairs
    q = torch.randn((L, wl.batch, wl.num_q_heads, wl.head_dim), generator=gen, device=device).to(torch.bfloat16)
    out = torch.empty((L, wl.batch, wl.num_q_heads, wl.head_dim), dtype=torch.float32, device=device)
    bits = args.mixed_bits
    mixed = []
    if bits:  # codes of every layer's unreserved kept values (untimed: once per eviction round)
        for layer in range(L):
            mb, t = cache.mixed_buffers(bits)
            cache.quantize_values(layer, bits, mb)
            mixed.append((mb, t))
        torch.cuda.synchronize()
        reserved = sum(int(((t["rmask"] >> i) & 1).sum()) for _, t in mixed for i in range(32))  # bf16 slots

    # device pointers computed once: the step is 28 C calls, not 28 tensor views
    ptrs = [(q[layer].data_ptr(), out[layer].data_ptr()) for layer in range(L)]
    stream_handle = torch.cuda.current_stream()

    def step():
        if bits:
            for layer in range(L):
                V.vase_decode_attention_mixed(cache.ctx, layer, bits, mixed[layer][0], ptrs[layer][0], ptrs[layer][1],
                                              stream_handle)
            return
        for layer in range(L):
            V.vase_decode_attention(cache.ctx, layer, ptrs[layer][0], ptrs[layer][1], stream_handle)

    for _ in range(args.warmup):
        step()
    st, code = cache.check_device_error()
    if st != 0:
        raise RuntimeError(f"device error during warm-up: {code:#x}")
    stream = torch.cuda.current_stream()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    # eager: one C call per layer per step
    torch.cuda.synchronize()
    ev0.record(stream)
    for _ in range(args.steps):
        step()
    ev1.record(stream)
    torch.cuda.synchronize()
    eager_ms = ev0.elapsed_time(ev1) / args.steps

    # the timed form: the step's 28 launches captured once in a CUDA graph (as a serving loop runs a decode
    # step), replayed; consecutive launches overlap prologue and epilogue (programmatic dependent launch)
    graph = torch.cuda.CUDAGraph()
    launches0 = cache.launch_count()
    with torch.cuda.graph(graph):
        stream_handle = torch.cuda.current_stream()
        step()
    per_step_launches = cache.launch_count() - launches0
    stream_handle = torch.cuda.current_stream()
    for _ in range(args.warmup):
        graph.replay()
    torch.cuda.synchronize()
    sampler = ClockSampler(0)
    sampler.start()
    ev0.record(stream)
    for _ in range(args.steps):
        graph.replay()
    ev1.record(stream)
    torch.cuda.synchronize()
    clocks = sampler.stop()
    st, code = cache.check_device_error()
    if st != 0:
        raise RuntimeError(f"device error in the timed steps: {code:#x}")
    launches = per_step_launches * args.steps
    ms = ev0.elapsed_time(ev1) / args.steps
    units = wl.batch * wl.num_kv_heads
    # K and V rows of the kept slots, the query rows in, the fp32 outputs out
    step_bytes_ = L * (units * K * 2 * 2 * wl.head_dim + wl.batch * wl.num_q_heads * wl.head_dim * (2 + 4))
    mixed_info = None
    if args.value_bits:
        # compressed value store: K rows, the code rows and (s, z) of every slot, the ring rows of the bf16 slots,
        # the masks and ring state
        vb = args.value_bits
        ring_rows = sum(int(cache.value_store(l)["state"][:, 1].sum().item()) for l in range(L))
        step_bytes_ = (L * units * K * (2 * wl.head_dim + wl.head_dim * vb // 8 + 8) + ring_rows * 2 * wl.head_dim +
                       L * units * (4 * ((K + Bf + 31) // 32) + 16) +
                       L * wl.batch * wl.num_q_heads * wl.head_dim * (2 + 4))
        mixed_info = {"value_bits": vb, "store": True, "reserved_fraction": round(ring_rows / (L * units * K), 4)}
    elif bits:
        # b-bit values: K rows, bf16 V rows of the reserved slots, code rows and (s, z) of the others, the masks
        coded = L * units * K - reserved
        step_bytes_ = (L * units * K * 2 * wl.head_dim + reserved * 2 * wl.head_dim +
                       coded * (wl.head_dim * bits // 8 + 8) + L * units * ((K + 31) // 32) * 4 +
                       L * wl.batch * wl.num_q_heads * wl.head_dim * (2 + 4))
        mixed_info = {"value_bits": bits, "reserved_fraction": round(reserved / (L * units * K), 4)}
    gbs = step_bytes_ / (ms / 1e3) / 1e9
    hbm_peak, _, peak_kind = measured_peaks()
    outj = {
        "metric": ("decode-step attention over the kept cache, bytes/s (K and V of every kept slot read once)" if not bits
                   else "decode-step attention over the kept cache with b-bit unreserved values, bytes/s (K rows, "
                        "bf16 reserved V rows, codes and scales read once)"),
        "value": gbs, "unit": "GB/s", "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": ms, "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic",
        "config": {"workload": wl.name, "layers": L, "global_batch": wl.batch, "kept_slots": K, **(mixed_info or {}),
                   "heads": f"{wl.num_q_heads}/{wl.num_kv_heads}", "parallelism": "dp1",
                   "l2": f"inputs larger than L2 ({step_bytes_ / 1e9:.2f} GB read per step)"},
        "roofline": {"bound": "hbm", "achieved": round(gbs, 1), "peak": hbm_peak, "unit": "GB/s",
                     "frac": round(gbs / hbm_peak, 4), "traffic": None,
                     "kernel": ("decode_simt_kernel" if bits or args.value_bits or wl.group < 3 else "decode_tc_kernel"),
                     "algorithmic_bytes_per_launch": step_bytes_ // L, "peak_source": peak_kind},
        "clocks": clocks, "gpu_launches": launches, "timed_as": "CUDA graph replay of the step's launches",
        "eager_ms_per_step": eager_ms,
    }
    print(json.dumps(outj))
    return 0


def sweep_grid(full):
    """(K, B, batch, value-outlier rate) points of the sweep on the Qwen3-8B geometry: the whole 5 x 3 x 4 x 3
    grid, or every (K, B) pair at batch 32 and rate 0.5 % plus the batch and rate axes through K 4096, B 128."""
    Ks, Bs, bs, rates = (1024, 2048, 4096, 8192, 16384), (32, 128, 512), (1, 8, 32, 128), (0.0, 0.005, 0.02)
    if full:
        return [(K, B, b, r) for K in Ks for B in Bs for b in bs for r in rates]
    pts = [(K, B, 32, 0.005) for K in Ks for B in Bs]
    pts += [(4096, 128, b, 0.005) for b in (1, 8, 128)]
    pts += [(4096, 128, 32, r) for r in (0.0, 0.02)]
    return pts


def run_sweep(args):
    """The eviction step (append B tokens to every layer, evict every layer) at each sweep point, on as many
    of the 36 layers as fit in --sweep-gb of cache (a resident subset: all 36 at most points; the step of a
    point covers the same number of layers every time, so per-layer-round figures compare across points)."""
    import torch

    torch.cuda.set_device(0)
    device = torch.device("cuda", 0)
    from paper_2606_03928_gb300 import workloads as Wm
    from paper_2606_03928_gb300 import build as B
    B.build()
    from paper_2606_03928_gb300 import vase as V

    hbm_peak, _, peak_kind = measured_peaks()
    stream = torch.cuda.current_stream()
    points = []
    launches = 0
    for (K, Bf, b, rate) in sweep_grid(args.sweep_full):
        wl = Wm.sweep_point(K, Bf, b, rate)
        units = wl.batch * wl.num_kv_heads
        per_layer = units * wl.slots * (2 * 2 * wl.head_dim + 8) + wl.batch * wl.num_q_heads * wl.window * 2 * wl.head_dim
        L = max(1, min(wl.num_layers, int(args.sweep_gb * 1e9 // per_layer)))
        wl = Wm.shrink(wl, num_layers=L)
        cache = V.VaseCache(V.Geometry(K, Bf, wl.window, wl.num_q_heads, wl.num_kv_heads, L, wl.batch),
                            variant="attnv", seed=0, device=device)
        gen = torch.Generator(device=device)
        gen.manual_seed(1000)
        for layer in range(L):  # prefill in pieces of at most 1024 tokens (bounded generator temporaries)
            for t0 in range(0, K, 1024):
                cache.append(layer, *gen_stream(wl, min(1024, K - t0), gen, device, torch))
        per_layer_new = [gen_stream(wl, Bf, gen, device, torch) for _ in range(L)]
        chunk = tuple(torch.stack([pl[i] for pl in per_layer_new]) for i in range(3))
        del per_layer_new

        def step():
            cache.append_all(*chunk)
            cache.evict_all()

        for _ in range(3):
            step()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        step()
        e1.record(stream)
        torch.cuda.synchronize()
        n_steps = max(5, min(100, int(100.0 / max(e0.elapsed_time(e1), 1e-3))))  # about 0.1 s of steps
        sampler = ClockSampler(0)
        sampler.start()
        l0 = cache.launch_count()
        e0.record(stream)
        for _ in range(n_steps):
            step()
        e1.record(stream)
        torch.cuda.synchronize()
        clocks = sampler.stop()
        launches += cache.launch_count() - l0
        st, code = cache.check_device_error()
        if st != 0:
            raise RuntimeError(f"device error at sweep point K={K} B={Bf} b={b} rate={rate}: {code:#x}")
        ms = e0.elapsed_time(e1) / n_steps
        # the same steps again with an event pair around every launch, for each kernel's duration
        cache.profile_enable(True)
        for _ in range(n_steps):
            step()
        torch.cuda.synchronize()
        cache.profile_enable(False)
        kern = {name: round(1e3 * kms / n, 1) for name, (kms, n) in cache.profile_collect().items() if n}
        roof_ms = L * step_bytes(wl, "attnv") / (hbm_peak * 1e9) * 1e3
        points.append({"budget_k": K, "buffer_b": Bf, "batch": b, "value_outlier_rate": rate, "layers": L,
                       "steps": n_steps, "ms_per_step": round(ms, 4),
                       "token_heads_per_s": L * units * wl.slots / (ms / 1e3),
                       "sequence_tokens_per_s": L * wl.batch * wl.slots / (ms / 1e3),
                       "step_roofline_ms": round(roof_ms, 4), "roofline_frac": round(roof_ms / ms, 4),
                       # the whole step (B appends + the eviction) of these L layers over the B decode steps it serves
                       "step_us_per_decode_token": round(1e3 * ms / Bf, 3), "kernels_us_per_launch": kern,
                       "clocks": clocks})
        del cache, chunk
        torch.cuda.empty_cache()
    ref = next(p for p in points if (p["budget_k"], p["buffer_b"], p["batch"], p["value_outlier_rate"]) ==
               (4096, 128, 32, 0.005))
    outj = {"metric": METRIC + " over the Qwen3-8B-geometry sweep", "value": ref["token_heads_per_s"], "unit": UNIT,
            "n_gpus": 1, "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic", "value_at": "K 4096, B 128, batch 32, 0.5 % outliers",
            "config": {"workload": "qwen3_8b_sweep", "heads": "32/8", "window": 32, "variant": "attnv",
                       "grid": "full" if args.sweep_full else "axes", "cache_gb_per_point": args.sweep_gb,
                       "parallelism": "dp1"},
            "peak": hbm_peak, "peak_source": peak_kind, "gpu_launches": launches, "points": points}
    print(json.dumps(outj))
    return 0


def variant_options(args):
    """The non-default variant switches of a run, for the config object of its JSON line."""
    opts = {}
    if args.reserve != "value":
        opts["reserve"] = args.reserve
    if args.gqa != "mean":
        opts["gqa"] = args.gqa
    if args.dkv_shared_g:
        opts["dkv_shared_g"] = True
    if args.value_bits:
        opts["value_bits"] = args.value_bits
    return opts


def main():
    args = parse_args()
    if args.impl == "reference":
        return run_reference(args)
    if args.sweep:
        return run_sweep(args)
    if args.decode:
        return run_decode(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
