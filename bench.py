"""Benchmark of the cached-reference joint attention on one GB300 (or N replicas).

One timed step = one layer's whole hot path for one generation of the
1024x1024, five-reference edit: refcache_build (cache write + [ST; R] prefill)
followed by T = 40 step_attention calls with fresh live Q/K/V each denoising
step (four live input sets cycled, so every step streams more than the 129 MB
L2: 252 MB of cache plus 85 MB of live Q/K/V).  `value` is the unmasked
TFLOP/s of that step (4 d FLOPs per visible (query, key) pair per head).

Also reported: the step-attention kernel alone (ms per call, TFLOP/s, its
roofline against the measured bf16 peak), the prefill alone, the
full-attention recompute on the same kernel, the measured and modelled
40-step speedups, an end-to-end number through the C ABI with host buffers,
SM clocks sampled during the timed region, and the CPU oracle timed on a
bounded sample (the reported CPU baseline).

`--impl reference` times the CPU oracle instead (this workload has no other
reference implementation), on bounded samples of the same workload.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "cached-ref attention TFLOP/s & ms/step (5 refs,1024²); modelled 40-step speedup"
UNIT = "TFLOP/s"
T_STEPS = 40
N_LIVE_SETS = 4
# ncu record of DRAM bytes per step-attention launch (1024^2, 5 references),
# valid only for the kernel sources it was taken with
TRAFFIC_RECORD = os.path.join(ROOT, "profiles", "attn_tc2_kernel_step_edit1024_5ref_traffic.txt")
KERNEL_SOURCES = ("attn_tc2.cuh", "attn_tc.cuh", "common.cuh", "ptx.cuh")


def kernel_source_hash() -> str:
    import hashlib

    h = hashlib.sha256()
    for name in KERNEL_SOURCES:
        with open(os.path.join(ROOT, "paper_2608_21229_gb300", "csrc", name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()


def recorded_traffic(workload: str, kernel: str):
    """DRAM bytes per launch from the committed ncu record, or None when the
    record is missing, is for another workload or kernel, or predates the
    current kernel sources."""
    if workload != "edit1024_5ref" or kernel != "tcgen05" or not os.path.exists(TRAFFIC_RECORD):
        return None
    fields = {}
    with open(TRAFFIC_RECORD) as f:
        for line in f:
            if ":" in line and not line.startswith((" ", "#", "|")):
                k, v = line.split(":", 1)
                fields[k.strip()] = v.strip()
    if fields.get("kernel_source_sha256") != kernel_source_hash():
        return None
    try:
        return float(fields["dram_bytes_per_launch"])
    except (KeyError, ValueError):
        return None


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return {"bf16_burst": float(p["bf16_tflops"]), "bf16_sustained": float(p["bf16_tflops_sustained"]),
                "hbm_gbs": float(p["hbm_gbs"]), "source": "measured"}
    except Exception:
        return {"bf16_burst": 1900.0, "bf16_sustained": 1700.0, "hbm_gbs": 6800.0, "source": "fallback"}


class ClockSampler:
    """nvidia-smi clock / throttle-reason samples while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.tmp = None

    def __enter__(self):
        try:
            self.tmp = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=self.tmp, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
            return self
        # nvidia-smi's start-up holds up kernel launches for a few milliseconds:
        # let it write its first sample before the timed region begins
        t_end = time.monotonic() + 5.0
        while time.monotonic() < t_end and self.proc.poll() is None and os.path.getsize(self.tmp.name) == 0:
            time.sleep(0.01)
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
        return False

    def summary(self):
        if self.proc is None or self.tmp is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.tmp.flush()
        rows = []
        with open(self.tmp.name) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.tmp.name)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}

        def num(x):
            try:
                return float(x)
            except ValueError:
                return None

        sm = [num(r[1]) for r in rows if num(r[1]) is not None]
        mx = [num(r[2]) for r in rows if num(r[2]) is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in rows for n, v in zip(names, r[5:9]) if v.lower() == "active"})
        loaded = [s for s in sm if s > 0.5 * max(sm)] if sm else []
        return {"sm_mhz": statistics.median(loaded) if loaded else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows),
                "power_w_max": max((num(r[3]) or 0.0) for r in rows)}


# ----------------------------------------------------------------------------- distributed
def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def aggregate(local_flops: float, local_seconds: float, world_size: int):
    """Whole-job throughput of weakly scaled replicas: every rank's work over
    the slowest rank's time (max over ranks), as the contract requires."""
    if world_size == 1:
        return local_flops, local_seconds
    import torch
    import torch.distributed as dist

    dev = torch.device("cuda", torch.cuda.current_device()) if dist.get_backend() == "nccl" else torch.device("cpu")
    t = torch.tensor([local_seconds], dtype=torch.float64, device=dev)
    f = torch.tensor([local_flops], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    dist.all_reduce(f, op=dist.ReduceOp.SUM)
    return float(f.item()), float(t.item())


# ----------------------------------------------------------------------------- our arm
def workload_config(w, kernel: str, ws: int) -> dict:
    """`config` of the bench line (both arms): the workload and how it is run."""
    from paper_2608_21229_gb300 import accounting as acc

    H, D = w.num_heads, w.head_dim
    live_rows = w.cu_live[-1]
    cache_b = acc.cache_bytes(w.requests, H, D)
    live_b = 3 * live_rows * H * D * 2
    return {
        "workload": w.name, "num_heads": H, "head_dim": D,
        "requests": [[x.n_st, x.n_lt, x.n_x, x.n_r] for x in w.requests],
        "segments": "(N_ST, N_LT, N_X, N_R) per request",
        "step": f"refcache_build + {T_STEPS} step_attention (one layer, one generation)",
        "mask": "beyond (Sec. 3.3)", "kernel": kernel,
        "l2": ("inputs larger than L2" if cache_b + live_b > 129e6 else "inputs smaller than L2 (not flushed)")
              + f": {cache_b / 1e6:.0f} MB cache + {N_LIVE_SETS} live Q/K/V sets of {live_b / 1e6:.0f} MB cycled",
        "parallelism": f"replicas x{ws}" if ws > 1 else "single GPU",
    }


def run_ours(args, ws, rank, local):
    import torch

    import workloads
    from paper_2608_21229_gb300 import accounting as acc
    from paper_2608_21229_gb300 import build as cbuild
    from paper_2608_21229_gb300 import refcache as rcb

    cbuild.build()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    rcb.set_kernel(args.kernel)
    w = workloads.ALL[args.workload]
    H, D = w.num_heads, w.head_dim
    seg = rcb.Segments.from_workload(w)
    cache = rcb.RefCache(seg, num_layers=1, mask_mode="beyond", device=dev, cache_dtype=args.cache)
    scale = 1.0 / math.sqrt(D)
    qs, ks, vs = (t.to(dev) for t in workloads.static_qkv(w))
    lives = [tuple(t.to(dev) for t in workloads.live_qkv(w, step=i)) for i in range(N_LIVE_SETS)]
    o_s = torch.empty(seg.static_rows, H, D, dtype=torch.bfloat16, device=dev)
    o_l = torch.empty(seg.live_rows, H, D, dtype=torch.bfloat16, device=dev)
    stream = torch.cuda.current_stream()

    pre_flops = acc.flops(acc.prefill_units(w.requests), H, D)
    step_flops = acc.flops(acc.step_units(w.requests), H, D)
    full_flops = acc.flops(acc.full_units(w.requests), H, D)
    flops_per_step = pre_flops + T_STEPS * step_flops
    launches_per_step = cache.launches("build") + T_STEPS * cache.launches("step")

    # Events only around the build and around the block of T step calls: an
    # event recorded between two launches would stop the next kernel's
    # prologue from overlapping the previous kernel's tail (programmatic
    # dependent launch), so the step time is the block's time / T.
    def one_step(ev=None):
        if ev is not None:
            ev[0].record(stream)
        cache.build(0, qs, ks, vs, o_s, scale=scale)
        if ev is not None:
            ev[1].record(stream)
        for t in range(T_STEPS):
            ql, kl, vl = lives[t % N_LIVE_SETS]
            cache.step(0, ql, kl, vl, o_l, scale=scale)
        if ev is not None:
            ev[2].record(stream)

    for _ in range(args.warmup):
        one_step()
    torch.cuda.synchronize()
    st = rcb.status()
    if st != rcb.OK:
        raise RuntimeError(f"device error during warm-up: {rcb.last_error()}")
    # the exponential unit's rate on this GPU (the softmax's secondary limit),
    # measured before the timed region
    ex2_rate = rcb.ex2_rate()

    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if ws > 1:
        import torch.distributed as dist

        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        start.record(stream)
        for k in range(args.steps):
            one_step(evs[k])
        end.record(stream)
        torch.cuda.synchronize()
    if ws > 1:
        dist.barrier()
    if rcb.status() != rcb.OK:
        raise RuntimeError(f"device error in the timed region: {rcb.last_error()}")
    total_s = start.elapsed_time(end) / 1e3
    pre_ms = [e[0].elapsed_time(e[1]) for e in evs]
    step_ms = [e[1].elapsed_time(e[2]) / T_STEPS for e in evs]
    t_pre = statistics.mean(pre_ms) / 1e3
    t_step = statistics.mean(step_ms) / 1e3

    # full-attention recompute of the same request on the same kernel (baseline, not timed above)
    t_full = float("nan")
    if not args.no_full:
        t_full = time_full(w, dev, stream, scale)
    e2e = None if args.no_e2e else run_e2e(args, w, cache, seg, dev, stream, scale, flops_per_step)
    cfg = None
    if w.name == "edit1024_5ref" and not args.no_cfg:
        cfg = time_cfg_pair(dev, stream, scale, t_step)
    # the sweep runs before the E4M3 and cuBLAS sections, on a GPU that has only run this kernel
    sweep = ragged = None
    if w.name == "edit1024_5ref" and not args.no_sweep:
        sweep = [time_step_workload(x, dev, stream, scale) for x in workloads.SWEEP_1024]
        ragged = time_step_workload(workloads.RAGGED_4REQ, dev, stream, scale)
    fp8 = None
    if w.name == "edit1024_5ref" and not args.no_fp8 and args.cache == "bf16":
        fp8 = time_fp8_cache(w, dev, stream, scale, t_step)
    linear = None
    if not args.no_linear and t_full == t_full:
        linear = linear_accounting(w, dev, stream, t_pre, t_step, t_full)
    flops_all, secs_all = aggregate(flops_per_step * args.steps, total_s, ws)
    pk = peaks()
    achieved = step_flops / t_step / 1e12
    # the E4M3 cache's cached tiles run on E4M3 MMAs: their peak is the bf16
    # measurement times the nominal E4M3 / bf16 ratio (2)
    peak_mult = 2.0 if args.cache == "fp8" else 1.0
    peak = peak_mult * pk["bf16_burst"]
    clocks = clk.summary()
    sms = torch.cuda.get_device_properties(dev).multi_processor_count

    def roof(flops, secs):
        """One kernel's (or sequence's) roofline figures against the measured
        burst peak (the kernels here run near the maximum SM clock; the
        sustained figure was measured at a lower, power-capped clock)."""
        a = flops / secs / 1e12
        return {"achieved": a, "peak": peak, "unit": "TFLOP/s", "frac": a / peak}
    traffic = recorded_traffic(w.name, args.kernel) if args.cache == "bf16" else None
    for entry in (sweep or []) + ([ragged] if ragged else []):
        for key in ("step", "prefill", "full"):
            if f"{key}_tflops" in entry:
                entry[f"{key}_frac"] = entry[f"{key}_tflops"] / peak
    line = {
        "metric": METRIC,
        "value": flops_all / secs_all / 1e12,
        "unit": UNIT,
        "n_gpus": ws,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": secs_all / args.steps * 1e3,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16" if args.cache == "bf16" else "e4m3 cache, bf16 live",
        "data": "synthetic",
        "config": dict(workload_config(w, args.kernel, ws), cache=args.cache),
        "step_attention": {"ms": t_step * 1e3, "tflops": achieved, "flops": step_flops,
                           "roofline": roof(step_flops, t_step),
                           "timing": f"CUDA events on the launching stream around each bench step's block of "
                                     f"{T_STEPS} calls (attention + combine of split items), / {T_STEPS}"},
        "prefill": {"ms": t_pre * 1e3, "tflops": pre_flops / t_pre / 1e12, "flops": pre_flops,
                    "roofline": roof(pre_flops, t_pre)},
        "full_attention": {"ms": t_full * 1e3, "tflops": full_flops / t_full / 1e12, "flops": full_flops,
                           "roofline": roof(full_flops, t_full)}
        if t_full == t_full else None,
        "speedup_40step": {
            "measured": acc.measured_ratio(t_full, t_pre, t_step, T_STEPS) if t_full == t_full else None,
            "interaction_model": acc.modelled_ratio(w.requests, T_STEPS),
            # the modelled 40-step times (one layer) against their tensor-pipe
            # floors: prefill + 40 steps with the cache, 40 full recomputes without
            "cached_40step": {"ms": (t_pre + T_STEPS * t_step) * 1e3,
                              "roofline_ms": flops_per_step / (peak * 1e12) * 1e3,
                              "frac": flops_per_step / (peak * 1e12) / (t_pre + T_STEPS * t_step)},
            "full_40step": {"ms": T_STEPS * t_full * 1e3,
                            "roofline_ms": T_STEPS * full_flops / (peak * 1e12) * 1e3,
                            "frac": full_flops / (peak * 1e12) / t_full} if t_full == t_full else None,
            "paper_end_to_end": {"5_refs": 3.92, "10_refs": 5.47, "note": "whole model, unnamed GPU (context)"},
        },
        "roofline": {
            "kernel": ("attn_mma_kernel (mma.sync)" if args.kernel == "mma_sync" else
                       "attn_tc2_kernel (tcgen05, CTA pairs, 128-key tiles"
                       + (")" if D == 128 else ", head dim 64 padded to 128)")
                       if args.kernel == "tcgen05_k128" or args.cache == "fp8"
                       else "attn_tc2_kernel (tcgen05, CTA pairs, 192-key tiles"
                       + (")" if D == 128 else ", head dim 64 padded to 128)")) + " in step_attention",
            "bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
            "frac": achieved / peak,
            "peak_kind": (f"bf16 dense, {pk['source']} burst (the timed region runs near the maximum SM clock)"
                          if args.cache == "bf16" else
                          f"E4M3 dense = 2 x bf16 {pk['source']} burst (nominal ratio)"),
            "frac_of_sustained": achieved / (peak_mult * pk["bf16_sustained"]),
            "sustained_note": "the sustained peak was measured at a power-capped median SM clock of about "
                              "1.4 GHz; this kernel's timed region runs near 2 GHz, so it is context only",
            "nominal_at_clock": nominal_at_clock(achieved, clocks.get("sm_mhz"), sms, peak_mult),
            "exp_floor": exp_floor(acc.step_units(w.requests) * H, t_step, clocks.get("sm_mhz"), sms, ex2_rate),
            "traffic": traffic,
            # DRAM bytes of one launch (ncu record) over this run's step time: the
            # cache and live streams' achieved bandwidth against the measured copy rate
            "dram_gbs": traffic / t_step / 1e9 if traffic else None,
            "dram_frac_of_hbm": traffic / t_step / 1e9 / pk["hbm_gbs"] if traffic else None,
            "traffic_source": "ncu dram__bytes_read.sum + dram__bytes_write.sum, one step_attention launch"
                              " (profiles/); null when the kernel sources changed since",
            "algorithmic_bytes": 2 * (seg.live_rows * H * D * 2) * 2
                                 + acc.cache_bytes(w.requests, H, D) // (2 if args.cache == "fp8" else 1),
        },
        "cfg_pair": cfg,
        "fp8_cache": fp8,
        "linear_accounting": linear,
        "reference_sweep": sweep,
        "ragged_batch": ragged,
        "e2e": e2e,
        "clocks": clocks,
        "gpu_launches": launches_per_step * args.steps,
    }
    if rank == 0 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(w, budget_s=args.cpu_budget)
    return line


def nominal_at_clock(achieved, sm_mhz, sms, mult=1.0):
    """The tensor pipe's own ceiling at the SM clock sampled during the timed
    region: 8192 dense bf16 FLOPs per clock per SM (the rate at which ncu's
    sm__pipe_tensor_cycles_active reads 100 %), times the SM count and clock."""
    if not sm_mhz:
        return None
    ceiling = mult * 8192.0 * sms * sm_mhz * 1e6 / 1e12
    return {"sm_mhz": sm_mhz, "sms": sms, "flop_per_clk_per_sm": mult * 8192, "tflops": ceiling,
            "frac": achieved / ceiling}


def exp_floor(units, secs, sm_mhz, sms, ex2_per_clk_per_sm):
    """The secondary ALU limit: one exponential per visible (query, key) pair
    of one head against the exponential unit's rate (ex2.approx.f32 per clock
    per SM, measured on this GPU by the library's probe kernel) at the sampled
    clock."""
    if not sm_mhz:
        return None
    floor = units / (ex2_per_clk_per_sm * sms * sm_mhz * 1e6)
    return {"exps": units, "ex2_per_clk_per_sm": ex2_per_clk_per_sm,
            "ex2_rate_source": "measured on this GPU (refcache_ex2_rate: one CTA per SM, 8 warps x 8 independent "
                               "ex2.approx.f32 chains, clock64)",
            "sm_mhz": sm_mhz, "floor_ms": floor * 1e3, "frac_of_step": floor / secs,
            "note": "time the exponentials need at the sampled clock, as a share of the step"}


def gpu_randn_bf16(shape, seed: int, dev):
    """N(0, 1) bf16 drawn on the device from a seeded generator (timing-only
    inputs; the parity tests use the workloads' CPU draws)."""
    import torch

    g = torch.Generator(device=dev)
    g.manual_seed(seed)
    return torch.randn(shape, generator=g, device=dev, dtype=torch.float32).to(torch.bfloat16)


def time_step_workload(w, dev, stream, scale, with_full=True):
    """One workload's step call (and, if asked, its full-attention recompute)
    timed on its own: build once, then 2 x 40 step calls over four live sets."""
    import torch

    import workloads
    from paper_2608_21229_gb300 import accounting as acc
    from paper_2608_21229_gb300 import refcache as rcb

    H, D = w.num_heads, w.head_dim
    seg = rcb.Segments.from_workload(w)
    cache = rcb.RefCache(seg, num_layers=1, mask_mode="beyond", device=dev)
    qs, ks, vs = (gpu_randn_bf16((seg.static_rows, H, D), 1000 * w.seed + i, dev) for i in range(3))
    lives = [tuple(gpu_randn_bf16((seg.live_rows, H, D), 1000 * w.seed + 10 + 3 * j + i, dev) for i in range(3))
             for j in range(N_LIVE_SETS)]
    o_s = torch.empty(seg.static_rows, H, D, dtype=torch.bfloat16, device=dev)
    o_l = torch.empty(seg.live_rows, H, D, dtype=torch.bfloat16, device=dev)
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    cache.build(0, qs, ks, vs, o_s, scale=scale)
    for _ in range(2):
        cache.build(0, qs, ks, vs, o_s, scale=scale)
    a.record(stream)
    cache.build(0, qs, ks, vs, o_s, scale=scale)
    b.record(stream)
    torch.cuda.synchronize()
    t_pre = a.elapsed_time(b) / 1e3
    for i in range(3):
        cache.step(0, *lives[i % N_LIVE_SETS], o_l, scale=scale)
    n = 2 * T_STEPS
    a.record(stream)
    for i in range(n):
        cache.step(0, *lives[i % N_LIVE_SETS], o_l, scale=scale)
    b.record(stream)
    torch.cuda.synchronize()
    if rcb.status() != rcb.OK:
        raise RuntimeError(f"device error in {w.name}: {rcb.last_error()}")
    t_step = a.elapsed_time(b) / n / 1e3
    step_flops = acc.flops(acc.step_units(w.requests), H, D)
    pre_flops = acc.flops(acc.prefill_units(w.requests), H, D)
    out = {
        "workload": w.name,
        "requests": [[x.n_st, x.n_lt, x.n_x, x.n_r] for x in w.requests],
        "step_ms": t_step * 1e3, "step_tflops": step_flops / t_step / 1e12,
        "prefill_ms": t_pre * 1e3, "prefill_tflops": pre_flops / t_pre / 1e12,
        "cache_mb_streamed_per_step": acc.cache_bytes(w.requests, H, D) / 1e6,
        "interaction_model_40step": acc.modelled_ratio(w.requests, T_STEPS),
    }
    del cache
    if with_full:
        t_full = time_full(w, dev, stream, scale, gpu_inputs=True)
        out["full_ms"] = t_full * 1e3
        out["full_tflops"] = acc.flops(acc.full_units(w.requests), H, D) / t_full / 1e12
        out["measured_40step"] = acc.measured_ratio(t_full, t_pre, t_step, T_STEPS)
    return out


def linear_accounting(w, dev, stream, t_pre, t_step, t_full):
    """Context only: the per-token linear work of one layer that caching also
    removes (App. C, "What the interaction model omits"), timed with cuBLAS
    (torch.matmul, bf16) on random weights, folded into a 40-step model of one
    layer.  Assumed layer shape (the paper does not state it): hidden =
    heads x head_dim, Q/K/V and output projections, a two-matrix FFN of width
    4 x hidden."""
    import torch

    H, D = w.num_heads, w.head_dim
    hid, ffn = H * D, 4 * H * D
    S = sum(x.n_lt + x.n_x for x in w.requests)
    R = sum(x.n_r for x in w.requests)
    ST = sum(x.n_st for x in w.requests)
    g = torch.Generator(device=dev)
    g.manual_seed(7)
    mk = lambda *shape: (torch.randn(shape, generator=g, device=dev) * 0.02).to(torch.bfloat16)  # noqa: E731
    w_qkv, w_o, w_up, w_dn = mk(hid, 3 * hid), mk(hid, hid), mk(hid, ffn), mk(ffn, hid)

    def t_linear(n):
        x = mk(n, hid)
        def run():
            qkv = x @ w_qkv
            o = qkv[:, :hid] @ w_o
            h = torch.nn.functional.gelu(o @ w_up, approximate="tanh")
            return h @ w_dn
        for _ in range(2):
            run()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(5):
            run()
        b.record(stream)
        torch.cuda.synchronize()
        return a.elapsed_time(b) / 5e3

    flops_tok = 2 * (4 * hid * hid + 2 * hid * ffn)
    tl_live, tl_static, tl_all = t_linear(S), t_linear(ST + R), t_linear(S + R)
    full = T_STEPS * (t_full + tl_all)
    cached = t_pre + tl_static + T_STEPS * (t_step + tl_live)
    return {
        "assumed_layer": f"hidden {hid}, QKV + O projections, FFN {ffn} (not stated by the paper)",
        "linear_gflop_per_token": flops_tok / 1e9,
        "linear_ms": {"live_tokens": tl_live * 1e3, "static_tokens": tl_static * 1e3, "all_tokens": tl_all * 1e3},
        "cublas_tflops": flops_tok * (S + R) / tl_all / 1e12,
        "modelled_40step_with_linear": full / cached,
        "note": "context only: one layer, attention times measured above, linear work timed with cuBLAS",
    }


def time_fp8_cache(w, dev, stream, scale, t_step_bf16):
    """The E4M3 reference cache (an approximate variant of the exact cache) on
    the same workload and inputs as the bf16 step: step time, cache bytes, and
    the outputs' distance from the exact kernel's on the same inputs."""
    import torch

    import workloads
    from paper_2608_21229_gb300 import accounting as acc
    from paper_2608_21229_gb300 import refcache as rcb

    H, D = w.num_heads, w.head_dim
    seg = rcb.Segments.from_workload(w)
    cache = rcb.RefCache(seg, num_layers=1, mask_mode="beyond", device=dev, cache_dtype="fp8")
    cache16 = rcb.RefCache(seg, num_layers=1, mask_mode="beyond", device=dev)
    qs, ks, vs = (t.to(dev) for t in workloads.static_qkv(w))
    lives = [tuple(t.to(dev) for t in workloads.live_qkv(w, step=i)) for i in range(N_LIVE_SETS)]
    o_s = torch.empty(seg.static_rows, H, D, dtype=torch.bfloat16, device=dev)
    o_l = torch.empty(seg.live_rows, H, D, dtype=torch.bfloat16, device=dev)
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(stream)
    cache.build(0, qs, ks, vs, o_s, scale=scale)
    b.record(stream)
    for i in range(3):
        cache.step(0, *lives[i % N_LIVE_SETS], o_l, scale=scale)
    torch.cuda.synchronize()
    t_build = a.elapsed_time(b) / 1e3
    n = 2 * T_STEPS
    a.record(stream)
    for i in range(n):
        cache.step(0, *lives[i % N_LIVE_SETS], o_l, scale=scale)
    b.record(stream)
    torch.cuda.synchronize()
    if rcb.status() != rcb.OK:
        raise RuntimeError(f"device error in the E4M3-cache step: {rcb.last_error()}")
    t = a.elapsed_time(b) / n / 1e3
    # distance from the exact (bf16-cache) kernel on live set 0
    o16 = torch.empty_like(o_l)
    cache16.build(0, qs, ks, vs, o_s, scale=scale)
    cache16.step(0, *lives[0], o16, scale=scale)
    cache.step(0, *lives[0], o_l, scale=scale)
    torch.cuda.synchronize()
    d = (o_l.float() - o16.float()).abs()
    flops = acc.flops(acc.step_units(w.requests), H, D)
    bf16_bytes = acc.cache_bytes(w.requests, H, D, "beyond")
    k8, vt8, sc = cache.fp8(0)
    fp8_bytes = k8.numel() + vt8.numel() + sc.numel() * 4
    return {
        "step_ms": t * 1e3,
        "tflops_equivalent": flops / t / 1e12,
        "vs_bf16_step": t / t_step_bf16,
        "build_ms": t_build * 1e3,
        "cache_mb_per_layer": fp8_bytes / 1e6,
        "bf16_cache_mb_per_layer": bf16_bytes / 1e6,
        "max_abs_vs_exact_kernel": float(d.max()),
        "mean_abs_vs_exact_kernel": float(d.mean()),
        "note": "approximate variant: cached K/V as E4M3 with per-tile scales, E4M3 tensor-core MMAs for "
                "cached tiles; same FLOP count as the exact step",
    }


def time_cfg_pair(dev, stream, scale, t_step_positive):
    """Step attention of a guided generation: the positive and the negative
    (blank-text) branch of the headline edit as two requests of one launch."""
    import torch

    import workloads
    from paper_2608_21229_gb300 import accounting as acc
    from paper_2608_21229_gb300 import refcache as rcb

    w = workloads.CFG_1024_5REF
    H, D = w.num_heads, w.head_dim
    seg = rcb.Segments.from_workload(w)
    cache = rcb.RefCache(seg, num_layers=1, mask_mode="beyond", device=dev)
    qs, ks, vs = (t.to(dev) for t in workloads.static_qkv(w))
    lives = [tuple(t.to(dev) for t in workloads.live_qkv(w, step=i)) for i in range(N_LIVE_SETS)]
    o_s = torch.empty(seg.static_rows, H, D, dtype=torch.bfloat16, device=dev)
    o_l = torch.empty(seg.live_rows, H, D, dtype=torch.bfloat16, device=dev)
    cache.build(0, qs, ks, vs, o_s, scale=scale)
    for i in range(3):
        cache.step(0, *lives[i % N_LIVE_SETS], o_l, scale=scale)
    n = 2 * T_STEPS
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for i in range(n):
        cache.step(0, *lives[i % N_LIVE_SETS], o_l, scale=scale)
    b.record(stream)
    torch.cuda.synchronize()
    if rcb.status() != rcb.OK:
        raise RuntimeError(f"device error in the guided step: {rcb.last_error()}")
    t = a.elapsed_time(b) / n / 1e3
    flops = acc.flops(acc.step_units(w.requests), H, D)
    return {
        "workload": w.name,
        "requests": [[x.n_st, x.n_lt, x.n_x, x.n_r] for x in w.requests],
        "step_ms": t * 1e3,
        "tflops": flops / t / 1e12,
        "flops": flops,
        "vs_positive_branch_alone": t / t_step_positive,
        "interaction_model_40step": acc.modelled_ratio(w.requests, T_STEPS),
        "note": "both branches of true CFG (App. D) in one step_attention launch; "
                "the negative branch has no instruction tokens and its own cache",
    }


def time_full(w, dev, stream, scale, gpu_inputs=False):
    """Seconds per full_attention call over every request's [LT; X; R]."""
    import torch

    import workloads
    from paper_2608_21229_gb300 import refcache as rcb

    H, D = w.num_heads, w.head_dim
    cu_full = [0]
    for x in w.requests:
        cu_full.append(cu_full[-1] + x.n_lt + x.n_x + x.n_r)
    n_full = cu_full[-1]
    if gpu_inputs:
        qf, kf, vf = (gpu_randn_bf16((n_full, H, D), 1000 * w.seed + 100 + i, dev) for i in range(3))
    else:
        qf, kf, vf = (workloads.randn_bf16((n_full, H, D), w.seed, f"full_{c}").to(dev) for c in "qkv")
    o_f = torch.empty(n_full, H, D, dtype=torch.bfloat16, device=dev)
    for _ in range(2):
        rcb.full_attention(cu_full, qf, kf, vf, o_f, scale=scale)
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for _ in range(3):
        rcb.full_attention(cu_full, qf, kf, vf, o_f, scale=scale)
    b.record(stream)
    torch.cuda.synchronize()
    if rcb.status() != rcb.OK:
        raise RuntimeError(f"device error in full_attention: {rcb.last_error()}")
    return a.elapsed_time(b) / 3e3


def run_e2e(args, w, cache, seg, dev, stream, scale, flops_per_step):
    """The same step through the public API with host buffers, as a serving
    loop runs it: every step's live Q/K/V are copied in from pinned host
    memory and its O copied back, inside the timed region.  Copies in run on a
    copy stream into two alternating device buffers, copies out on a third
    stream, so transfers overlap the attention kernels; events order the
    reuse of every buffer."""
    import torch

    import workloads

    H, D = w.num_heads, w.head_dim
    hs = [t.pin_memory() for t in workloads.static_qkv(w)]
    hl = [[t.pin_memory() for t in workloads.live_qkv(w, step=i)] for i in range(N_LIVE_SETS)]
    ds = [torch.empty_like(t, device=dev) for t in hs]
    dl = [[torch.empty_like(t, device=dev) for t in hl[0]] for _ in range(2)]
    o_s = torch.empty(seg.static_rows, H, D, dtype=torch.bfloat16, device=dev)
    o_l = [torch.empty(seg.live_rows, H, D, dtype=torch.bfloat16, device=dev) for _ in range(2)]
    ho_s = torch.empty(o_s.shape, dtype=torch.bfloat16).pin_memory()
    ho_l = [torch.empty(o_l[0].shape, dtype=torch.bfloat16).pin_memory() for _ in range(2)]
    h2d = sum(t.numel() * 2 for t in hs) + T_STEPS * sum(t.numel() * 2 for t in hl[0])
    d2h = ho_s.numel() * 2 + T_STEPS * ho_l[0].numel() * 2
    cin, cout = torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)
    ev = lambda: torch.cuda.Event()  # noqa: E731
    loaded, computed, drained = [ev(), ev()], [ev(), ev()], [ev(), ev()]
    for e in computed + drained:  # buffers start free
        e.record(stream)

    def one():
        with torch.cuda.stream(cin):
            for d, h in zip(ds, hs):
                d.copy_(h, non_blocking=True)
            static_in = ev()
            static_in.record(cin)
        stream.wait_event(static_in)
        cache.build(0, ds[0], ds[1], ds[2], o_s, scale=scale, stream=stream)
        built = ev()
        built.record(stream)
        cout.wait_event(built)
        with torch.cuda.stream(cout):
            ho_s.copy_(o_s, non_blocking=True)
        for t in range(T_STEPS):
            b = t & 1
            cin.wait_event(computed[b])  # step t - 2 has read dl[b]
            with torch.cuda.stream(cin):
                for d, h in zip(dl[b], hl[t % N_LIVE_SETS]):
                    d.copy_(h, non_blocking=True)
                loaded[b].record(cin)
            stream.wait_event(loaded[b])
            stream.wait_event(drained[b])  # o_l[b] of step t - 2 is on the host
            cache.step(0, dl[b][0], dl[b][1], dl[b][2], o_l[b], scale=scale, stream=stream)
            computed[b].record(stream)
            cout.wait_event(computed[b])
            with torch.cuda.stream(cout):
                ho_l[b].copy_(o_l[b], non_blocking=True)
                drained[b].record(cout)
        stream.wait_event(drained[0])
        stream.wait_event(drained[1])
        stream.wait_stream(cin)

    one()
    torch.cuda.synchronize()
    # each step timed on its own (events after the stream has waited for the
    # last copies out); the value is the median step, so that a stray slow
    # step (the host is shared) does not decide it -- every step is listed
    n = max(5, min(args.steps, 7))
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n)]
    with ClockSampler(torch.cuda.current_device()) as clk:
        for a, b_ in evs:
            a.record(stream)
            one()
            b_.record(stream)
        torch.cuda.synchronize()
    ms = [a.elapsed_time(b_) for a, b_ in evs]
    secs = statistics.median(ms) / 1e3
    return {"value": flops_per_step / secs / 1e12, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "ms_per_step": secs * 1e3, "steps": n, "timing": "median of the steps",
            "step_ms": [round(x, 3) for x in ms], "mean_ms": statistics.mean(ms), "clocks": clk.summary(),
            "overlap": "copies in on a copy stream (2 device buffers), copies out on a third stream, "
                       "ordered by events; every byte moves inside the timed region"}


# ----------------------------------------------------------------------------- CPU oracle
def oracle_sample(w, n_pairs_step, n_pairs_pre, seed=0):
    """A bounded sample of the workload for the CPU oracle: (row, head) pairs of
    the step and of the prefill, in proportion to their share of the FLOPs."""
    import numpy as np

    import workloads

    rng = np.random.default_rng(seed)
    r = w.requests[0]
    static = [workloads.bf16_bits(t) for t in workloads.static_qkv(w)]
    live = [workloads.bf16_bits(t) for t in workloads.live_qkv(w)]
    sp = np.stack([rng.integers(0, r.n_live, n_pairs_step), rng.integers(0, w.num_heads, n_pairs_step)], 1)
    pp = np.stack([rng.integers(0, r.n_static, n_pairs_pre), rng.integers(0, w.num_heads, n_pairs_pre)], 1)
    return static, live, sp.astype(np.int32), pp.astype(np.int32)


def time_oracle_sample(w, static, live, sp, pp):
    """Time the oracle's attention on the sampled outputs (the joint sequences
    are assembled before the clock starts)."""
    import oracle

    r = w.requests[0]
    scale = 1.0 / math.sqrt(w.head_dim)
    kc, vc = oracle.cached_kv(static[1], static[2], r.n_st, "beyond")
    joint = oracle.step_inputs(*live, kc, vc, r.n_lt, r.n_x, r.n_st, r.n_r, "beyond")
    t0 = time.perf_counter()
    oracle.joint_attention(*static, 0, 0, r.n_st, r.n_r, "beyond", scale, pp)
    oracle.joint_attention(*joint, r.n_lt, r.n_x, r.n_st, r.n_r, "beyond", scale, sp)
    secs = time.perf_counter() - t0
    d = w.head_dim
    flops = 4 * d * (len(sp) * (r.n_live + r.n_r) + len(pp) * (r.n_st + r.n_r))
    return flops, secs


def sample_sizes(w, total_pairs):
    from paper_2608_21229_gb300 import accounting as acc

    r = w.requests[0]
    pre = acc.prefill_units(w.requests)
    stp = T_STEPS * acc.step_units(w.requests)
    # a step pair costs (N_live + N_R) units, a prefill pair (N_ST + N_R): keep
    # the sample's prefill/step FLOP ratio equal to the workload's
    n_step = max(1, int(total_pairs))
    n_pre = max(1, round(n_step * (pre / stp) * (r.n_live + r.n_r) / (r.n_st + r.n_r)))
    return n_step, n_pre


def cpu_baseline(w, budget_s=15.0):
    import oracle

    oracle.build()
    static, live, sp, pp = oracle_sample(w, *sample_sizes(w, 64))
    f, s = time_oracle_sample(w, static, live, sp, pp)  # calibration
    scale = max(1.0, budget_s / max(s, 1e-3))
    n_step, n_pre = sample_sizes(w, int(64 * scale))
    static, live, sp, pp = oracle_sample(w, n_step, n_pre, seed=1)
    f, s = time_oracle_sample(w, static, live, sp, pp)
    cores = oracle.max_threads()
    return {"value": f / s / 1e12, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"{len(sp)} (row, head) outputs of the step and {len(pp)} of the prefill of {w.name}, "
                      f"fp64 plain definition, {s:.1f} s",
            "seconds": s, "flops": f, "single_thread": single_thread_oracle(cores)}


def single_thread_oracle(cores_after, pairs=512):
    """The oracle on one host core for the two small workloads (context for
    the multi-core figure): a bounded sample of each, GFLOP/s."""
    import oracle
    import workloads

    out = []
    oracle.set_threads(1)
    try:
        for w in (workloads.TINY, workloads.EDIT_512_2REF):
            static, live, sp, pp = oracle_sample(w, *sample_sizes(w, pairs), seed=2)
            f, s = time_oracle_sample(w, static, live, sp, pp)
            out.append({"workload": w.name, "outputs": int(len(sp) + len(pp)), "seconds": s, "gflops": f / s / 1e9})
    finally:
        oracle.set_threads(cores_after)
    return out


def run_reference(args, ws, rank):
    if rank != 0:
        return None
    import oracle

    import workloads

    oracle.build()
    w = workloads.ALL[args.workload]
    n_step, n_pre = sample_sizes(w, args.ref_pairs)
    static, live, sp, pp = oracle_sample(w, n_step, n_pre)
    for _ in range(args.warmup):
        time_oracle_sample(w, static, live, sp[:8], pp[:1])
    tot_f = tot_s = 0.0
    for _ in range(args.steps):
        f, s = time_oracle_sample(w, static, live, sp, pp)
        tot_f += f
        tot_s += s
    v = tot_f / tot_s / 1e12
    sample = f"per step {len(sp)} step and {len(pp)} prefill (row, head) outputs of {w.name}"
    return {"metric": METRIC, "value": v, "unit": UNIT, "n_gpus": ws, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": tot_s / args.steps * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic", "impl": "reference",
            "config": dict(workload_config(w, "cpu oracle (plain fp64 definition) on bounded samples", ws),
                           cache=args.cache),
            "cpu_baseline": {"value": v, "unit": UNIT, "cores": oracle.max_threads(), "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="edit1024_5ref")
    ap.add_argument("--kernel", choices=["tcgen05", "tcgen05_k128", "mma_sync"], default="tcgen05")
    ap.add_argument("--cpu-budget", type=float, default=15.0, help="seconds of oracle work for cpu_baseline")
    ap.add_argument("--ref-pairs", type=int, default=192, help="oracle (row, head) outputs per reference step")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true", help="skip the host-buffer end-to-end measurement")
    ap.add_argument("--no-full", action="store_true", help="skip the full-attention baseline")
    ap.add_argument("--no-cfg", action="store_true", help="skip the guided (positive + negative branch) step")
    ap.add_argument("--no-fp8", action="store_true", help="skip the E4M3-cache variant")
    ap.add_argument("--cache", choices=("bf16", "fp8"), default="bf16",
                    help="format of the main run's reference cache (fp8: the approximate E4M3 variant)")
    ap.add_argument("--no-linear", action="store_true", help="skip the cuBLAS-timed linear-work accounting")
    ap.add_argument("--no-sweep", action="store_true",
                    help="skip the 1024^2 reference sweep (1-10 refs) and the ragged serving batch")
    args = ap.parse_args(argv)
    ws, rank, local = dist_env()
    if args.warmup < 3:
        args.warmup = 3
    if ws > 1 and args.impl == "ours":
        import torch
        import torch.distributed as dist

        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    if args.impl == "reference":
        line = run_reference(args, ws, rank)
    else:
        line = run_ours(args, ws, rank, local)
    if rank == 0 and line is not None:
        print(json.dumps(line), flush=True)
    if ws > 1 and args.impl == "ours":
        import torch.distributed as dist

        dist.destroy_process_group()


if __name__ == "__main__":
    main()
