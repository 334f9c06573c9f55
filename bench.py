#!/usr/bin/env python
"""Throughput of the CLEAR-MoE FFN layer on GB300; prints one JSON line.

A step is one CLEAR-MoE FFN forward (routing, fc1 + GELU, shared-basis factor, grouped residual
experts with the scatter) over one batch of synthetic ViT tokens, through the library's C ABI.
The headline workload is the DeiT-B / ViT-B-shaped layer (T = 256 images x 197 tokens = 50,432,
d = 768, H = 3,072, E = 8, r = 128, bf16), the shape the GEMM target is quoted on. The same line
carries the other workloads under "configs": the DeiT-T fp32 layer, the DeiT-S bf16 layer, the
DeiT-S expert-count x rank sweep with Zipf cluster sizes, and the 12-sublayer ViT-B stack.

  value  tokens/s over K timed steps (inputs resident in HBM), CUDA events on the launch stream
         around each step only; before every step (outside the events) L2 is flushed without
         leaving dirty lines: a 256 MB zero-fill, then a 512 MB read of a second buffer
  stages per-kernel durations from a second pass with an event between consecutive kernels;
         their fractions use the burst bf16 peak (a sub-second pass), the sustained one beside it
         the routing stage also gives its rate net of the launch floor (the event time of a
         one-element kernel after the same flush), beside the raw figure, which stays the headline
  e2e    the same call with x copied from pinned host memory and out copied back inside each step
  roofline  the dominant kernel's algorithmic FLOPs (or bytes) per launch / its event-timed duration
  cpu_baseline  the float64 CPU oracles on a bounded sample of the same workload (rank 0, N = 1):
         the numpy oracle (value), the plain-C oracle on one thread and on every host core

--impl reference times the CPU oracle itself (the method has no other reference code).
Multi-GPU (torchrun): every rank runs an independent replica on its own tokens (weak scaling;
the layer needs no exchange between token shards); value = all tokens / max rank time.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import pathlib
import statistics
import subprocess
import sys
import time

ROOT = pathlib.Path(__file__).resolve().parent
sys.path.insert(0, str(ROOT))

METRIC = ("CLEAR-MoE FFN tokens/sec/layer (1×GB300) + % HBM peak (dispatch), "
          "% tensor peak (GEMMs)")
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
# the GB300's nominal figures (HBM3e ~7.9 TB/s; dense bf16 2.25 PFLOP/s), reported beside the
# measured peaks for context
NOMINAL_PEAKS = {"hbm_gbs": 7900.0, "bf16_tflops": 2250.0}
# The fp32 layer's GEMMs run on the TF32 tensor cores, three TF32 products per fp32 product: their
# peak in fp32 FLOP/s is the measured bf16 peak x the nominal TF32 / bf16 ratio (1.1 / 2.25 PFLOP/s
# dense) / 3
TF32X3_OF_BF16 = 1.1 / 2.25 / 3
STAGES = ("route", "fc1_gelu", "basis", "grouped")
KERNEL_OF_STAGE = {"route": "cm::route_tc_kernel",
                   "fc1_gelu": "cm::tc_gemm2_kernel<256, 0, 0> (2-SM dense, rows stored at their routing slots)",
                   "basis": "cm::tc_gemm2_kernel<128, 0, 0> (2-SM dense, column scale)",
                   "grouped": "cm::tc_gemm2_kernel<256, 2, 0> (2-SM grouped, rows stored at perm[slot])"}
# DRAM traffic per launch (dram__bytes_read.sum + dram__bytes_write.sum) from the committed ncu
# capture (profiles/clearmoe_kernels_deit_base_T50432_full.md), with the hash of the kernel's sources
# it was taken on (source_hash); a different hash means the kernel changed and the figure is void.
TRAFFIC = {
    "route": {"bytes": 78.52416e6, "src": "3deea90ad96906dc"},
    "fc1_gelu": {"bytes": 338.377472e6, "src": "eb41af172793f61c"},
    "basis": {"bytes": 316.010752e6, "src": "eb41af172793f61c"},
    "grouped": {"bytes": 426.028544e6, "src": "eb41af172793f61c"},
}


def init_replicas(backend="nccl"):
    """One process per GPU (torchrun's RANK / WORLD_SIZE / LOCAL_RANK): (world, rank, local, dist),
    dist None for a single process. Each rank runs an independent replica on its own token shard;
    the only collectives are the barriers and the max of the rank times. A rank that dies between
    steps is detected by the others at their next collective, which fails with an error within the
    process group's timeout (CLEARMOE_PG_TIMEOUT_S seconds, default 600) instead of waiting forever."""
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dist = None
    if world > 1:
        import datetime

        import torch.distributed as dist
        timeout = datetime.timedelta(seconds=float(os.environ.get("CLEARMOE_PG_TIMEOUT_S", "600")))
        dist.init_process_group(backend, timeout=timeout)
    return world, rank, local, dist


def max_over_ranks(x: float, dist, device="cuda") -> float:
    """The largest of the ranks' values (a time: the job is as slow as its slowest rank)."""
    if not dist:
        return float(x)
    import torch
    t = torch.tensor([float(x)], device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_rank: int, world: int, steps: int, ms: float) -> float:
    """Units per second over all ranks (weak scaling: every rank processes units_per_rank per step)."""
    return world * units_per_rank * steps / (ms / 1e3)


def workloads():
    import synth
    return {"deit_base_bf16": synth.DEIT_BASE_BF16, "deit_small_bf16": synth.DEIT_SMALL_BF16,
            "deit_tiny_fp32": synth.DEIT_TINY_FP32, "vit_base_stack12": synth.VIT_BASE_STACK12,
            "deit_small_zipf_sweep": None}


def peaks():
    p = ROOT / "MEASURED_PEAKS.json"
    if p.exists():
        d = json.loads(p.read_text())
        return {k: float(d[k]) for k in FALLBACK_PEAKS}, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


def stage_work(s):
    """Algorithmic work per launch of each kernel (per-token figures x T)."""
    esz = 2 if s.dtype == "bf16" else 4
    T, d, H, E, r = s.T, s.d, s.H, s.E, s.r
    return {
        "route": {"bytes": T * d * esz + (E * d + E) * esz + 8 * T + 8 * E, "flops": 2 * T * d * E},
        "fc1_gelu": {"flops": 2 * T * d * H},
        "basis": {"flops": 2 * T * H * r},
        "grouped": {"flops": 2 * T * d * r + 2 * T * d * H},
    }


def layer_flops(s):
    return s.T * (2 * s.d * s.H + 2 * s.r * (s.H + s.d) + 2 * s.d * s.H + 2 * s.d * s.E)


def layer_roofline_s(s, pk, tensor_key="bf16_tflops_sustained"):
    """The slower of the layer's FLOPs at the tensor peak pk[tensor_key] and its minimum bytes
    (tokens in and out, weights once) at the HBM peak."""
    esz = 2 if s.dtype == "bf16" else 4
    T, d, H, E, r = s.T, s.d, s.H, s.E, s.r
    weights = (H * d + H + d * r + r + r * H + E * d * H + E * d + E) * esz
    bytes_ = 2 * T * d * esz + weights
    return max(layer_flops(s) / (pk[tensor_key] * 1e12), bytes_ / (pk["hbm_gbs"] * 1e9))


KERNEL_SOURCES = {"route": ("route.cu", "common.cuh", "internal.h"),
                  "fc1_gelu": ("tc_gemm2.cu", "common.cuh", "internal.h"),
                  "basis": ("tc_gemm2.cu", "common.cuh", "internal.h"),
                  "grouped": ("tc_gemm2.cu", "common.cuh", "internal.h")}


def source_hash(stage):
    """Hash of the sources the stage's kernel is compiled from: a capture's traffic figure holds
    only while they are unchanged."""
    h = hashlib.sha256()
    for f in KERNEL_SOURCES[stage]:
        h.update((ROOT / "paper_2606_28516_gb300" / "csrc" / f).read_bytes())
    return h.hexdigest()[:16]


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 100 ms during the timed region."""

    Q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *a):
        self.rows = []
        if self.proc is None:
            return
        time.sleep(0.2)
        self.proc.terminate()
        out, _ = self.proc.communicate(timeout=10)
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) == 7:
                self.rows.append(f)

    def summary(self):
        if not getattr(self, "rows", None):
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"]}
        sm = [float(r[0]) for r in self.rows if r[0].replace(".", "").isdigit()]
        mx = [float(r[1]) for r in self.rows if r[1].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in self.rows for i in range(4) if r[3 + i] == "Active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons,
                "samples": len(self.rows)}


def oracle_rate(L, budget_s=12.0, chunk=1024, max_tokens=None, warm=True):
    """Oracle tokens/s on row chunks of the workload until budget_s of CPU time is spent."""
    from oracle import clearmoe as O
    s = L["shape"]
    if warm:  # start the BLAS threads outside the timed part
        O.route(L["x"][: min(s.T, 8192)], L["Wg"], L["bg"])
    done, t0 = 0, time.perf_counter()
    limit = max_tokens or s.T
    while done < limit:
        n = min(chunk, limit - done)
        rows = slice(done, done + n)
        a = O.route(L["x"][rows], L["Wg"], L["bg"])["a"]
        O.ffn_forward(L["x"][rows], L["W1"], L["b1"], L["U"], L["S"], L["Vh"], L["residuals"],
                      a=a, z_bf16=s.dtype == "bf16")
        done += n
        if time.perf_counter() - t0 >= budget_s:
            break
    el = time.perf_counter() - t0
    return done / el, done, el


def c_oracle_rates(L, budget_s=8.0, chunk=32):
    """The plain-C float64 oracle (oracle/clearmoe_ref.c) on row chunks of the workload: routing
    (logits, argmax), fc1 + GELU and the experts with W_shared formed once beforehand (excluded from
    the time), on one thread and then on one thread per host core (ctypes releases the interpreter
    lock during each C call, so chunks run in parallel). Returns a dict of both rates."""
    import concurrent.futures as cf
    import ctypes

    import numpy as np

    from oracle import ref_c as R
    lib = R.lib()
    s = L["shape"]
    d64 = lambda a: np.ascontiguousarray(a, dtype=np.float64)
    x, W1, b1, Wg, bg, res = (d64(L[k]) for k in ("x", "W1", "b1", "Wg", "bg", "residuals"))
    Wsh = R.shared_weight(L["U"], L["S"], L["Vh"])
    P, I = ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_int32)
    p = lambda a: a.ctypes.data_as(P)
    E, d, H = s.E, s.d, s.H
    zb = int(s.dtype == "bf16")

    def run_chunk(t0):
        n = min(chunk, s.T - t0)
        xr = x[t0:t0 + n]
        lg, a = np.empty((n, E)), np.empty(n, np.int32)
        z, y = np.empty((n, H)), np.empty((n, d))
        lib.cmref_router_logits(p(xr), n, d, p(Wg), p(bg), E, p(lg))
        lib.cmref_argmax(p(lg), n, E, 0, a.ctypes.data_as(I))
        lib.cmref_fc1_gelu(p(xr), n, d, H, p(W1), p(b1), zb, p(z))
        lib.cmref_experts_forward(p(z), n, d, H, p(Wsh), p(res), E, a.ctypes.data_as(I), None, None, p(y))
        return n

    starts = list(range(0, s.T, chunk))
    done, k, t0 = 0, 0, time.perf_counter()
    while time.perf_counter() - t0 < budget_s / 2 and k < len(starts):
        done += run_chunk(starts[k])
        k += 1
    one = done / (time.perf_counter() - t0)
    cores = len(os.sched_getaffinity(0))
    deadline = time.perf_counter() + budget_s / 2
    todo = iter(starts)

    def worker():
        n = 0
        for st in todo:  # next() on a shared iterator hands each chunk out once
            n += run_chunk(st)
            if time.perf_counter() > deadline:
                break
        return n

    t1 = time.perf_counter()
    with cf.ThreadPoolExecutor(cores) as ex:
        done_all = sum(ex.map(lambda _: worker(), range(cores)))
    allc = done_all / (time.perf_counter() - t1)
    return {"one_thread": {"value": one, "unit": "tokens/s", "cores": 1, "tokens": done},
            "all_cores": {"value": allc, "unit": "tokens/s", "cores": cores, "tokens": done_all},
            "sample": f"{chunk}-token chunks from the start of the workload, ~{budget_s / 2:.0f} s each; "
                      "W_shared formed once beforehand (not timed); gcc -O2, contraction off"}


def blas_threads():
    try:
        from threadpoolctl import threadpool_info
        n = [i.get("num_threads") for i in threadpool_info() if i.get("user_api") == "blas"]
        if n:
            return int(max(n))
    except Exception:
        pass
    return len(os.sched_getaffinity(0))


def run_reference(args):
    import numpy as np  # noqa: F401
    import synth
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    shape = workloads()[args.workload]
    if not isinstance(shape, synth.LayerShape):  # the sweep and the stack: one of their layers
        shape = (synth.deit_small_zipf(4, 64) if args.workload == "deit_small_zipf_sweep"
                 else synth.DEIT_BASE_BF16.with_(T=synth.VIT_BASE_STACK12.T))
    L = synth.make_layer(shape)
    # per-step sample sized so that warmup + steps take about --ref-budget-s of CPU time in total
    probe, _, _ = oracle_rate(L, budget_s=min(2.0, args.ref_budget_s / 4), chunk=256, max_tokens=512)
    per_step = max(16, min(4096, int(probe * args.ref_budget_s / max(1, args.steps + args.warmup))))
    for _ in range(args.warmup):
        oracle_rate(L, budget_s=1e9, chunk=per_step, max_tokens=per_step, warm=False)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        oracle_rate(L, budget_s=1e9, chunk=per_step, max_tokens=per_step, warm=False)
    el = time.perf_counter() - t0
    value = per_step * args.steps / el
    cores = blas_threads()
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": el * 1e3 / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": shape.name, "T": shape.T, "d": shape.d, "H": shape.H,
                   "E": shape.E, "r": shape.r, "sample_tokens_per_step": per_step},
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                         "sample": f"{per_step} tokens of the workload per step (float64 numpy "
                                   f"oracle, Algorithm 3 order, W_shared materialised per call)"},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
        "gpu_launches": 0,
    }
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------ GPU timing helpers
class L2Flush:
    """Before a timed step: a 256 MB zero-fill (twice L2), then a 512 MB read of a second buffer.
    The read evicts the zero-fill's dirty lines, so their write-back happens here, outside the
    timed events, rather than in the step's first kernel; L2 is left holding clean lines of a
    buffer the step never touches. A read of only 256 MB after the fill measured as leaving dirty
    lines behind (the routing kernel after it 22.5 against 20.5 us, the same as after a read-only
    1 GB pass)."""

    def __init__(self):
        import torch
        # float32 throughout: a sum whose result type differs from its input's (int32 into int64)
        # first copies the input into a wider temporary
        self.w = torch.empty(64 * 1024 * 1024, dtype=torch.float32, device="cuda")
        self.r = torch.ones(128 * 1024 * 1024, dtype=torch.float32, device="cuda")
        self.sink = torch.empty((), dtype=torch.float32, device="cuda")

    def __call__(self):
        import torch
        self.w.zero_()
        torch.sum(self.r, 0, out=self.sink)


def time_steps(fn, K, warmup, flush, stream):
    """ms of each of K calls of fn, events on the launching stream around fn only, flush before each."""
    import torch
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(K)]
    for k in range(warmup + K):
        flush()
        if k >= warmup:
            ev[k - warmup][0].record(stream)
        fn()
        if k >= warmup:
            ev[k - warmup][1].record(stream)
    torch.cuda.synchronize()
    return [e[0].elapsed_time(e[1]) for e in ev]


def stage_pass(cm, h, fn, K, flush):
    """Per-kernel ms over K forwards: the library records an event between consecutive kernels."""
    import torch
    sev = [[torch.cuda.Event(enable_timing=True) for _ in range(5)] for _ in range(K)]
    torch.cuda.synchronize()
    for k in range(K):
        flush()
        cm.clearmoe_set_profile_events(h, sev[k])
        fn()
    torch.cuda.synchronize()
    cm.clearmoe_set_profile_events(h, [])
    return {st: [sev[k][i].elapsed_time(sev[k][i + 1]) for k in range(K)] for i, st in enumerate(STAGES)}


def launch_floor_us(flush, K=50):
    """Median event time of a one-element torch kernel after the same L2 flush, timed like a stage:
    the share of an event-timed stage that is the launch of a kernel rather than its work."""
    import torch
    tiny = torch.zeros(1, device="cuda")
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(K)]
    for k in range(K + 3):
        flush()
        if k >= 3:
            ev[k - 3][0].record()
        tiny.add_(1)
        if k >= 3:
            ev[k - 3][1].record()
    torch.cuda.synchronize()
    return statistics.median(e[0].elapsed_time(e[1]) for e in ev) * 1e3


def stage_summary(s, stage_ms, pk, floor_us=None):
    """Mean duration of each kernel with its achieved rate against the burst peak (the stage pass
    is sub-second), the sustained and the nominal peaks beside it. floor_us: the measured launch
    floor; the routing stage, whose kernel is short, also reports its rate with the floor taken out
    (beside the raw figures, which stay the ones used elsewhere)."""
    work = stage_work(s)
    out = {}
    for st, v in stage_ms.items():
        us = statistics.mean(v) * 1e3
        if st == "route":
            g = work[st]["bytes"] / (us * 1e-6) / 1e9
            out[st] = {"us": us, "GB_s": g, "hbm_frac": g / pk["hbm_gbs"],
                       "hbm_frac_nominal": g / NOMINAL_PEAKS["hbm_gbs"]}
            if floor_us is not None and us > floor_us:
                gn = work[st]["bytes"] / ((us - floor_us) * 1e-6) / 1e9
                out[st].update(launch_floor_us=floor_us, us_less_launch_floor=us - floor_us,
                               hbm_frac_less_launch_floor=gn / pk["hbm_gbs"])
        else:
            tf = work[st]["flops"] / (us * 1e-6) / 1e12
            out[st] = {"us": us, "TFLOP_s": tf}
            if s.dtype == "bf16":
                out[st].update(tensor_frac=tf / pk["bf16_tflops"],
                               tensor_frac_sustained=tf / pk["bf16_tflops_sustained"],
                               tensor_frac_nominal=tf / NOMINAL_PEAKS["bf16_tflops"])
            else:
                out[st].update(tensor_frac=tf / (pk["bf16_tflops"] * TF32X3_OF_BF16),
                               tensor_frac_sustained=tf / (pk["bf16_tflops_sustained"] * TF32X3_OF_BF16))
    return out


def layer_block(s, D, h, cm, args, world, dist, flush, stream, pk):
    """One layer workload timed like the headline: tokens/s of the whole forward, the per-kernel
    stage pass, the layer's roofline fraction and the same-shape dense FFN."""
    import torch
    out = torch.empty(s.T, s.d, device="cuda", dtype=D["x"].dtype)

    def forward():
        cm.clearmoe_ffn_forward(h, D["x"], D["W1"], D["b1"], D["U"], D["S"], D["Vh"], D["residuals"],
                                D["Wg"], D["bg"], out)

    K = max(1, args.steps)
    ms = time_steps(forward, K, args.warmup, flush, stream)
    assert cm.clearmoe_layer_status(h) == 0
    mean_ms = max_over_ranks(statistics.mean(ms), dist)
    st = stage_pass(cm, h, forward, min(K, 300), flush)
    assert cm.clearmoe_layer_status(h) == 0
    floor = launch_floor_us(flush)
    dms = time_steps(lambda: cm.clearmoe_dense_ffn_forward(h, D["x"], D["W1"], D["b1"], D["W2"], out),
                     min(K, 300), args.warmup, flush, stream)
    dense_ms = max_over_ranks(statistics.mean(dms), dist)
    res = {"workload": s.name, "T": s.T, "d": s.d, "H": s.H, "E": s.E, "r": s.r, "dtype": s.dtype,
           "value": whole_job_rate(s.T, world, 1, mean_ms), "unit": "tokens/s", "ms_per_step": mean_ms,
           "steps": K, "stages": stage_summary(s, st, pk, floor),
           "dense_ffn": {"value": whole_job_rate(s.T, world, 1, dense_ms), "unit": "tokens/s",
                         "ms_per_step": dense_ms}}
    if s.dtype == "bf16":
        res["layer_roofline_frac"] = layer_roofline_s(s, pk, "bf16_tflops") / (mean_ms / 1e3)
        res["layer_roofline_frac_sustained"] = layer_roofline_s(s, pk) / (mean_ms / 1e3)
    else:  # fp32 on the TF32 tensor cores, three products per fp32 product
        tf = layer_flops(s) / (mean_ms * 1e-3) / 1e12
        peak = pk["bf16_tflops"] * TF32X3_OF_BF16
        res["roofline"] = {"bound": "tensor", "achieved": tf, "peak": peak, "unit": "TFLOP/s",
                           "frac": tf / peak,
                           "peak_source": "measured burst bf16 x nominal TF32 / bf16 (1.1 / 2.25) / 3 (three "
                                          "TF32 products per fp32 product)"}
    return res, out


def sweep_block(args, world, rank, dist, flush, cm):
    """The expert-count x rank sweep on the DeiT-S shape with Zipf(1.2) cluster sizes (E in
    {2, 3, 4, 6, 8} x r in {16, 32, 64, 128, 256}, T = 12,608, bf16): tokens/s of the whole layer at
    each point, timed like the headline, beside the same-shape dense FFN. value = the median."""
    import torch

    import synth
    K = max(1, min(args.steps, 100))
    stream = torch.cuda.current_stream()
    points, dense = [], None
    for E in synth.ZIPF_E:
        for r in synth.ZIPF_R:
            shape = synth.deit_small_zipf(E, r, seed=rank).with_(n_cal=8000)
            L = synth.make_layer(shape)
            D = synth.to_torch(L)
            h = cm.clearmoe_layer_create(shape.T, shape.d, shape.H, E, r, cm.BF16)
            out = torch.empty(shape.T, shape.d, device="cuda", dtype=torch.bfloat16)
            ms = time_steps(lambda: cm.clearmoe_ffn_forward(h, D["x"], D["W1"], D["b1"], D["U"], D["S"], D["Vh"],
                                                            D["residuals"], D["Wg"], D["bg"], out),
                            K, args.warmup, flush, stream)
            ms = max_over_ranks(statistics.mean(ms), dist)
            if dense is None:
                dms = time_steps(lambda: cm.clearmoe_dense_ffn_forward(h, D["x"], D["W1"], D["b1"], D["W2"], out),
                                 K, args.warmup, flush, stream)
                dms = max_over_ranks(statistics.mean(dms), dist)
                dense = {"value": whole_job_rate(shape.T, world, 1, dms), "unit": "tokens/s", "ms_per_step": dms}
            assert cm.clearmoe_layer_status(h) == 0
            counts = torch.empty(E, dtype=torch.int32, device="cuda")
            cm.clearmoe_get_routing(h, counts=counts)
            c = counts.cpu().tolist()
            points.append({"E": E, "r": r, "tokens_s": whole_job_rate(shape.T, world, 1, ms), "ms": ms,
                           "largest_expert_share": max(c) / shape.T})
            cm.clearmoe_layer_destroy(h)
            del D, L
    return {"workload": "deit_small_zipf_sweep", "T": 12608, "d": 384, "H": 1536, "E": list(synth.ZIPF_E),
            "r": list(synth.ZIPF_R), "sizes": "zipf(1.2)", "n_cal": 8000,
            "value": statistics.median(p["tokens_s"] for p in points), "unit": "tokens/s",
            "value_is": "median over the 25 points", "steps": K,
            "ms_per_step": statistics.median(p["ms"] for p in points), "points": points, "dense_ffn": dense}


def stack_block(args, world, rank, dist, cm, with_cpu=False, with_variants=True):
    """The 12-sublayer ViT-B stack (odd sublayers CLEAR-MoE, x_{l+1} = LN(y_l)), end to end on one
    stream: tokens / time of one pass through all 12 sublayers. The pass's input (155 MB) and
    weights exceed L2, so no flush is needed between passes."""
    import numpy as np
    import torch

    import synth
    sh = synth.VIT_BASE_STACK12
    S = synth.make_stack(sh)
    T = S["T"]
    dev = lambda a: torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to("cuda", torch.bfloat16)
    layers = []
    for L in S["layers"]:
        G = dict(moe=L["moe"], W1=dev(L["W1"]), b1=dev(L["b1"]))
        if L["moe"]:
            G.update(U=dev(L["U"]), S=torch.from_numpy(L["S"].astype(np.float32)).cuda(), Vh=dev(L["Vh"]),
                     residuals=dev(L["residuals"]), Wg=dev(L["Wg"]), bg=dev(L["bg"]))
        else:
            G["W2"] = dev(L["W2"])
        layers.append(G)
    h = cm.clearmoe_layer_create(T, sh.d, sh.H, sh.E, sh.r, cm.BF16)
    x0 = dev(S["x"])
    buf = [torch.empty_like(x0) for _ in range(2)]
    y = torch.empty_like(x0)

    def stack_pass(x_in, folded=False, ln_fold=False):
        """ln_fold: each LayerNorm folded into the next sublayer's router and fc1 (that sublayer is
        given y itself); the last one still runs, so that both forms return LN(y_11)."""
        x = x_in
        for l, G in enumerate(layers):
            if ln_fold:
                ln, yl = l > 0, buf[l & 1]
                if G["moe"] and folded:
                    cm.clearmoe_ffn_forward_folded_ex(h, x, G["W1"], G["b1"], G["W_comb"], G["Wg"], G["bg"], yl,
                                                      input_layernorm=ln)
                elif G["moe"]:
                    cm.clearmoe_ffn_forward_ex(h, x, G["W1"], G["b1"], G["U"], G["S"], G["Vh"], G["residuals"],
                                               G["Wg"], G["bg"], yl, input_layernorm=ln)
                else:
                    cm.clearmoe_dense_ffn_forward_opt(h, x, G["W1"], G["b1"], G["W2"], yl, input_layernorm=ln)
                x = yl
                continue
            if G["moe"] and folded:
                cm.clearmoe_ffn_forward_folded(h, x, G["W1"], G["b1"], G["W_comb"], G["Wg"], G["bg"], y)
            elif G["moe"]:
                cm.clearmoe_ffn_forward(h, x, G["W1"], G["b1"], G["U"], G["S"], G["Vh"], G["residuals"],
                                        G["Wg"], G["bg"], y)
            else:
                cm.clearmoe_dense_ffn_forward(h, x, G["W1"], G["b1"], G["W2"], y)
            x = buf[l & 1]
            cm.clearmoe_layer_norm(h, y, x)
        if ln_fold:
            cm.clearmoe_layer_norm(h, x, y)
            x = y
        return x

    def timed(K, folded=False, ln_fold=False):
        for _ in range(args.warmup):
            stack_pass(x0, folded, ln_fold)
        torch.cuda.synchronize()
        assert cm.clearmoe_layer_status(h) == 0
        ev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(K)]
        if dist:
            dist.barrier()
        torch.cuda.synchronize()
        for k in range(K):
            ev[k][0].record()
            stack_pass(x0, folded, ln_fold)
            ev[k][1].record()
        torch.cuda.synchronize()
        assert cm.clearmoe_layer_status(h) == 0
        ms = max_over_ranks(float(sum(e[0].elapsed_time(e[1]) for e in ev)), dist)
        return ms / K

    K = max(1, min(args.steps, 50))
    ms = timed(K)
    res = {"workload": sh.name, "T": T, "d": sh.d, "H": sh.H, "E": sh.E, "r": sh.r, "layers": sh.layers,
           "moe_layers": list(sh.moe_layers), "value": whole_job_rate(T, world, 1, ms), "unit": "tokens/s",
           "ms_per_step": ms, "steps": K,
           "l2": "no flush: each pass reads 155 MB of tokens and ~100 MB of weights (> L2)",
           "gpu_launches_per_pass": 6 * 4 + 6 * 2 + 12}
    if with_variants:
        for G in layers:  # the folded form of the same stack (each converted sublayer's basis folded once)
            if G["moe"]:
                G["W_comb"] = torch.empty_like(G["residuals"])
                cm.clearmoe_fold_basis(h, G["U"], G["S"], G["Vh"], G["residuals"], G["W_comb"])
        for key, kw in (("folded", dict(folded=True)), ("layernorm_folded", dict(ln_fold=True)),
                        ("folded_and_layernorm_folded", dict(folded=True, ln_fold=True))):
            v = timed(K, **kw)
            res[key] = {"value": whole_job_rate(T, world, 1, v), "unit": "tokens/s", "ms_per_step": v}
    # end to end: the tokens copied in from pinned host memory, the last output copied back
    xh = x0.cpu().pin_memory()
    outh = torch.empty(x0.shape, dtype=x0.dtype).pin_memory()
    xd = torch.empty_like(x0)
    Ke = max(1, min(K, 10))
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    e0.record()
    for _ in range(Ke):
        xd.copy_(xh, non_blocking=True)
        outh.copy_(stack_pass(xd), non_blocking=True)
    e1.record()
    torch.cuda.synchronize()
    res["e2e"] = {"value": whole_job_rate(T, world, Ke, max_over_ranks(e0.elapsed_time(e1), dist)),
                  "unit": "tokens/s", "h2d_bytes_per_step": int(x0.numel() * 2),
                  "d2h_bytes_per_step": int(x0.numel() * 2), "note": "copies not overlapped with compute"}
    if with_cpu and rank == 0 and world == 1:
        from oracle import clearmoe as O
        n = 2048
        t0 = time.perf_counter()
        xs = S["x"][:n].astype(np.float64)
        for L in S["layers"]:
            xs = O.stack_next_input(O.stack_layer(xs, L))
        el = time.perf_counter() - t0
        res["cpu_baseline"] = {"value": n / el, "unit": "tokens/s", "cores": blas_threads(), "kind": "oracle",
                               "sample": f"the first {n} tokens through all 12 sublayers ({el:.1f} s; float64 oracle)"}
    cm.clearmoe_layer_destroy(h)
    return res


def _gpu_setup():
    import torch

    import __graft_entry__
    from paper_2606_28516_gb300 import clearmoe as cm
    world, rank, local, dist = init_replicas("nccl")
    torch.cuda.set_device(local)
    if rank == 0:
        __graft_entry__.build()
    if dist:
        dist.barrier()
    cm.lib()
    return cm, world, rank, local, dist


def run_sweep(args):
    cm, world, rank, local, dist = _gpu_setup()
    flush = L2Flush()
    with ClockSampler(local) as clk:
        res = sweep_block(args, world, rank, dist, flush, cm)
    if rank == 0:
        print(json.dumps({
            "metric": "CLEAR-MoE FFN tokens/sec/layer over the E x r sweep (DeiT-S shape, Zipf cluster sizes)",
            "value": res["value"], "unit": "tokens/s", "n_gpus": world, "steps": res["steps"],
            "warmup": args.warmup, "ms_per_step": res["ms_per_step"], "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {k: res[k] for k in ("workload", "T", "d", "H", "E", "r", "sizes", "n_cal", "value_is")}
            | {"l2": "flushed between steps (zero-fill, then a read of another buffer)",
               "parallelism": f"replicas{world}"},
            "points": res["points"], "dense_ffn": res["dense_ffn"], "clocks": clk.summary(),
            "gpu_launches": 4 * res["steps"] * len(res["points"]),
        }), flush=True)
    if dist:
        dist.destroy_process_group()


def run_stack(args):
    cm, world, rank, local, dist = _gpu_setup()
    with ClockSampler(local) as clk:
        res = stack_block(args, world, rank, dist, cm, with_cpu=not args.no_cpu_baseline)
    line = {
        "metric": "ViT-B 12-sublayer FFN stack tokens/sec (6 CLEAR-MoE + 6 dense sublayers, LayerNorm between)",
        "value": res["value"], "unit": "tokens/s", "n_gpus": world, "steps": res["steps"], "warmup": args.warmup,
        "ms_per_step": res["ms_per_step"], "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16", "data": "synthetic",
        "config": {k: res[k] for k in ("workload", "T", "d", "H", "E", "r", "layers", "moe_layers", "l2")}
        | {"parallelism": f"replicas{world}"},
        "e2e": res["e2e"], "gpu_launches": res["gpu_launches_per_pass"] * res["steps"],
        "cpu_baseline": res.get("cpu_baseline"), "clocks": clk.summary(),
    }
    for k in ("folded", "layernorm_folded", "folded_and_layernorm_folded"):
        line[k] = res.get(k)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="deit_base_bf16", choices=sorted(workloads()))
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=200)
    ap.add_argument("--ref-budget-s", type=float, default=60.0,
                    help="--impl reference: CPU seconds the oracle's warm-up and timed steps take in total")
    ap.add_argument("--no-variants", action="store_true",
                    help="skip the variant timings (folded, materialised, class tokens, MLP router, one residual)")
    ap.add_argument("--no-other-configs", action="store_true",
                    help="skip the other workloads (DeiT-T, DeiT-S, the sweep, the stack) in the headline line")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)
    if args.impl == "reference":
        return run_reference(args)
    if args.workload == "vit_base_stack12":
        return run_stack(args)
    if args.workload == "deit_small_zipf_sweep":
        return run_sweep(args)

    import torch

    import synth
    cm, world, rank, local, dist = _gpu_setup()
    pk, pk_src = peaks()

    shape = workloads()[args.workload].with_(seed=rank)
    L = synth.make_layer(shape)
    D = synth.to_torch(L)
    s = shape
    dt = cm.BF16 if s.dtype == "bf16" else cm.F32
    h = cm.clearmoe_layer_create(s.T, s.d, s.H, s.E, s.r, dt)
    out = torch.empty(s.T, s.d, device="cuda", dtype=D["x"].dtype)
    flush = L2Flush()
    stream = torch.cuda.current_stream()

    def forward(x=None):
        cm.clearmoe_ffn_forward(h, D["x"] if x is None else x, D["W1"], D["b1"], D["U"], D["S"],
                                D["Vh"], D["residuals"], D["Wg"], D["bg"], out)

    for _ in range(args.warmup):
        flush()
        forward()
    torch.cuda.synchronize()
    assert cm.clearmoe_layer_status(h) == 0

    # Headline: K forwards, each bracketed by events on the launching stream and nothing between
    # its kernels (an event between two launches would cancel the programmatic launch overlap of
    # the GEMM kernels). The L2 flush before each step lies outside the events.
    K = args.steps
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(K)]
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        wall0 = time.perf_counter()
        for k in range(K):
            flush()
            ev[k][0].record(stream)
            forward()
            ev[k][1].record(stream)
        torch.cuda.synchronize()
        wall = time.perf_counter() - wall0
    if dist:
        dist.barrier()
    assert cm.clearmoe_layer_status(h) == 0
    step_ms = [ev[k][0].elapsed_time(ev[k][1]) for k in range(K)]
    total_ms = max_over_ranks(float(sum(step_ms)), dist)
    value = whole_job_rate(s.T, world, K, total_ms)

    # Per-kernel durations (roofline, stage breakdown): a second timed pass with an event between
    # consecutive kernels, recorded by the library on the launching stream.
    Ks = min(K, 300)
    stage_ms = stage_pass(cm, h, forward, Ks, flush)
    floor_us = launch_floor_us(flush)
    assert cm.clearmoe_layer_status(h) == 0

    # Variants of the same layer, same timing rules (events around each forward only, L2 flushed
    # before each). Reported beside the headline, not as it.
    def time_variant(fn, note):
        v_ms = max_over_ranks(statistics.mean(time_steps(fn, min(K, 300), args.warmup, flush, stream)), dist)
        assert cm.clearmoe_layer_status(h) == 0
        return {"value": whole_job_rate(s.T, world, 1, v_ms), "unit": "tokens/s", "ms_per_step": v_ms,
                "note": note}

    folded = materialized = class_tokens = mlp_router = scaled = layernorm = router_in_fc1 = None
    if s.dtype == "bf16" and not args.no_variants:
        fused = lambda: cm.clearmoe_ffn_forward_ex(h, D["x"], D["W1"], D["b1"], D["U"], D["S"], D["Vh"],
                                                   D["residuals"], D["Wg"], D["bg"], out, router_in_fc1=True)
        router_in_fc1 = time_variant(
            fused, "the router's logits inside fc1 (one 256 x 32 MMA unit per 256-token tile on the x tiles "
                   "fc1 loads), a slot kernel over 128-token ranges, t stored at the slots, z rows gathered "
                   "by perm in the grouped GEMM (TMA four-row gathers)")
        fst = stage_pass(cm, h, fused, min(K, 300), flush)
        router_in_fc1["stages_us"] = {name: statistics.mean(v) * 1e3 for name, v in
                                      zip(("fc1_with_router", "slots", "basis", "grouped"), fst.values())}
        fw = stage_work(s)
        router_in_fc1["stages_us"]["fc1_with_router_tensor_frac"] = (
            (fw["fc1_gelu"]["flops"] + fw["route"]["flops"]) / (router_in_fc1["stages_us"]["fc1_with_router"] * 1e-6)
            / 1e12 / pk["bf16_tflops"])
        W_comb = torch.empty_like(D["residuals"])
        cm.clearmoe_fold_basis(h, D["U"], D["S"], D["Vh"], D["residuals"], W_comb)
        folded = time_variant(
            lambda: cm.clearmoe_ffn_forward_folded(h, D["x"], D["W1"], D["b1"], W_comb, D["Wg"], D["bg"], out),
            "W_e^comb = U_r diag(S_r) V_r^T + W_e^res formed once (clearmoe_fold_basis); "
            "forward = routing, fc1, one grouped GEMM over z")
        del W_comb
        W_sh = torch.empty(s.d, s.H, device="cuda", dtype=D["x"].dtype)
        cm.clearmoe_materialize_basis(h, D["U"], D["S"], D["Vh"], W_sh)
        materialized = time_variant(
            lambda: cm.clearmoe_ffn_forward_materialized(h, D["x"], D["W1"], D["b1"], W_sh, D["residuals"],
                                                         D["Wg"], D["bg"], out),
            "the paper's materialised W_shared (clearmoe_materialize_basis once); grouped K chain "
            "[z | z] x [W_e^res | W_shared]")
        del W_sh
        class_tokens = time_variant(
            lambda: cm.clearmoe_ffn_forward_ex(h, D["x"], D["W1"], D["b1"], D["U"], D["S"], D["Vh"],
                                               D["residuals"], D["Wg"], D["bg"], out, b2=D["b2"], W2=D["W2"],
                                               cls_stride=197),
            "class token of each 197-token image on the dense path (W2), fc2 bias b2 added")
        scaled = time_variant(
            lambda: cm.clearmoe_ffn_forward_scaled(h, D["x"], D["W1"], D["b1"], D["U"], D["S"], D["Vh"], D["R"],
                                                   D["scales"], D["Wg"], D["bg"], out),
            "Algorithm 2's residuals as s_e R: one residual matrix, token order, no sort or scatter")
        M = synth.to_torch(synth.mlp_router(L, act="gelu") | {"dtype": s.dtype})
        mlp = cm.mlp_router(M["W_in"], M["b_in"], M["W_out"], M["b_out"], "gelu")
        mlp_router = time_variant(
            lambda: cm.clearmoe_ffn_forward_ex(h, D["x"], D["W1"], D["b1"], D["U"], D["S"], D["Vh"],
                                               D["residuals"], None, None, out, mlp=mlp, E=s.E),
            f"MLP router d -> {s.d // 6} -> E (GELU) in place of the linear router")
        # The sublayer's input as the LayerNorm of an un-normalised stream y: the LayerNorm kernel
        # then the forward, against the forward with the LayerNorm folded in (input_layernorm).
        try:
            y_in = synth.to_torch({"x": synth.residual_stream(L["x"], s.dtype), "dtype": s.dtype})["x"]
            x_ln = torch.empty_like(y_in)
            layernorm = {
                "layernorm_then_forward": time_variant(
                    lambda: (cm.clearmoe_layer_norm(h, y_in, x_ln),
                             cm.clearmoe_ffn_forward(h, x_ln, D["W1"], D["b1"], D["U"], D["S"], D["Vh"],
                                                     D["residuals"], D["Wg"], D["bg"], out)),
                    "clearmoe_layer_norm(y) into a T x d buffer, then the forward on it"),
                "layernorm_folded": time_variant(
                    lambda: cm.clearmoe_ffn_forward_ex(h, y_in, D["W1"], D["b1"], D["U"], D["S"], D["Vh"],
                                                       D["residuals"], D["Wg"], D["bg"], out,
                                                       input_layernorm=True),
                    "input_layernorm: per-token statistics and fc1's augmentation block in one launch; "
                    "the router and fc1 read y itself"),
            }
            del y_in, x_ln
        except (cm.ClearMoEError, RuntimeError, TypeError, NameError, KeyError) as exc:
            layernorm = {"error": f"{type(exc).__name__}: {exc}"}

    # same-GPU dense FFN, same timing rules (events around each forward only)
    dout = torch.empty_like(out)
    dense_ms = time_steps(lambda: cm.clearmoe_dense_ffn_forward(h, D["x"], D["W1"], D["b1"], D["W2"], dout),
                          min(K, 300), args.warmup, flush, stream)
    dense_value = whole_job_rate(s.T, world, 1, max_over_ranks(statistics.mean(dense_ms), dist))

    # End to end through the C ABI with host buffers: every step copies its tokens from pinned
    # host memory and its output back. Steps are pipelined over three streams (copy-in of step
    # k + 1 and copy-out of step k - 1 overlap the forward of step k), with double buffers.
    Ke = max(1, min(args.e2e_steps, K))
    x_host = D["x"].cpu().pin_memory()
    out_host = [torch.empty(out.shape, dtype=out.dtype).pin_memory() for _ in range(2)]
    x_dev = [torch.empty_like(D["x"]) for _ in range(2)]
    o_dev = [torch.empty_like(out) for _ in range(2)]
    s_in, s_cmp, s_out = torch.cuda.Stream(), torch.cuda.Stream(), torch.cuda.Stream()
    mk = lambda: torch.cuda.Event()
    x_ready, x_free = [mk(), mk()], [mk(), mk()]
    o_ready, o_free = [mk(), mk()], [mk(), mk()]
    e2e_t0, e2e_t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()

    def e2e_steps(n, timed):
        for k in range(n):
            b = k & 1
            with torch.cuda.stream(s_in):
                if k == 0 and timed:
                    e2e_t0.record(s_in)
                if k >= 2:
                    s_in.wait_event(x_free[b])
                x_dev[b].copy_(x_host, non_blocking=True)
                x_ready[b].record(s_in)
            with torch.cuda.stream(s_cmp):
                s_cmp.wait_event(x_ready[b])
                if k >= 2:
                    s_cmp.wait_event(o_free[b])
                cm.clearmoe_ffn_forward(h, x_dev[b], D["W1"], D["b1"], D["U"], D["S"], D["Vh"],
                                        D["residuals"], D["Wg"], D["bg"], o_dev[b], stream=s_cmp)
                x_free[b].record(s_cmp)
                o_ready[b].record(s_cmp)
            with torch.cuda.stream(s_out):
                s_out.wait_event(o_ready[b])
                out_host[b].copy_(o_dev[b], non_blocking=True)
                o_free[b].record(s_out)
                if k == n - 1 and timed:
                    e2e_t1.record(s_out)
        torch.cuda.synchronize()

    e2e_steps(args.warmup, False)
    if dist:
        dist.barrier()
    e2e_steps(Ke, True)
    e2e_ms = e2e_t0.elapsed_time(e2e_t1)
    if not torch.equal(out_host[(Ke - 1) & 1].cuda(), o_dev[(Ke - 1) & 1]):
        raise RuntimeError("end-to-end output copy mismatch")
    e2e_ms = max_over_ranks(e2e_ms, dist)
    e2e_value = whole_job_rate(s.T, world, Ke, e2e_ms)
    assert cm.clearmoe_layer_status(h) == 0
    cm.clearmoe_layer_destroy(h)
    del x_host, out_host, x_dev, o_dev, dout

    per_stage = stage_summary(s, stage_ms, pk, floor_us)
    avg = {st: statistics.mean(v) for st, v in stage_ms.items()}
    dom = max(avg, key=avg.get)
    work = stage_work(s)
    dur_s = avg[dom] / 1e3
    if dom == "route":
        ach = work[dom]["bytes"] / dur_s / 1e9
        roof = {"bound": "hbm", "achieved": ach, "peak": pk["hbm_gbs"], "unit": "GB/s"}
    else:  # the stage pass is sub-second: the burst peak; the sustained one beside it
        ach = work[dom]["flops"] / dur_s / 1e12
        scale = 1.0 if s.dtype == "bf16" else TF32X3_OF_BF16  # fp32: three TF32 products each
        roof = {"bound": "tensor", "achieved": ach, "peak": pk["bf16_tflops"] * scale, "unit": "TFLOP/s",
                "frac_sustained": ach / (pk["bf16_tflops_sustained"] * scale)}
    roof["frac"] = roof["achieved"] / roof["peak"]
    # the traffic table and kernel names are the bf16 layer's (the DeiT-B capture)
    tr = TRAFFIC.get(dom) if s.dtype == "bf16" else None
    roof["traffic"] = tr["bytes"] if tr and tr["src"] == source_hash(dom) else None
    if tr and roof["traffic"] is None:
        roof["traffic_note"] = ("the kernel's sources changed after its ncu capture "
                                f"(hash {source_hash(dom)} vs {tr['src']}): not re-captured yet")
    if s.dtype == "bf16":
        roof["kernel"] = KERNEL_OF_STAGE[dom]
        roof["peak_source"] = (f"{pk_src} ({'burst bf16: the stage pass is sub-second' if roof['bound'] == 'tensor' else 'HBM copy'})")
    else:
        roof["kernel"] = ("cm::route_f32_kernel" if dom == "route" else
                          "cm::tc_gemm_kernel<BN, mode, true> (fp32 operands, three TF32 products)")
        roof["peak_source"] = (f"{pk_src} (HBM copy)" if dom == "route" else
                               f"{pk_src} burst bf16 x nominal TF32 / bf16 (1.1 / 2.25) / 3")
    for st in STAGES:  # per-kernel DRAM traffic where the committed capture still applies
        t = TRAFFIC.get(st) if s.dtype == "bf16" else None
        per_stage[st]["traffic"] = t["bytes"] if t and t["src"] == source_hash(st) else None

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        rate, n, el = oracle_rate(L, budget_s=12.0)
        cpu = {"value": rate, "unit": "tokens/s", "cores": blas_threads(), "kind": "oracle",
               "sample": f"first {n} tokens of the workload in 1,024-token chunks ({el:.1f} s; "
                         f"float64 numpy oracle, routing + Algorithm 3)"}
        try:
            cpu["c_oracle"] = c_oracle_rates(L, budget_s=16.0)
        except (OSError, RuntimeError) as exc:  # no C compiler on the host
            cpu["c_oracle"] = {"error": f"{type(exc).__name__}: {exc}"}

    # The other workloads, each with its own figures (not part of the headline's timed region)
    configs = None
    if not args.no_other_configs and args.workload == "deit_base_bf16":
        configs = {}
        for name, sh in (("deit_tiny_fp32", synth.DEIT_TINY_FP32), ("deit_small_bf16", synth.DEIT_SMALL_BF16)):
            Lc = synth.make_layer(sh.with_(seed=rank))
            Dc = synth.to_torch(Lc)
            hc = cm.clearmoe_layer_create(sh.T, sh.d, sh.H, sh.E, sh.r, cm.BF16 if sh.dtype == "bf16" else cm.F32)
            configs[name], _ = layer_block(sh, Dc, hc, cm, args, world, dist, flush, stream, pk)
            cm.clearmoe_layer_destroy(hc)
            del Dc, Lc
        configs["deit_small_zipf_sweep"] = sweep_block(args, world, rank, dist, flush, cm)
        configs["vit_base_stack12"] = stack_block(args, world, rank, dist, cm, with_variants=False)

    mean_step = total_ms / K
    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": K,
        "warmup": args.warmup, "ms_per_step": mean_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": s.dtype, "data": "synthetic",
        "config": {"workload": s.name, "T": s.T, "d": s.d, "H": s.H, "E": s.E, "r": s.r,
                   "tokens": "Gaussian-mixture ViT tokens, layer-normalised; weights N(0, 0.02^2) "
                             "converted by truncated SVD + k-means (seeded)",
                   "l2": "flushed before every step outside the timed events: 256 MB zero-fill, then "
                         "a 512 MB read of another buffer (no dirty lines left for the step)",
                   "parallelism": f"replicas{world}"},
        "e2e": {"value": e2e_value, "unit": "tokens/s",
                "h2d_bytes_per_step": int(D["x"].numel() * D["x"].element_size()),
                "d2h_bytes_per_step": int(out.numel() * out.element_size())},
        "gpu_launches": 4 * K,
        "roofline": roof,
        "cpu_baseline": cpu,
        "clocks": clk.summary(),
        "stages": per_stage,
        "stage_timing": f"separate pass of {Ks} steps with an event between consecutive kernels "
                        "(which also cancels their programmatic launch overlap)",
        "layer_roofline_frac": layer_roofline_s(s, pk, "bf16_tflops") / (mean_step / 1e3),
        "layer_roofline_frac_sustained": layer_roofline_s(s, pk) / (mean_step / 1e3),
        "layer_roofline_frac_nominal": layer_roofline_s(
            s, {"bf16_tflops_sustained": NOMINAL_PEAKS["bf16_tflops"], "hbm_gbs": NOMINAL_PEAKS["hbm_gbs"]})
        / (mean_step / 1e3),
        "dense_ffn": {"value": dense_value, "unit": "tokens/s",
                      "ms_per_step": statistics.mean(dense_ms)},
        "folded": folded,
        "materialized": materialized,
        "class_tokens": class_tokens,
        "mlp_router": mlp_router,
        "scaled_residual": scaled,
        "input_layernorm": layernorm,
        "router_in_fc1": router_in_fc1,
        "configs": configs,
        "wall_s_timed": wall,
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
