#!/usr/bin/env python3
"""Benchmark: decoded queries/s of the neural-texture decode on one GB300.

Headline workload (one "step" = one ntc_decode over one batch): 4 frames of a
3840x2160 G-buffer query stream -- 33,177,600 queries from 2000 Voronoi regions
over 512 texture sets of 2048^2 (latents 1024^2x8 + 512^2x8 fp16 with their mip
chains, 13.3 GiB), 8 shared decoders 16->128->128->9, a continuous lod per
region in [0, 3) (trilinear: two mips per latent grid).  Inputs are resident in
HBM; L2 is flushed (a 256 MiB write, then a 256 MiB read of another buffer, so
no dirty flush lines are written back inside a step) before every timed step
and the flush is outside the step's CUDA events.

The same JSON line carries every other workload (a 256^2 texel-centre raster,
4M uniform queries over 16 decoders, the 1080p and 2160p G-buffers under each
of their decoder groupings), the unsorted mma.sync ("divergent") and per-lane
FMA ("divergent_fma") kernels on the headline batch, a sweep over exactly d
distinct decoders per warp, a mirror of the paper's Tables 5-6, the decode
under the groupings of Table 2, and Sec. 4's own decoder shape.

``--impl reference`` times the CPU oracle instead (the only other code that
computes the same result) on a bounded, evenly spaced query sample.

Multi-GPU (torchrun): every rank decodes its own query stream of the same
recipe against a full replica of the assets -- queries are independent, so
there is no collective on the data path (weak scaling); the step time is the
max over ranks.
"""
from __future__ import annotations

import argparse
import ctypes
import hashlib
import re
import json
import os
import statistics
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "decoded queries/sec on 1 GB300 vs distinct decoders per warp; % of roofline"
UNIT = "queries/s"
HEADLINE = "gbuffer-2160p-x4-trilinear"
DESCRIPTIONS = {
    "gbuffer-2160p-x4-trilinear": "gbuffer-2160p-x4-trilinear: 4 frames of a 3840x2160 G-buffer (33,177,600 queries, "
                                  "2000 Voronoi regions, lod ~U[0,3) per region, trilinear) over 512 texture sets of "
                                  "2048^2 (latents 1024^2x8 + 512^2x8 fp16 with mip chains), 8 decoders "
                                  "16->128->128->9 (random partition)",
    "uniform-4m": "uniform-4m: 16 texture sets of 1024^2 (latents 512^2x8 + 256^2x8 fp16), 16 decoders "
                  "16->64->64->8 (one per set), 4,194,304 queries: uniform set id, uniform UV, lod 0",
}
L2_FLUSH_BYTES = 256 << 20
KERNEL_NAMES = {("bucketed", False): "k_decode_tm (tcgen05/TMEM gather-decode)",
                ("bucketed", True): "k_decode_fp32 (FFMA gather-decode)",
                ("bucketed_mma", False): "k_decode_mma (mma.sync gather-decode)",
                ("divergent", False): "k_decode_divergent (mma.sync, unsorted)",
                ("divergent_fma", False): "k_decode_divergent_fma (per-lane FFMA, unsorted)",
                ("divergent_fma", True): "k_decode_divergent_fma (per-lane FFMA, unsorted)"}
NAMED = ("raster-256", "uniform-4m", "gbuffer-1080p", "gbuffer-2160p", "gbuffer-2160p-x4-trilinear")


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=20)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", default="ntc", choices=["ntc", "reference"])
    p.add_argument("--mode", default="bucketed", choices=["bucketed", "bucketed_mma", "divergent", "divergent_fma"])
    p.add_argument("--precision", default="fp16", choices=["fp16", "bf16", "fp32"])
    p.add_argument("--workload", default=HEADLINE, choices=list(NAMED) + ["paper-decoder"],
                   help="the timed batch (default: the 4-frame 2160p trilinear G-buffer); paper-decoder is "
                        "Sec. 4's decoder (256^2x4 grid, positional encoding, LeakyReLU, 64x3) on a 1080p G-buffer")
    p.add_argument("--variant", default=None, help="decoder grouping of the timed gbuffer-1080p / gbuffer-2160p batch")
    p.add_argument("--no-workloads", action="store_true", help="skip the per-workload table")
    p.add_argument("--no-sweep", action="store_true", help="skip the decoders-per-warp sweep")
    p.add_argument("--no-cpu", action="store_true", help="skip the CPU oracle baseline")
    p.add_argument("--no-mirror", action="store_true", help="skip the mirror of the paper's Tables 5-6")
    p.add_argument("--no-maps", action="store_true", help="skip the Table 2 groupings of a 586-set workload")
    p.add_argument("--no-variants", action="store_true", help="skip Sec. 4's decoder shape")
    p.add_argument("--no-fp16-out", action="store_true", help="skip the fp16-output-row step")
    p.add_argument("--variants", action="store_true", help="also time every A x B size of Sec. 4's MLP ablation")
    p.add_argument("--small", action="store_true", help="the small size of the timed workload")
    p.add_argument("--medium", action="store_true",
                   help="the profiling size of gbuffer-2160p-x4-trilinear: one frame over 32 sets (a few GB)")
    a = p.parse_args()
    a.size = "small" if a.small else ("medium" if a.medium else "full")
    a.small = a.small or a.medium  # every reduced size skips the other legs
    return a


# ------------------------------------------------------------------ clocks

class ClockSampler:
    """Polls NVML (read-only) for SM clock and clock-event reasons."""
    REASONS = {0x1: "gpu_idle", 0x2: "applications_clocks_setting", 0x4: "sw_power_cap",
               0x8: "hw_slowdown", 0x10: "sync_boost", 0x20: "sw_thermal_slowdown",
               0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown",
               0x100: "display_clock_setting"}

    def __init__(self, index: int):
        self.ok = False
        self.samples = []
        try:
            self.nvml = ctypes.CDLL("libnvidia-ml.so.1")
            if self.nvml.nvmlInit_v2() != 0:
                return
            self.h = ctypes.c_void_p()
            if self.nvml.nvmlDeviceGetHandleByIndex_v2(ctypes.c_uint(index), ctypes.byref(self.h)) != 0:
                return
            mx = ctypes.c_uint()
            self.nvml.nvmlDeviceGetMaxClockInfo(self.h, 1, ctypes.byref(mx))  # 1 = SM clock
            self.max_mhz = int(mx.value)
            self.ok = True
        except OSError:
            pass

    def _poll(self):
        clk, rs, pw = ctypes.c_uint(), ctypes.c_ulonglong(), ctypes.c_uint()
        while not self._stop.is_set():
            self.nvml.nvmlDeviceGetClockInfo(self.h, 1, ctypes.byref(clk))
            self.nvml.nvmlDeviceGetCurrentClocksEventReasons(self.h, ctypes.byref(rs))
            self.nvml.nvmlDeviceGetPowerUsage(self.h, ctypes.byref(pw))
            self.samples.append((int(clk.value), int(rs.value), pw.value / 1000.0))
            time.sleep(0.002)

    def start(self):
        if not self.ok:
            return
        self._stop = threading.Event()
        self._t = threading.Thread(target=self._poll, daemon=True)
        self._t.start()

    def stop(self):
        if not self.ok:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvml unavailable"]}
        self._stop.set()
        self._t.join()
        s = self.samples
        bits = 0
        for _, r, _ in s:
            bits |= r
        reasons = sorted(v for k, v in self.REASONS.items() if bits & k)
        return {"sm_mhz": statistics.median(c for c, _, _ in s) if s else None,
                "sm_max_mhz": self.max_mhz, "reasons": reasons, "samples": len(s),
                "power_w_max": max((p for _, _, p in s), default=None)}


# --------------------------------------------------------------- helpers

def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


# the sources each recorded decode kernel is built from
KERNEL_SOURCES = {
    "k_decode_tm": ("decode_tc.cuh", "decode_tc.cu", "tcgen05.cuh", "ntc_internal.cuh"),
    "k_decode_gen_tc": ("decode_gen.cu", "tcgen05.cuh", "ntc_internal.cuh"),
}


def kernel_source_hash(kernel):
    """Hash of one decode kernel's sources with comments and blank space
    removed, so a comment edit does not detach the recorded DRAM traffic."""
    h = hashlib.sha1()
    for f in KERNEL_SOURCES[kernel]:
        with open(os.path.join(ROOT, "paper_2608_27888_gb300", "csrc", f)) as fh:
            src = fh.read()
        src = re.sub(r"/\*.*?\*/", " ", src, flags=re.S)
        src = re.sub(r"//[^\n]*", " ", src)
        h.update(" ".join(src.split()).encode())
    return h.hexdigest()[:12]


def recorded_traffic(kernel, workload):
    """DRAM bytes per decode launch from the committed ncu summary, if it was
    taken on the current kernel source (a capture on a reduced case is scaled
    to the full launch by its query count, as the record says)."""
    path = os.path.join(ROOT, "profiles", "decode_traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f)
        r = rec.get(f"{kernel}:{workload}")
        if r and r.get("source_hash") == kernel_source_hash(kernel):
            return float(r["dram_bytes_per_launch"])
    except Exception:
        pass
    return None


def compulsory(workload):
    """The oracle's count of the bytes a decode of this workload must move
    (tests/golden/compulsory_bytes.json, written by make_compulsory.py)."""
    try:
        with open(os.path.join(ROOT, "tests", "golden", "compulsory_bytes.json")) as f:
            return json.load(f)["workloads"].get(workload)
    except Exception:
        return None


def cpu_model():
    """The host CPU as /proc/cpuinfo names it (Arm parts by implementer/part)."""
    arm_parts = {0xd4f: "Neoverse-V2", 0xd40: "Neoverse-V1", 0xd0c: "Neoverse-N1", 0xd49: "Neoverse-N2"}
    try:
        txt = open("/proc/cpuinfo").read()
    except OSError:
        return "unknown"
    m = re.search(r"^model name\s*:\s*(.+)$", txt, re.M)
    if m:
        return m.group(1).strip()
    imp = re.search(r"^CPU implementer\s*:\s*(\S+)", txt, re.M)
    part = re.search(r"^CPU part\s*:\s*(\S+)", txt, re.M)
    if part:
        p = int(part.group(1), 16)
        name = arm_parts.get(p, f"part {part.group(1)}")
        return f"{'Arm ' if imp and imp.group(1) == '0x41' else ''}{name}"
    return "unknown"


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def shape_costs(a, q):
    """Algorithmic bytes and FLOPs per query of a workload: the query record,
    every tap's latent texel (both mips when the lod is fractional), the fp32
    outputs; 2 x the MACs of the MLP; and the fp16 weights of every decoder."""
    tri = a.num_mips > 1 and bool((q["lod"] != np.floor(q["lod"])).any())
    bpq = 16 + (2 if tri else 1) * a.num_levels * 4 * a.channels * 2 + 4 * a.out_dim
    H = a.hidden
    flops = 2 * (a.in_dim * H + (a.num_hidden_layers - 1) * H * H + H * a.out_dim)
    w_bytes = a.num_decoders * (a.in_dim * H + (a.num_hidden_layers - 1) * H * H + a.out_dim * H) * 2
    return bpq, flops, w_bytes


def workload(name: str, small, rank: int, variant=None):
    """The benchmark batch of one rank: the same assets on every rank, a
    rank-specific query stream of the same recipe (queries are sharded, assets
    replicated).  small: True / "small", "medium", or False / "full"."""
    from paper_2608_27888_gb300 import workloads as W
    size = small if isinstance(small, str) else ("small" if small else "full")
    if name == "paper-decoder":
        return W.paper_decoder("small" if size != "full" else "full")
    return W.named(name, size, variant, query_tag=rank if size != "medium" else 0)


def aggregate(n_per_rank: int, ms_local: float, dist=None):
    """Whole-job throughput: all ranks' queries over the slowest rank's step time."""
    ws = 1
    ms = ms_local
    if dist is not None and dist.is_initialized():
        import torch
        ws = dist.get_world_size()
        t = torch.tensor([ms_local], dtype=torch.float64,
                         device="cuda" if dist.get_backend() == "nccl" else "cpu")
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ms = float(t.item())
    return n_per_rank * ws / (ms / 1e3), ms


def mean_distinct(q, assets):
    d = assets.set_to_decoder[q["set_id"]]
    nw = len(d) // 32
    x = np.sort(d[:nw * 32].reshape(nw, 32), axis=1)
    return float((1 + (np.diff(x, axis=1) != 0).sum(1)).mean())


# -------------------------------------------------------------- reference arm

def ordinal(k: int) -> str:
    """1st, 2nd, 3rd, 4th, ..., 11th, 12th, 13th, 21st, 31st."""
    suf = "th" if 10 <= k % 100 <= 20 else {1: "st", 2: "nd", 3: "rd"}.get(k % 10, "th")
    return f"{k}{suf}"


def cpu_sample(q):
    """The bounded CPU sample of a batch: every (n // 2^20)-th query (every
    31st of the headline's 33.2M, 1.07M queries), so it spans every frame and
    region."""
    stride = max(1, len(q) // (1 << 20))
    return q[::stride], stride


def run_reference(args, ws, rank):
    if rank != 0:
        return
    import oracle
    w = workload(args.workload, args.size, 0, args.variant)
    q, stride = cpu_sample(w.queries)
    sample = len(q)
    cores = os.cpu_count() or 1
    for _ in range(max(0, args.warmup)):
        oracle.decode(w.assets, q[:4096], nthreads=cores)
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        oracle.decode(w.assets, q, nthreads=cores)
        times.append(time.perf_counter() - t0)
    ms = 1e3 * statistics.mean(times)
    value = sample / (ms / 1e3)
    desc = (f"every {ordinal(stride)} query of the workload ({sample:,} of {len(w.queries):,}) per step, oracle on "
            f"{cores} host threads ({cpu_model()})")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": DESCRIPTIONS.get(args.workload, w.name), "sample_queries": sample},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "cpu_model": cpu_model(), "kind": "oracle",
                         "sample": desc},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }), flush=True)


# ------------------------------------------------------------------- GPU arm

def main():
    args = parse()
    ws, rank, local = dist_env()
    if args.impl == "reference":
        run_reference(args, ws, rank)
        return
    import torch
    torch.cuda.set_device(local)
    dist = None
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    from paper_2608_27888_gb300 import ntc

    w = workload(args.workload, args.size, rank, args.variant)
    n = len(w.queries)
    C = w.assets.out_dim
    dec = ntc.Decoder(w.assets, args.precision)
    qd = ntc.queries_to_device(w.queries)
    out = torch.empty((n, C), dtype=torch.float32, device="cuda")
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device="cuda")
    flush_rd = torch.ones(L2_FLUSH_BYTES // 4, dtype=torch.float32, device="cuda")
    stream = torch.cuda.current_stream()

    def flush_l2():
        # a write larger than L2, then a read of another buffer larger than L2:
        # none of our data and no dirty lines are left in L2 when a step starts
        flush.zero_()
        flush_rd.sum()

    def barrier():
        if dist is not None:
            dist.barrier()

    def timed_steps(mode, steps, warmup, stages=False):
        dec.set_stage_timing(stages)
        for _ in range(warmup):
            dec.decode(qd, out, mode=mode)
        torch.cuda.synchronize()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
        st_times = []
        l0 = dec.launches()
        barrier()
        torch.cuda.synchronize()
        for i in range(steps):
            flush_l2()
            ev[i][0].record(stream)
            dec.decode(qd, out, mode=mode)
            ev[i][1].record(stream)
            if stages:
                st_times.append(dec.stage_times())
        torch.cuda.synchronize()
        barrier()
        launches = dec.launches() - l0
        ms = [a.elapsed_time(b) for a, b in ev]
        dec.set_stage_timing(False)
        return ms, st_times, launches

    sampler = ClockSampler(local)
    sampler.start()
    ms, _, launches = timed_steps(args.mode, args.steps, args.warmup)
    clocks = sampler.stop()
    value, ms_step = aggregate(n, statistics.mean(ms), dist)
    # per-stage times from a second pass with the library's stage events (the
    # events sit between the kernels, so the headline pass runs without them)
    _, stages, _ = timed_steps(args.mode, args.steps, 2, stages=True)
    bucket_ms = statistics.mean(s[0] for s in stages)
    decode_ms = statistics.mean(s[1] for s in stages)

    # roofline of the dominant kernel (the gather-decode), by algorithmic bytes;
    # beside it the compulsory bytes the oracle counted (distinct texels)
    peak, peak_kind = peaks()
    bpq, flops_q, w_bytes = shape_costs(w.assets, w.queries)
    alg_bytes = n * bpq + w_bytes
    achieved = alg_bytes / (decode_ms / 1e3) / 1e9
    general = args.workload == "paper-decoder"
    kernel = "k_decode_gen_tc" if general else "k_decode_tm"
    roofline = {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                "frac": achieved / peak, "traffic": recorded_traffic(kernel, args.workload),
                "kernel": ("k_decode_gen_tc (general-shape tcgen05 gather-decode)" if general
                           else KERNEL_NAMES[(args.mode, args.precision == "fp32")]),
                "kernel_ms": decode_ms, "bucketing_ms": bucket_ms,
                "peak_kind": f"{peak_kind} HBM copy bandwidth",
                "algorithmic_bytes_per_launch": alg_bytes, "algorithmic_bytes_per_query": bpq,
                "step_frac": (n * bpq + w_bytes) / (ms_step / 1e3) / 1e9 / peak}
    comp = compulsory(args.workload) if not args.small else None
    if comp and comp["queries"] == n:
        cb = comp["compulsory_bytes_excluding_weights"] + w_bytes
        roofline["compulsory"] = {
            "bytes_per_launch": cb, "bytes_per_query": cb / n,
            "touched_texels": comp["touched_texels"],
            "achieved": cb / (decode_ms / 1e3) / 1e9, "frac": cb / (decode_ms / 1e3) / 1e9 / peak,
            "step_frac": cb / (ms_step / 1e3) / 1e9 / peak,
            "what": "queries + outputs + distinct latent texels touched (counted by the oracle) + weights"}

    # end to end through the public host-buffer call
    hq = torch.from_numpy(np.ascontiguousarray(w.queries).view(np.int32).reshape(-1, 4)).pin_memory()
    e2e_reps = max(3, min(args.steps, 10))
    e2e = end_to_end(torch, dec, hq, n, C, ws, args.mode, e2e_reps)

    # the same step with fp16 output rows (Sec. 4.4's fp16 kernels write fp16)
    out_fp16 = None
    if args.precision != "fp32" and args.mode == "bucketed" and not args.no_fp16_out:
        d16 = ntc.Decoder(w.assets, args.precision, output="fp16")
        o16 = torch.empty((n, C), dtype=torch.float16, device="cuda")
        ms16 = time_decode(torch, d16, qd, o16, "bucketed", flush, flush_rd, reps=e2e_reps, warm=2)
        out_fp16 = {"value": n * ws / (ms16 / 1e3), "unit": UNIT, "ms_per_step": ms16,
                    "output_bytes_per_query": 2 * C,
                    "e2e": end_to_end(torch, d16, hq, n, C, ws, "bucketed", e2e_reps)}
        d16.close()
        del o16, d16
    del hq

    # the in-run comparison: the unsorted kernels on the same batch
    extra = {}
    for other in ("divergent", "divergent_fma"):
        if args.mode == other or (other == "divergent" and (args.precision == "fp32" or general)):
            continue
        dms, _, _ = timed_steps(other, 3 if n > 10_000_000 else 5, 1)
        extra[other] = {"value": n * ws / (statistics.mean(dms) / 1e3), "unit": UNIT,
                        "ms_per_step": statistics.mean(dms)}
    dd = mean_distinct(w.queries, w.assets)
    headline_row = {"workload": w.name, "queries": n, "decoders": w.assets.num_decoders,
                    "hidden": w.assets.hidden, "mean_distinct_decoders_per_warp": dd,
                    "divergence_score_eq1": dd - 1.0, "bucketed": value / ws, "ms_per_step": ms_step,
                    "bucketing_ms": bucket_ms, "decode_ms": decode_ms, "bytes_per_query": bpq,
                    "roofline_rate": peak * 1e9 / bpq, "frac_of_roofline": value / ws / (peak * 1e9 / bpq),
                    **{k: v["value"] / ws for k, v in extra.items()}}
    dec.close()
    del qd, out, dec
    torch.cuda.empty_cache()

    result = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_step,
        "ms_per_step_median": statistics.median(ms), "ms_per_step_best": min(ms),
        "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f16" if args.precision == "fp16" else args.precision.replace("fp", "f"),
        "data": "synthetic",
        "config": {"workload": DESCRIPTIONS.get(args.workload, w.name) if not args.small else w.name,
                   "queries_per_gpu": n,
                   "decoders": w.assets.num_decoders, "mode": args.mode, "precision": args.precision,
                   "mean_distinct_decoders_per_warp": dd,
                   "l2": "flushed before every timed step (256 MiB write, then a 256 MiB read of another buffer; "
                         "outside the step events); inputs larger than L2",
                   "parallelism": f"{ws} independent replicas (queries sharded, no collective)"},
        "roofline": roofline, "e2e": e2e, "gpu_launches": launches, "clocks": clocks,
        **({"output_fp16": out_fp16} if out_fp16 else {}),
        "flops_per_query": flops_q, "bytes_per_query": bpq,
        **extra,
    }
    if rank == 0 and not args.small:
        if not args.no_workloads:
            result["workloads"] = per_workload(ntc, torch, args.precision, headline=(args.workload, headline_row))
        if not args.no_sweep:
            result["sweep"] = sweep(ntc, torch, args.precision)
        if not args.no_mirror and args.precision != "fp32":
            result["paper_mirror"] = paper_mirror(ntc, torch, args.precision)
        if not args.no_maps:
            result["maps"] = map_sources(ntc, torch, args.precision)
        if not args.no_variants:
            result["variants"] = decoder_variants(ntc, torch, args.precision, every_size=args.variants)
    if rank == 0 and not args.no_cpu and ws == 1:
        result["cpu_baseline"] = cpu_baseline(w)
    if rank == 0:
        print(json.dumps(result), flush=True)
    if dist is not None:
        dist.destroy_process_group()


def end_to_end(torch, dec, hq, n, C, ws, mode, reps):
    """The metric through ntc_decode_host: pinned host queries in, host output
    rows out (the context's output format), copies inside the timed region."""
    half = dec.output == "fp16"
    hout = torch.empty((n, C), dtype=torch.float16 if half else torch.float32).pin_memory()
    for _ in range(2):
        dec.decode_host(hq, hout, mode=mode)
    ts = []
    for _ in range(reps):
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        dec.decode_host(hq, hout, mode=mode)
        ts.append(time.perf_counter() - t0)
    ms = 1e3 * statistics.mean(ts)
    link = host_link_ms(torch, hq, hout, reps)
    return {"value": n * ws / (ms / 1e3), "unit": UNIT, "h2d_bytes_per_step": n * 16,
            "d2h_bytes_per_step": n * C * (2 if half else 4), "ms_per_step": ms,
            "host_link": {"copy_ms_per_step": link, "frac": link / ms,
                          "what": "the same upload and download alone, issued together on two streams "
                                  "(no decode): the bound of this end-to-end number"}}


def host_link_ms(torch, hq, hout, reps):
    """The host link's own time for one step's bytes: the query upload and the
    row download of a decode_host call, as two plain copies on two streams."""
    dq = torch.empty(hq.shape, dtype=hq.dtype, device="cuda")
    dout = torch.zeros(hout.shape, dtype=hout.dtype, device="cuda")
    up, down = torch.cuda.Stream(), torch.cuda.Stream()

    def once():
        with torch.cuda.stream(up):
            dq.copy_(hq, non_blocking=True)
        with torch.cuda.stream(down):
            hout.copy_(dout, non_blocking=True)
        torch.cuda.synchronize()

    once()
    once()
    ts = []
    for _ in range(reps):
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        once()
        ts.append(time.perf_counter() - t0)
    del dq, dout
    return 1e3 * statistics.mean(ts)


def time_decode(torch, dec, qd, out, mode, flush, flush_rd, reps=5, warm=2):
    """Mean ms of one ntc_decode on the current stream, L2 flushed before each."""
    for _ in range(warm):
        dec.decode(qd, out, mode=mode)
    ts = []
    for _ in range(reps):
        flush.zero_()
        flush_rd.sum()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        dec.decode(qd, out, mode=mode)
        e1.record()
        torch.cuda.synchronize()
        ts.append(e0.elapsed_time(e1))
    return statistics.mean(ts)


def launch_floor_ms(torch, flush, flush_rd, reps=20):
    """The step time of a kernel that does nothing (a one-element fill), timed
    as time_decode times a decode: one launch between two events after the L2
    flush.  No call that launches a kernel can take less, so for a small batch
    it caps the fraction of the roofline that any decode could reach."""
    tiny = torch.zeros(1, dtype=torch.float32, device="cuda")
    for _ in range(3):
        tiny.zero_()
    ts = []
    for _ in range(reps):
        flush.zero_()
        flush_rd.sum()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        tiny.zero_()
        e1.record()
        torch.cuda.synchronize()
        ts.append(e0.elapsed_time(e1))
    return statistics.median(ts)


def paper_mirror(ntc, torch, precision, sizes=(512, 1024, 2048, 4096, 8192), ds=(5, 10)):
    """The setting of the paper's Tables 5-6 on this GPU: an N x N texel-centre
    raster where every 32-query warp holds d distinct texture sets (32 sets of
    1024^2), decoded once with one decoder shared by all sets ("Shared-Decoder")
    and once with one decoder per set (d distinct decoders per warp).  Times in
    microseconds: shared = the warp-level mma.sync kernel on the shared map (one
    decoder per warp, no loop); wmma / fma = the unsorted mma.sync and per-lane
    FMA kernels on the per-set map ("Non-Shared WMMA / FMA"); bucketed = this
    library's default path (sort by decoder, tcgen05 decode) on the per-set map.
    avg_increase_* is the paper's statistic, mean(t_nonshared / t_shared) - 1."""
    from paper_2608_27888_gb300 import workloads as W
    S, T = 32, 1024
    seed = W.BASE_SEED + 100
    a_sh = W.make_assets(seed, S, T, 1, 1, W.map_shared(S))
    a_ns = W.make_assets(seed, S, T, 1, S, W.map_identity(S))
    dsh, dns = ntc.Decoder(a_sh, precision), ntc.Decoder(a_ns, precision)
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device="cuda")
    flush_rd = torch.ones(L2_FLUSH_BYTES // 4, dtype=torch.float32, device="cuda")
    rows = []
    for d in ds:
        for N in sizes:
            q = W.queries_controlled(seed + d, N, S, d)
            qd = ntc.queries_to_device(q)
            out = torch.empty((len(q), a_ns.out_dim), dtype=torch.float32, device="cuda")
            reps = 5 if N <= 4096 else 3
            row = {"d": d, "N": N,
                   "shared_us": 1e3 * time_decode(torch, dsh, qd, out, "divergent", flush, flush_rd, reps),
                   "shared_bucketed_us": 1e3 * time_decode(torch, dsh, qd, out, "bucketed", flush, flush_rd, reps),
                   "wmma_us": 1e3 * time_decode(torch, dns, qd, out, "divergent", flush, flush_rd, reps),
                   "fma_us": 1e3 * time_decode(torch, dns, qd, out, "divergent_fma", flush, flush_rd, reps),
                   "bucketed_us": 1e3 * time_decode(torch, dns, qd, out, "bucketed", flush, flush_rd, reps)}
            rows.append(row)
            del qd, out
    dsh.close()
    dns.close()
    summary = {}
    for d in ds:
        rs = [r for r in rows if r["d"] == d]
        for k in ("wmma", "fma", "bucketed"):
            summary[f"d{d}_avg_increase_{k}_over_shared"] = statistics.mean(
                r[f"{k}_us"] / r["shared_us"] for r in rs) - 1.0
    return {"rows": rows, "summary": summary,
            "what": "32 sets of 1024^2, N x N texel-centre raster, d distinct sets per warp; times in us"}


def decoder_variants(ntc, torch, precision, every_size=False):
    """Sec. 4's decoder (one 256x256x4 grid per set with a 4-mip chain,
    positional encoding of 4 frequencies, LeakyReLU, 64 x 3), and with
    every_size the A x B sizes of its MLP ablation (A neurons, B layers), 16
    sets in 4 clusters, on a 1920x1080 G-buffer with a continuous lod
    (trilinear).  Queries/s of the whole ntc_decode (bucketed: the general
    tcgen05 kernel for fp16/bf16) and of the per-lane FMA mode, with the
    HBM-bound rate of the algorithmic bytes."""
    from paper_2608_27888_gb300 import workloads as W
    peak, _ = peaks()
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device="cuda")
    flush_rd = torch.ones(L2_FLUSH_BYTES // 4, dtype=torch.float32, device="cuda")
    rows = []
    shapes = [(64, 3)]
    if every_size:
        shapes += [(a, b) for a in (32, 64, 128) for b in (2, 3, 4, 5) if (a, b) != (64, 3)]
    for A_, B_ in shapes:
        w = W.paper_decoder("full", hidden=A_, layers=B_ - 1)
        a, q = w.assets, w.queries
        n = len(q)
        dec = ntc.Decoder(a, precision)
        qd = ntc.queries_to_device(q)
        out = torch.empty((n, a.out_dim), dtype=torch.float32, device="cuda")
        tri = bool((q["lod"] != np.floor(q["lod"])).any())
        bpq = 16 + (2 if tri else 1) * a.num_levels * 4 * a.channels * 2 + 4 * a.out_dim
        flops = 2 * (a.in_dim * A_ + (B_ - 2) * A_ * A_ + A_ * a.out_dim)
        row = {"A": A_, "B": B_, "in_dim": a.in_dim, "queries": n, "bytes_per_query": bpq,
               "flops_per_query": flops, "roofline_rate": peak * 1e9 / bpq}
        row["bucketed"] = n / (time_decode(torch, dec, qd, out, "bucketed", flush, flush_rd, reps=10, warm=3) / 1e3)
        row["frac_of_roofline"] = row["bucketed"] / row["roofline_rate"]
        row["divergent_fma"] = n / (time_decode(torch, dec, qd, out, "divergent_fma", flush, flush_rd, reps=3,
                                                warm=1) / 1e3)
        rows.append(row)
        dec.close()
        del qd, out
        torch.cuda.empty_cache()
    return {"rows": rows, "what": "16 sets of 256^2x4 (4 mips), PE 4 frequencies, LeakyReLU, 4 decoders; "
                                  "1920x1080 G-buffer, lod in [0, 3]"}


def map_sources(ntc, torch, precision):
    """The five groupings of the paper's accuracy study (Sec. 4.1, Table 2) as a
    decode-throughput experiment: 586 texture sets of 1024^2 (4 mips; Table 1's
    dataset size), a 1920x1080 G-buffer with 600 regions, decoded with one
    decoder per set ("baseline"), one for all ("single"), k-means groups of
    synthetic 512-d embeddings computed by ntc_kmeans_map ("clustered", 11
    groups), a random grouping with the clustered group sizes ("random") and
    Table 1's categories ("category")."""
    import dataclasses
    from paper_2608_27888_gb300 import workloads as W
    seed = W.BASE_SEED + 50
    S, T, m = 586, 1024, len(W.CATEGORY_SIZES)
    F = W.embeddings(seed, W.CATEGORY_SIZES)
    km_map, _, km_it = ntc.kmeans_map(F, m, W.kmeans_init(seed, S, m))
    km_sizes = np.bincount(km_map, minlength=m)
    maps = {"baseline": (W.map_identity(S), S), "single": (W.map_shared(S), 1), "clustered": (km_map, m),
            "random": (W.map_random_sizes(seed, km_sizes), m), "category": (W.map_category(), m)}
    base = W.make_assets(seed, S, T, 4, 1, W.map_shared(S))
    q = W.queries_gbuffer(seed, 1920, 1080, 600, S, T, lod_mode=0)
    qd = ntc.queries_to_device(q)
    out = torch.empty((len(q), base.out_dim), dtype=torch.float32, device="cuda")
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device="cuda")
    flush_rd = torch.ones(L2_FLUSH_BYTES // 4, dtype=torch.float32, device="cuda")
    rows = []
    for name, (mp, D) in maps.items():
        a = dataclasses.replace(base, num_decoders=D, set_to_decoder=np.asarray(mp, dtype=np.uint32),
                                weights=W.make_weights(seed, D, base.in_dim, base.hidden, 2, base.out_dim))
        dec = ntc.Decoder(a, precision)
        dd = mean_distinct(q, a)
        row = {"map": name, "decoders": D, "group_sizes": np.bincount(mp, minlength=D).tolist() if D <= 16 else None,
               "mean_distinct_decoders_per_warp": dd, "divergence_score_eq1": dd - 1.0}
        row["bucketed"] = len(q) / (time_decode(torch, dec, qd, out, "bucketed", flush, flush_rd, reps=10, warm=3) / 1e3)
        for mode in (("divergent_fma",) if precision == "fp32" else ("divergent", "divergent_fma")):
            row[mode] = len(q) / (time_decode(torch, dec, qd, out, mode, flush, flush_rd, reps=5, warm=1) / 1e3)
        rows.append(row)
        dec.close()
        torch.cuda.empty_cache()
    return {"rows": rows, "kmeans_assignments": km_it, "queries": len(q),
            "what": "586 sets of 1024^2, 1920x1080 G-buffer, 600 regions; Gq/s of the whole ntc_decode"}


def per_workload(ntc, torch, precision, headline=None):
    """Every full-size workload under each of its decoder groupings: queries/s
    of the whole ntc_decode (bucketed), the bucketing / gather-decode split,
    the unsorted kernels, and the whole step against the roofline rate of that
    workload's algorithmic bytes and against the compulsory bytes the oracle
    counted.  The headline workload's row is the one measured above."""
    from paper_2608_27888_gb300 import workloads as W
    peak, _ = peaks()
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device="cuda")
    flush_rd = torch.ones(L2_FLUSH_BYTES // 4, dtype=torch.float32, device="cuda")
    floor_ms = launch_floor_ms(torch, flush, flush_rd)
    rows = []
    for name, variant in (("raster-256", None), ("uniform-4m", None), ("gbuffer-1080p", "identity"),
                          ("gbuffer-1080p", "clustered4"), ("gbuffer-1080p", "shared"), ("gbuffer-2160p", "128"),
                          ("gbuffer-2160p", "16"), ("gbuffer-2160p", "8"), ("gbuffer-2160p", "1"),
                          ("gbuffer-2160p-x4-trilinear", None)):
        comp = compulsory(name)
        if headline and headline[0] == name and variant is None:
            row = dict(headline[1])
        else:
            w = W.named(name, "full", variant)
            a, q = w.assets, w.queries
            n, C = len(q), a.out_dim
            dec = ntc.Decoder(a, precision)
            qd = ntc.queries_to_device(q)
            out = torch.empty((n, C), dtype=torch.float32, device="cuda")
            ms = time_decode(torch, dec, qd, out, "bucketed", flush, flush_rd, reps=10, warm=3)
            dec.set_stage_timing(True)
            st = []
            for _ in range(5):
                flush.zero_()
                flush_rd.sum()
                dec.decode(qd, out, mode="bucketed")
                st.append(dec.stage_times())
            dec.set_stage_timing(False)
            bpq, _, _ = shape_costs(a, q)
            dd = mean_distinct(q, a)
            row = {"workload": w.name, "queries": n, "decoders": a.num_decoders, "hidden": a.hidden,
                   "mean_distinct_decoders_per_warp": dd, "divergence_score_eq1": dd - 1.0,
                   "bucketed": n / (ms / 1e3), "ms_per_step": ms,
                   "bucketing_ms": statistics.mean(t[0] for t in st), "decode_ms": statistics.mean(t[1] for t in st),
                   "bytes_per_query": bpq, "roofline_rate": peak * 1e9 / bpq}
            row["frac_of_roofline"] = row["bucketed"] / row["roofline_rate"]
            reps = 3 if n > 10_000_000 else 5
            for m in (("divergent_fma",) if precision == "fp32" else ("divergent", "divergent_fma")):
                row[m] = n / (time_decode(torch, dec, qd, out, m, flush, flush_rd, reps=reps, warm=1) / 1e3)
            dec.close()
            del qd, out, w, a, q
            torch.cuda.empty_cache()
        # the best fraction a decode taking no time at all would show
        row["launch_floor_ms"] = floor_ms
        row["frac_of_roofline_cap"] = min(1.0, row["queries"] / (floor_ms / 1e3) / row["roofline_rate"])
        if comp and comp["queries"] == row["queries"]:
            cpq = comp["compulsory_bytes_per_query_excluding_weights"]
            row["compulsory_bytes_per_query"] = cpq
            row["frac_of_compulsory_roofline"] = row["bucketed"] / (peak * 1e9 / cpq)
        rows.append(row)
    return rows


def sweep(ntc, torch, precision):
    """Queries/s vs exactly d distinct decoders per warp (32 sets of 1024^2, 32
    decoders, identity map, 4096^2 texel-centre raster), bucketed vs divergent."""
    from paper_2608_27888_gb300 import workloads as W
    rows = []
    a = None
    for d in (1, 2, 4, 8, 16, 32):
        wl = W.sweep(d, 4096)
        if a is None:
            a = wl.assets
            dec = ntc.Decoder(a, precision)
        qd = ntc.queries_to_device(wl.queries)
        out = torch.empty((len(wl.queries), a.out_dim), dtype=torch.float32, device="cuda")
        flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device="cuda")
        flush_rd = torch.ones(L2_FLUSH_BYTES // 4, dtype=torch.float32, device="cuda")
        row = {"d": d}
        modes = ("bucketed", "divergent_fma") if precision == "fp32" else ("bucketed", "divergent", "divergent_fma")
        for mode in modes:
            ms = time_decode(torch, dec, qd, out, mode, flush, flush_rd, reps=5)
            row[mode] = len(wl.queries) / (ms / 1e3)
        for mode in modes[1:]:
            row[f"bucketed_over_{mode}"] = row["bucketed"] / row[mode]
        rows.append(row)
        del qd, out, flush, flush_rd
    dec.close()
    return rows


def cpu_baseline(w):
    import oracle
    cores = os.cpu_count() or 1
    q, stride = cpu_sample(w.queries)
    t0 = time.perf_counter()
    oracle.decode(w.assets, q, nthreads=cores)
    dt = time.perf_counter() - t0
    return {"value": len(q) / dt, "unit": UNIT, "cores": cores, "cpu_model": cpu_model(), "kind": "oracle",
            "sample": f"every {ordinal(stride)} query of the timed batch ({len(q):,} of {len(w.queries):,}), oracle on "
                      f"{cores} host threads, {dt:.1f} s"}


if __name__ == "__main__":
    main()
