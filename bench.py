#!/usr/bin/env python3
"""Benchmark of the packed LM-head forward (ARCHead, paper Section 3.2, Eq. 7)
on GB300 through the library's C ABI.

A step is one forward of the whole hot path -- rank-r pre-pass, INT4 residual
stream with group promotion, low-rank epilogue, logits store -- over one batch
of seeded synthetic hidden states already resident in device memory.  The
default workload is the Qwen3-8B-shaped head (V=151936, d=4096, r_c=128,
r_r=32, g=128) at M=1 token (decode); the same line also carries the decode
sweep M=2..16, the M=4096 prefill (logits and fused cross entropy), a dense
BF16 cuBLAS head on the same shapes, the batch sweep M=1..8192 through both
kernels, the same head in the paper's own packed format, the
Gemma-4-E4B-shaped head, the tiny head (a latency entry beside the oracle),
the offline construction of the Qwen head (Algorithm 1) and the headline
figures of those blocks again as flat top-level keys.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

With --impl reference the fp64 CPU oracle is timed on the host cores on a
bounded sample of the same workload (the baseline, not the target).
Multi-GPU runs (torchrun, one rank per GPU) are independent replicas: the
head does not shard in this build, so no collective is on the data path.
"""

from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

METRIC = "LM-head tokens/s and achieved HBM GB/s (M=1) / TFLOP/s (M=4096), % of roofline"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}

WORKLOADS = {
    "qwen3-8b-decode": ("qwen3-8b", 1, "logits"),
    "qwen3-8b-prefill": ("qwen3-8b", 4096, "logits"),
    "qwen3-8b-prefill-ce": ("qwen3-8b", 4096, "ce"),
    # the same head shape in the paper's own packed format (r_c = 10, r_r = 6, g = 64)
    "qwen3-8b-sc4-decode": ("qwen3-8b-sc4", 1, "logits"),
    "qwen3-8b-sc4-prefill": ("qwen3-8b-sc4", 4096, "logits"),
    "gemma-4-e4b-decode": ("gemma-4-e4b", 1, "logits"),
    "gemma-4-e4b-prefill": ("gemma-4-e4b", 2048, "logits"),
    "tiny": ("tiny", 4, "logits"),
}


KERNEL_SOURCES = {
    "decode": ("decode.cu", "decode_sc4.cu", "decode_kernel.cuh", "device.cuh", "internal.h"),
    "prefill": ("prefill.cu", "prefill_sc4.cu", "prefill_kernel.cuh", "device.cuh", "internal.h"),
}


def kernel_source_hash(kernel: str) -> str:
    """sha256 over the sources a kernel is compiled from (its traffic figure
    is only valid for the sources it was captured with)."""
    import hashlib

    h = hashlib.sha256()
    for f in KERNEL_SOURCES[kernel]:
        with open(os.path.join(ROOT, "paper_2608_02703_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


def captured_traffic(kernel: str, workload: str, M: int):
    """DRAM bytes (read + write) per launch of `kernel` from the committed ncu
    capture summary (profiles/traffic.json), or None if there is none for this
    workload or the kernel's sources changed since it was taken."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        table = json.load(f)
    e = table.get(f"{kernel}/{workload}/M={M}")
    if not e or e.get("sources_sha256") != kernel_source_hash(kernel):
        return None
    return e["dram_bytes_per_launch"]


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return {k: float(p[k]) for k in FALLBACK_PEAKS}, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


# ---------------------------------------------------------------------------
# Algorithmic work (what the method must move or compute per call).
# ---------------------------------------------------------------------------
def packed_vocab_bytes(shape) -> int:
    """Bytes of the V-indexed packed components the streaming kernel reads
    (in the paper's packed format: 4-bit group-scale codes, fp16 row scales
    and 5-bit core left codes in place of fp16 group scales and INT8 codes)."""
    V, d, rc, rr, g = shape.V, shape.d, shape.core_rank, shape.corr_rank, shape.group_size
    G = d // g
    if getattr(shape, "fmt", "int8") == "sc4":
        scales, core = V * ((G + 1) // 2) + V * 2, V * ((5 * rc + 7) // 8)
    else:
        scales, core = V * G * 2, V * rc
    return V * d // 2 + scales + core + V * rr + (V * 2 if rr else 0)


def packed_bytes(shape) -> int:
    """Eq. 10 over all stored components."""
    V, d, rc, rr, g = shape.V, shape.d, shape.core_rank, shape.corr_rank, shape.group_size
    G = d // g
    return packed_vocab_bytes(shape) + rc * 2 + d * rc + rc * 2 + d * rr + G * rr * 2


def call_bytes(shape, M, mode) -> int:
    out = 2 * M * shape.V if mode == "logits" else 4 * M
    return packed_bytes(shape) + 2 * M * shape.d + out


def kernel_bytes(shape, M, mode) -> int:
    """Algorithmic bytes of one launch of the streaming kernel."""
    out = 2 * M * shape.V if mode == "logits" else 4 * M
    return packed_vocab_bytes(shape) + 2 * M * shape.d + out


def call_flops(shape, M) -> int:
    r = shape.core_rank + shape.corr_rank
    return 2 * M * shape.V * shape.d + 2 * M * (shape.V + shape.d) * r


# ---------------------------------------------------------------------------
# Clock sampling during the timed region.
# ---------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.idx = device_index
        self.proc = None
        self.path = None

    def __enter__(self):
        import tempfile

        fd, self.path = tempfile.mkstemp(prefix="clocks", suffix=".csv")
        os.close(fd)
        try:
            self.out = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.idx}", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=self.out, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
        if hasattr(self, "out"):
            self.out.close()

    def summary(self):
        if self.proc is None or not self.path or not os.path.exists(self.path):
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 8:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}

        def num(v):
            try:
                return float(v)
            except ValueError:
                return None

        sm = [num(r[0]) for r in rows if num(r[0]) is not None]
        mx = [num(r[1]) for r in rows if num(r[1]) is not None]
        reasons = set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            for name, v in zip(names, r[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(name)
        loaded = sorted(sm)[len(sm) // 4:] if len(sm) >= 4 else sm
        return {"sm_mhz": statistics.median(loaded) if loaded else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(rows),
                "power_w_max": max((num(r[2]) or 0.0) for r in rows)}


# ---------------------------------------------------------------------------
# Distributed helpers (replicas; host-side logic covered by the gloo tests).
# ---------------------------------------------------------------------------
def dist_env():
    return int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")), int(
        os.environ.get("LOCAL_RANK", "0"))


def max_over_ranks(value: float, world: int, device=None) -> float:
    if world <= 1:
        return value
    import torch
    import torch.distributed as dist

    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(world: int):
    if world > 1:
        import torch.distributed as dist

        dist.barrier()


# ---------------------------------------------------------------------------
# Our arm.
# ---------------------------------------------------------------------------
class Workload:
    def __init__(self, shape_name: str, seed: int = 0):
        from synth import SHAPES, make_head

        self.shape = SHAPES[shape_name]
        self.head = make_head(self.shape, seed=seed)
        self.pack = None

    def open(self):
        from paper_2608_02703_gb300 import archead

        self.pack = archead.archead_pack_create(self.head, self.shape)
        return self.pack


def timed_loop(fn, steps: int, warmup: int, world: int):
    import torch

    for _ in range(warmup):
        fn()
    torch.cuda.synchronize()
    barrier(world)
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(steps):
        fn()
    e1.record(stream)
    torch.cuda.synchronize()
    barrier(world)
    return e0.elapsed_time(e1) / 1e3


def profiled_kernels(pack, fn, steps: int):
    """Per-kernel mean launch duration (ms) from the library's CUDA events."""
    import torch

    from paper_2608_02703_gb300 import archead

    archead.archead_profile_read(pack)  # drain
    base = {s["name"]: (s["launches"], s["total_ms"]) for s in archead.archead_profile_read(pack)}
    archead.archead_profile_enable(pack, True)
    for _ in range(steps):
        fn()
    torch.cuda.synchronize()
    archead.archead_profile_enable(pack, False)
    out = {}
    for s in archead.archead_profile_read(pack):
        l0, t0 = base.get(s["name"], (0, 0.0))
        n, t = s["launches"] - l0, s["total_ms"] - t0
        if n > 0:
            out[s["name"]] = {"launches_per_step": n / steps, "mean_ms": t / n}
    return out


def run_ours(args, rank, world, local_rank):
    import torch

    from paper_2608_02703_gb300 import archead
    from paper_2608_02703_gb300.build import build
    from synth import make_hidden, make_targets

    build()
    torch.cuda.set_device(local_rank)
    if world > 1:
        import torch.distributed as dist

        dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    peaks, peak_src = load_peaks()
    shape_name, M, mode = WORKLOADS[args.workload]
    if args.M:
        M = args.M
    wl = Workload(shape_name)
    shape = wl.shape
    pack = wl.open()
    x_np = make_hidden(shape.d, M, seed=1, n_outliers=shape.n_outliers)
    x = torch.from_numpy(x_np.view(np.int16)).cuda()
    t_np = make_targets(shape.V, M, seed=1)
    tgt = torch.from_numpy(t_np).cuda()
    y = torch.empty((M, shape.V), dtype=torch.bfloat16, device="cuda")
    ce = torch.empty(M, dtype=torch.float32, device="cuda")

    def step():
        if mode == "logits":
            archead.archead_forward(pack, x, M, y, archead.OUT_BF16)
        else:
            archead.archead_forward_ce(pack, x, M, tgt, ce)

    steps, warmup = args.steps, args.warmup
    if steps is None:
        steps = 20000 if M <= 16 else 20
    with ClockSampler(local_rank) as clk:
        secs = timed_loop(step, steps, warmup, world)
    st = archead.archead_sync_status(pack)
    if st != archead.OK:
        raise RuntimeError(f"device error after timed loop: {archead.archead_status_string(st)}")
    secs_max = max_over_ranks(secs, world, torch.device("cuda", local_rank))
    tokens_s = world * M * steps / secs_max

    prof = profiled_kernels(pack, step, max(3, min(steps, 2000)))
    main_kernel = "decode" if "decode" in prof else max(prof, key=lambda k: prof[k]["mean_ms"])
    launches_per_step = sum(v["launches_per_step"] for v in prof.values())
    kb = kernel_bytes(shape, M, mode)
    kms = prof[main_kernel]["mean_ms"]
    if M <= 64:
        achieved = kb / (kms / 1e3) / 1e9
        roof = {"kernel": main_kernel, "bound": "hbm", "achieved": round(achieved, 1), "peak": peaks["hbm_gbs"],
                "unit": "GB/s", "frac": round(achieved / peaks["hbm_gbs"], 4),
                "traffic": captured_traffic(main_kernel, args.workload, M),
                "peak_source": peak_src, "algorithmic_bytes_per_launch": kb, "mean_launch_ms": kms}
    else:
        fl = call_flops(shape, M) / prof[main_kernel]["launches_per_step"]
        achieved = fl / (kms / 1e3) / 1e12
        peak = peaks["bf16_tflops"]
        roof = {"kernel": main_kernel, "bound": "tensor", "achieved": round(achieved, 1), "peak": peak,
                "unit": "TFLOP/s", "frac": round(achieved / peak, 4),
                "traffic": captured_traffic(main_kernel, args.workload, M), "peak_source": peak_src,
                "algorithmic_flops_per_launch": fl, "mean_launch_ms": kms}

    # End to end through the public host-buffer entry point.
    e2e = None
    if mode == "logits":
        xh = torch.from_numpy(x_np.view(np.int16).copy()).pin_memory()
        yh = torch.empty((M, shape.V), dtype=torch.bfloat16).pin_memory()
        k2 = max(3, min(steps, 2000 if M <= 16 else 5))
        for _ in range(3):
            archead.archead_forward_host(pack, xh, M, yh, archead.OUT_BF16)
        barrier(world)
        t0 = time.perf_counter()
        for _ in range(k2):
            archead.archead_forward_host(pack, xh, M, yh, archead.OUT_BF16)
        t_e2e = max_over_ranks(time.perf_counter() - t0, world, torch.device("cuda", local_rank))
        e2e = {"value": round(world * M * k2 / t_e2e, 2), "unit": "tokens/s", "h2d_bytes_per_step": M * shape.d * 2,
               "d2h_bytes_per_step": M * shape.V * 2, "steps": k2}

    result = {
        "metric": METRIC, "value": round(tokens_s, 2), "unit": "tokens/s", "n_gpus": world, "steps": steps,
        "warmup": warmup, "ms_per_step": round(secs_max / steps * 1e3, 5), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": f"{shape_name} head, {'decode' if M <= 16 else 'prefill'} M={M}, "
                               f"{'logits bf16' if mode == 'logits' else 'fused CE'}",
                   "V": shape.V, "d": shape.d, "core_rank": shape.core_rank, "corr_rank": shape.corr_rank,
                   "group_size": shape.group_size, "format": shape.fmt, "M": M,
                   "parallelism": f"replicas x{world}",
                   "l2": "inputs larger than L2: the packed head (%.1f MB) exceeds the 129 MB L2, so every "
                         "forward streams it from HBM" % (packed_bytes(shape) / 1e6)},
        "roofline": roof,
        "gpu_launches": int(round(launches_per_step * steps)),
        "kernels": {k: {"launches_per_step": v["launches_per_step"], "mean_us": round(v["mean_ms"] * 1e3, 3)}
                    for k, v in prof.items()},
        "e2e": e2e,
        "clocks": clk.summary(),
        "algorithmic": {"bytes_per_call": call_bytes(shape, M, mode), "flops_per_call": call_flops(shape, M),
                        "gbs_per_call": round(call_bytes(shape, M, mode) / (secs_max / steps) / 1e9, 1)},
    }

    if not args.no_extras and args.workload == "qwen3-8b-decode":
        result["decode_sweep"] = decode_sweep(pack, shape, peaks, world, local_rank)
        result["prefill"] = prefill_block(pack, shape, peaks, world, local_rank)
        result["dense_bf16_cublas"] = dense_comparator(shape, world, local_rank)
        result["crossover"] = crossover_sweep(pack, shape, world, local_rank)
    pack.close()
    if not args.no_extras and args.workload == "qwen3-8b-decode":
        result["sc4"] = sc4_block(peaks, world, local_rank)
        result["gemma"] = gemma_block(peaks, world, local_rank)
        result["tiny"] = tiny_block(world, local_rank, with_oracle=rank == 0 and world == 1)
        result["construct"] = construct_block()
        result.update(flat_keys(result))
    if rank == 0 and not args.no_cpu_baseline and world == 1:
        result["cpu_baseline"] = cpu_baseline(wl, x_np, M, budget_s=args.cpu_budget)
    return result


def tiny_block(world, local_rank, with_oracle=True):
    """The tiny head (V=4096, d=512, r_c=64, r_r=16, g=64) at M=4: a latency
    entry next to the oracle on the same workload.  Its 1.5 MB pack stays in
    the 129 MB L2, so no roofline fraction is claimed for it."""
    import torch

    from paper_2608_02703_gb300 import archead
    from synth import make_hidden

    wl = Workload("tiny")
    pack = wl.open()
    M = 4
    x_np = make_hidden(wl.shape.d, M, seed=1, n_outliers=wl.shape.n_outliers)
    x = torch.from_numpy(x_np.view(np.int16)).cuda()
    y = torch.empty((M, wl.shape.V), dtype=torch.bfloat16, device="cuda")
    fn = lambda: archead.archead_forward(pack, x, M, y, archead.OUT_BF16)  # noqa: E731
    k = 2000
    secs = max_over_ranks(timed_loop(fn, k, 20, world), world, torch.device("cuda", local_rank))
    res = {"workload": "tiny head (V=4096, d=512, r_c=64, r_r=16, g=64), decode M=4, logits bf16",
           "M": M, "us_per_call": round(secs / k * 1e6, 2), "tokens_s": round(world * M * k / secs, 1),
           "packed_bytes": packed_bytes(wl.shape),
           "note": "L2-resident (packed head 1.5 MB < 129 MB L2): a latency figure, no roofline claim"}
    st = archead.archead_sync_status(pack)
    res["status"] = archead.archead_status_string(st)
    pack.close()
    if with_oracle:
        import oracle

        t = min(oracle_rows_time(wl.head, wl.shape, x_np, wl.shape.V) for _ in range(3))
        res["oracle"] = {"us_per_call": round(t * 1e6, 1), "cores": oracle.threads(),
                         "sample": "the whole forward (all 4096 rows, M=4), best of 3"}
    return res


def construct_block(N: int = 4096):
    """Offline construction (Algorithm 1) of the Qwen3-8B-shaped head in the
    paper's format (r_c=10, r_r=6, g=64, p=0.75, ridge 1e-3) from a seeded
    dense head and N calibration states, fp32 linear algebra: wall time on the
    device, and the error left in the activation metric by the realized core
    and by core plus the unquantised correction, relative to ||W T_p||^2."""
    import torch

    from paper_2608_02703_gb300 import construct as gc
    from synth import SHAPES, make_dense_head_device, make_hidden, make_test_matrix

    sh = SHAPES["qwen3-8b-sc4"]
    W = make_dense_head_device(sh.V, sh.d, seed=0)
    H = torch.from_numpy(make_hidden(sh.d, N, seed=7).view(np.int16)).cuda().view(torch.bfloat16).float()
    om_c = torch.from_numpy(make_test_matrix(sh.d, sh.core_rank + 10, seed=1)).cuda().float()
    om_r = torch.from_numpy(make_test_matrix(sh.d, sh.corr_rank + 10, seed=2)).cuda().float()
    args = dict(fmt="sc4", omega_core=om_c, omega_corr=om_r, dtype=torch.float32)
    gc.construct(W[:4096], H, sh.core_rank, sh.corr_rank, sh.group_size, **args)  # warm-up (library load, cuSOLVER)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    head = gc.construct(W, H, sh.core_rank, sh.corr_rank, sh.group_size, keep_intermediates=True, **args)
    torch.cuda.synchronize()
    secs = time.perf_counter() - t0
    T = head["_T"]
    ref = float(((W @ T) ** 2).sum())
    e_core = float((head["_E"] @ T).pow(2).sum()) / ref
    e_corr = float(((head["_E"] - head["_A_w"] @ head["_B_w"]) @ T).pow(2).sum()) / ref
    res = {"workload": f"qwen3-8b-shaped dense head (V={sh.V}, D={sh.d}), N={N} calibration states, paper's format "
                       "(r_c=10, r_r=6, g=64), p=0.75, ridge 1e-3, fp32 linear algebra",
           "seconds": round(secs, 3), "rel_metric_error_core": round(e_core, 6),
           "rel_metric_error_core_plus_correction": round(e_corr, 6)}
    del head, W, H
    torch.cuda.empty_cache()
    return res


def flat_keys(result):
    """The headline numbers of the nested blocks as top-level scalars."""
    out = {}
    pf = result.get("prefill") or {}
    for mode in ("logits", "ce"):
        if mode in pf:
            out[f"qwen_prefill_m{pf['M']}_{mode}_ms"] = pf[mode]["ms_per_call"]
            out[f"qwen_prefill_m{pf['M']}_{mode}_frac_bf16_peak"] = pf[mode]["frac_bf16_peak"]
    for row in result.get("decode_sweep") or []:
        out[f"qwen_decode_m{row['M']}_us"] = row["us_per_call"]
        out[f"qwen_decode_m{row['M']}_kernel_frac_hbm"] = row["frac_hbm"]
    for blk, name in (("sc4", "qwen_sc4"), ("gemma", "gemma")):
        b = result.get(blk) or {}
        for row in b.get("decode_sweep") or []:
            out[f"{name}_decode_m{row['M']}_us"] = row["us_per_call"]
            out[f"{name}_decode_m{row['M']}_kernel_frac_hbm"] = row["frac_hbm"]
        bp = b.get("prefill") or {}
        for mode in ("logits", "ce"):
            if mode in bp:
                out[f"{name}_prefill_m{bp['M']}_{mode}_ms"] = bp[mode]["ms_per_call"]
                out[f"{name}_prefill_m{bp['M']}_{mode}_frac_bf16_peak"] = bp[mode]["frac_bf16_peak"]
    for row in (result.get("crossover") or {}).get("rows") or []:
        if row["M"] in (32, 64, 256, 4096):
            out[f"qwen_crossover_m{row['M']}_auto_us"] = row["auto_us"]
            out[f"qwen_crossover_m{row['M']}_dense_bf16_us"] = row["dense_bf16_us"]
    c = result.get("construct") or {}
    if "seconds" in c:
        out["construct_qwen_sc4_seconds"] = c["seconds"]
    t = result.get("tiny") or {}
    if "us_per_call" in t:
        out["tiny_m4_us"] = t["us_per_call"]
        if "oracle" in t:
            out["tiny_m4_oracle_us"] = t["oracle"]["us_per_call"]
    return out


def gemma_block(peaks, world, local_rank):
    """The Gemma-4-E4B-shaped head (V=262144, d=2560, r_c=128, r_r=32, g=128):
    decode M=1 and 8, prefill M=2048 (logits and fused CE)."""
    wl = Workload("gemma-4-e4b")
    pack = wl.open()
    res = {"workload": "gemma-4-e4b head (V=262144, d=2560, r_c=128, r_r=32, g=128)",
           "packed_bytes": packed_bytes(wl.shape),
           "decode_sweep": decode_sweep(pack, wl.shape, peaks, world, local_rank, Ms=(1, 8)),
           "prefill": prefill_block(pack, wl.shape, peaks, world, local_rank, M=2048)}
    pack.close()
    return res


def sc4_block(peaks, world, local_rank):
    """The Qwen3-8B head in the paper's own packed format (5-bit core left
    codes, 4-bit group-scale codes, r_c = 10, r_r = 6, g = 64): decode and
    prefill on the same footing as the lines above."""
    wl = Workload("qwen3-8b-sc4")
    pack = wl.open()
    res = {"workload": "qwen3-8b-sc4 head (V=151936, d=4096, r_c=10, r_r=6, g=64, paper's packed format)",
           "packed_bytes": packed_bytes(wl.shape),
           "decode_sweep": decode_sweep(pack, wl.shape, peaks, world, local_rank, Ms=(1, 4, 8, 16)),
           "prefill": prefill_block(pack, wl.shape, peaks, world, local_rank)}
    pack.close()
    return res


def decode_sweep(pack, shape, peaks, world, local_rank, Ms=(1, 2, 4, 8, 16)):
    import torch

    from paper_2608_02703_gb300 import archead
    from synth import make_hidden

    out = []
    for M in Ms:
        x = torch.from_numpy(make_hidden(shape.d, M, seed=2, n_outliers=shape.n_outliers).view(np.int16)).cuda()
        y = torch.empty((M, shape.V), dtype=torch.bfloat16, device="cuda")
        fn = lambda: archead.archead_forward(pack, x, M, y, archead.OUT_BF16)  # noqa: E731
        k = 2000
        secs = max_over_ranks(timed_loop(fn, k, 20, world), world, torch.device("cuda", local_rank))
        prof = profiled_kernels(pack, fn, 500)
        kms = prof["decode"]["mean_ms"]
        gbs = kernel_bytes(shape, M, "logits") / (kms / 1e3) / 1e9
        out.append({"M": M, "tokens_s": round(world * M * k / secs, 1), "us_per_call": round(secs / k * 1e6, 2),
                    "decode_kernel_us": round(kms * 1e3, 2), "decode_gbs": round(gbs, 1),
                    "frac_hbm": round(gbs / peaks["hbm_gbs"], 4)})
    return out


def prefill_block(pack, shape, peaks, world, local_rank, M=4096):
    import torch

    from paper_2608_02703_gb300 import archead
    from synth import make_hidden, make_targets

    x = torch.from_numpy(make_hidden(shape.d, M, seed=3, n_outliers=shape.n_outliers).view(np.int16)).cuda()
    y = torch.empty((M, shape.V), dtype=torch.bfloat16, device="cuda")
    tgt = torch.from_numpy(make_targets(shape.V, M, seed=3)).cuda()
    ce = torch.empty(M, dtype=torch.float32, device="cuda")
    res = {"M": M}
    for mode, fn in (("logits", lambda: archead.archead_forward(pack, x, M, y, archead.OUT_BF16)),
                     ("ce", lambda: archead.archead_forward_ce(pack, x, M, tgt, ce))):
        k = 5
        secs = max_over_ranks(timed_loop(fn, k, 3, world), world, torch.device("cuda", local_rank))
        tf = call_flops(shape, M) / (secs / k) / 1e12
        res[mode] = {"tokens_s": round(world * M * k / secs, 1), "ms_per_call": round(secs / k * 1e3, 3),
                     "tflops": round(tf, 1), "frac_bf16_peak": round(tf / peaks["bf16_tflops"], 4)}
    st = archead.archead_sync_status(pack)
    res["status"] = archead.archead_status_string(st)
    return res


def crossover_sweep(pack, shape, world, local_rank):
    """Batch sweep on one head: per M the decode kernel (one launch per 16,
    32 or 64 tokens), the prefill kernel, the automatic choice and a dense
    BF16 cuBLAS GEMM of the same shape, each as microseconds per call (bf16
    logits out)."""
    import torch

    from paper_2608_02703_gb300 import archead
    from synth import make_hidden

    g = torch.Generator(device="cuda")
    g.manual_seed(0)
    W = (torch.randn((shape.V, shape.d), generator=g, device="cuda", dtype=torch.float32) * 0.01).to(torch.bfloat16)
    dev = torch.device("cuda", local_rank)
    rows = []
    for M in (1, 4, 16, 32, 64, 128, 256, 1024, 4096, 8192):
        x = torch.from_numpy(make_hidden(shape.d, M, seed=5, n_outliers=shape.n_outliers).view(np.int16)).cuda()
        y = torch.empty((M, shape.V), dtype=torch.bfloat16, device="cuda")
        k = 200 if M <= 16 else (20 if M <= 1024 else 4)
        row = {"M": M}
        for name, path in (("decode_us", archead.PATH_DECODE), ("prefill_us", archead.PATH_PREFILL),
                           ("auto_us", archead.PATH_AUTO)):
            fn = lambda: archead.archead_forward_path(pack, x, M, y, archead.OUT_BF16, path)  # noqa: E731
            kk = max(2, k // 8) if (path == archead.PATH_DECODE and M >= 1024) else k
            secs = max_over_ranks(timed_loop(fn, kk, 3, world), world, dev)
            row[name] = round(secs / kk * 1e6, 2)
        xb = x.view(torch.bfloat16)
        fn = lambda: torch.matmul(xb, W.t())  # noqa: E731
        secs = max_over_ranks(timed_loop(fn, k, 3, world), world, dev)
        row["dense_bf16_us"] = round(secs / k * 1e6, 2)
        row["auto_tokens_s"] = round(world * M / (row["auto_us"] / 1e6), 1)
        rows.append(row)
        del y
    st = archead.archead_sync_status(pack)
    del W
    torch.cuda.empty_cache()
    return {"rows": rows, "status": archead.archead_status_string(st)}


def dense_comparator(shape, world, local_rank):
    """Dense BF16 V x d head through cuBLAS (torch.matmul) on the same shapes."""
    import torch

    g = torch.Generator(device="cuda")
    g.manual_seed(0)
    W = (torch.randn((shape.V, shape.d), generator=g, device="cuda", dtype=torch.float32) * 0.01).to(torch.bfloat16)
    res = {}
    for M in (1, 16, 4096):
        x = torch.randn((M, shape.d), generator=g, device="cuda", dtype=torch.float32).to(torch.bfloat16)
        fn = lambda: torch.matmul(x, W.t())  # noqa: E731
        k = 200 if M <= 16 else 10
        secs = max_over_ranks(timed_loop(fn, k, 5, world), world, torch.device("cuda", local_rank))
        res[f"M={M}"] = {"tokens_s": round(world * M * k / secs, 1), "us_per_call": round(secs / k * 1e6, 2),
                         "tflops": round(2 * M * shape.V * shape.d / (secs / k) / 1e12, 2)}
    del W
    torch.cuda.empty_cache()
    return res


# ---------------------------------------------------------------------------
# CPU oracle (baseline leg and reference arm).
# ---------------------------------------------------------------------------
def oracle_rows_time(head, shape, x_np, rows: int) -> float:
    import oracle

    t0 = time.perf_counter()
    oracle.logits(head, shape, x_np, row0=0, nrows=rows)
    return time.perf_counter() - t0


def cpu_baseline(wl, x_np, M, budget_s: float = 15.0):
    """Time the oracle as it stands on a bounded sample of vocabulary rows."""
    import oracle

    shape = wl.shape
    rows = min(shape.V, 1024)
    t = oracle_rows_time(wl.head, shape, x_np, rows)
    while t < budget_s / 4 and rows < shape.V:
        rows = min(shape.V, int(rows * max(2.0, budget_s / 2 / max(t, 1e-3))))
        t = oracle_rows_time(wl.head, shape, x_np, rows)
    full = t * shape.V / rows
    return {"value": round(M / full, 4), "unit": "tokens/s", "cores": oracle.threads(), "kind": "oracle",
            "sample": f"fp64 oracle logits of the first {rows} of {shape.V} vocabulary rows for M={M} token(s), "
                      f"{t:.2f} s; scaled by V/rows to a full forward"}


def run_reference(args, rank, world):
    import oracle
    from synth import make_hidden

    if rank != 0:
        return None
    oracle.build()
    shape_name, M, mode = WORKLOADS[args.workload]
    if args.M:
        M = args.M
    wl = Workload(shape_name)
    shape = wl.shape
    x_np = make_hidden(shape.d, M, seed=1, n_outliers=shape.n_outliers)
    steps = args.steps if args.steps is not None else 20
    warmup = args.warmup
    # Size one step so that the whole run takes about two minutes.
    t1 = oracle_rows_time(wl.head, shape, x_np, 256)
    per_row = max(t1 / 256, 1e-7)
    rows = int(max(16, min(shape.V, (args.ref_budget / max(steps + warmup, 1)) / per_row)))
    for _ in range(warmup):
        oracle_rows_time(wl.head, shape, x_np, rows)
    t0 = time.perf_counter()
    for _ in range(steps):
        oracle_rows_time(wl.head, shape, x_np, rows)
    secs = time.perf_counter() - t0
    tokens_s = M * steps * rows / shape.V / secs
    sample = (f"each step: fp64 oracle logits of {rows} of {shape.V} vocabulary rows for M={M} token(s) "
              f"(a {rows / shape.V:.4f} fraction of one forward)")
    return {
        "metric": METRIC, "value": round(tokens_s, 4), "unit": "tokens/s", "n_gpus": world, "steps": steps,
        "warmup": warmup, "ms_per_step": round(secs / steps * 1e3, 3), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic", "impl": "reference",
        "config": {"workload": f"{shape_name} head, {'decode' if M <= 16 else 'prefill'} M={M}, "
                               f"{'logits' if mode == 'logits' else 'CE'}", "V": shape.V, "d": shape.d, "M": M},
        "cpu_baseline": {"value": round(tokens_s, 4), "unit": "tokens/s", "cores": oracle.threads(),
                         "kind": "oracle", "sample": sample},
        "e2e": {"value": round(tokens_s, 4), "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", choices=sorted(WORKLOADS), default="qwen3-8b-decode")
    ap.add_argument("--M", type=int, default=None)
    ap.add_argument("--no-extras", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-budget", type=float, default=15.0)
    ap.add_argument("--ref-budget", type=float, default=90.0)
    args = ap.parse_args(argv)
    if args.warmup < 3:
        ap.error("--warmup must be at least 3")
    rank, world, local_rank = dist_env()
    if args.impl == "reference":
        res = run_reference(args, rank, world)
    else:
        res = run_ours(args, rank, world, local_rank)
    if rank == 0 and res is not None:
        print(json.dumps(res), flush=True)
    if world > 1 and args.impl == "ours":
        import torch.distributed as dist

        dist.destroy_process_group()


if __name__ == "__main__":
    main()
