#!/usr/bin/env python3
"""Benchmark of the sparse spiral-conv hot path on one GB300 (or N replicas).

One step = one pass of the hot path over one batch of the 10475-vertex
workload (B = 32 frames, spiral length L = 12, 64 -> 128 channels, bf16,
clustered contact masks at ~5% density):
    hc_mask_compact_rulebook     mask -> coords, row_of, offsets, count (Eq. 2) and
                                 the tap -> input-row mapping (Eq. 4): a count pass,
                                 then one fused pass per (frame, 1024 vertices)
    hc_sparse_conv_rulebook_fwd  gather + tcgen05 contraction + bias + ELU (Eq. 5),
                                 writing the compact rows and, fused into the same
                                 epilogue, their scatter into the dense [B, V, 128]
Inputs are resident in HBM; every step reads its own input set (mask and
features) from a rotation whose total size is more than twice the L2, so
consecutive steps do not hit in L2. The timed steps are replayed from CUDA
graphs captured on the bench stream.

Printed (one JSON line, rank 0): active rows/s over all ranks, the roofline
of the dominant kernel (the tensor-core conv, timed alone with CUDA events),
the CPU oracle as a reported baseline, an end-to-end number through the
C-ABI with host buffers, the dense operator and the speed-up over it, the
density sweep, and the SM clocks sampled around the timed region.

--impl reference times the CPU oracle (test infrastructure, plain C, fp64)
on bounded samples of the same workload; it is the only other place this
script runs the oracle.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

METRIC = "active vertex-rows/s & % roofline, sparse spiral-conv layer; speed-up vs dense"
WORKLOAD = "layer10475_bf16"


E2E_IN_FLIGHT = 8  # default requests in flight of the end-to-end loop


def parse_args():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=400)
    p.add_argument("--warmup", type=int, default=10)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--no-extras", action="store_true",
                   help="skip the side measurements (density sweep, group norm, mask score, "
                        "backward)")
    p.add_argument("--extra", choices=["all", "sweep", "group_norm", "mask_score", "backward",
                                       "kappa", "configs", "stages"],
                   default="all", help="run only this side measurement")
    p.add_argument("--clocks-csv", default=None, help="also write the raw clock samples here")
    p.add_argument("--e2e-steps", type=int, default=200)
    p.add_argument("--e2e-in-flight", type=int, default=E2E_IN_FLIGHT,
                   help="requests in flight in the end-to-end loop (buffer sets and streams)")
    p.add_argument("--no-e2e", action="store_true",
                   help="skip the end-to-end measurement (for targeted profiler captures)")
    p.add_argument("--case", default=None,
                   help="profiler target instead of the bench: run one layer call of the "
                        "density sweep's workload --steps times and print its CUDA-event "
                        "times; 'sweep:D' the sparse conv at mask density D (compaction and "
                        "mapping done before), 'sweep-dense' the dense layer, 'mask-score' "
                        "the mask-score update on the encoder outputs (K = 10, 41,920 x 64)")
    return p.parse_args()


# ----------------------------------------------------------------- helpers

def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        d = json.load(open(path))
        return {"hbm_gbs": d["hbm_gbs"], "bf16_tflops": d["bf16_tflops"],
                "bf16_tflops_sustained": d.get("bf16_tflops_sustained"), "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
            "source": "fallback"}


def kernel_source_hash():
    h = hashlib.sha256()
    for f in ("conv_tc.cu", "hc_internal.cuh"):
        h.update(open(os.path.join(ROOT, "paper_2608_09388_gb300", "csrc", f), "rb").read())
    return h.hexdigest()[:16]


def ncu_traffic():
    """DRAM bytes per launch of the conv kernel from the committed ncu summary,
    or None if the summary is missing or the kernel source changed since."""
    path = os.path.join(ROOT, "profiles", "conv_tc_layer10475_bf16.json")
    if not os.path.exists(path):
        return None, None
    d = json.load(open(path))
    if d.get("kernel_source_hash") != kernel_source_hash():
        return None, d.get("kernel_source_hash")
    return d.get("dram_bytes_per_launch"), d.get("kernel_source_hash")


class ClockSampler:
    """nvidia-smi samples (every 200 ms) while the load runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index, csv_path=None):
        self.proc = None
        self.out = None
        self.csv_path = csv_path
        sel = []
        try:
            import torch
            u = str(torch.cuda.get_device_properties(device_index).uuid)
            sel = ["-i", u if u.startswith("GPU-") else "GPU-" + u]
        except Exception:
            vis = os.environ.get("CUDA_VISIBLE_DEVICES")
            if vis:
                sel = ["-i", vis.split(",")[device_index]]
        self.cmd = ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                    "-lms", "200", *sel]

    def start(self):
        import tempfile
        self.out = tempfile.TemporaryFile(mode="w+")
        try:
            self.proc = subprocess.Popen(self.cmd, stdout=self.out, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.out.seek(0)
        text = self.out.read()
        if self.csv_path:
            with open(self.csv_path, "w") as f:
                f.write(self.FIELDS + "\n" + text)
        sm, mx, power, reasons = [], [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in text.strip().splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
                power.append(float(parts[3]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "samples": len(sm),
                "power_w_max": max(power) if power else None, "reasons": sorted(reasons)}


# ----------------------------------------------------------------- ranks

def reduce_over_ranks(rows, ms, world, device):
    """Whole-job figures of one timed region: the rows every rank processed,
    summed, and the slowest rank's time (replicas run independent batches;
    this is the only cross-rank exchange, two scalars, off the data path)."""
    if world <= 1:
        return rows, ms
    import torch
    t = torch.tensor([rows, ms], dtype=torch.float64, device=device)
    r_sum = t.clone()
    torch.distributed.all_reduce(r_sum, op=torch.distributed.ReduceOp.SUM)
    r_max = t.clone()
    torch.distributed.all_reduce(r_max, op=torch.distributed.ReduceOp.MAX)
    return float(r_sum[0].item()), float(r_max[1].item())


def any_rank(flag, world, device):
    """True if the flag is set on any rank (all ranks get the same answer)."""
    if world <= 1:
        return bool(flag)
    import torch
    t = torch.tensor([1 if flag else 0], dtype=torch.int32, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return bool(int(t.item()))


# ----------------------------------------------------------------- our arm

class LayerSet:
    """One rotation entry: a batch's mask and features plus its outputs."""


def build_sets(torch, w, R, seed_base, dev):
    """Input set 0 is the seeded workload itself; sets 1..R-1 use the same
    recipe with their own seeds (masks from numpy, features drawn on the
    device from a seeded torch generator)."""
    from paper_2608_09388_gb300 import inputs
    ly = w.layers[0]
    B, V = w.B, w.V
    sets = []
    for i in range(R):
        s = LayerSet()
        if i == 0:
            mask = w.masks[0]
            x = torch.from_numpy(w.x.view(np.int16)).view(torch.bfloat16).to(dev)
        else:
            rng = np.random.default_rng(seed_base + 7919 * i)
            mask = inputs.clustered_mask(rng, w.points, B, 8, 0.05)
            g = torch.Generator(device=dev)
            g.manual_seed(seed_base + 104729 * i)
            x = torch.randn((B, V, ly.C_in), generator=g, device=dev,
                            dtype=torch.float32).to(torch.bfloat16)
        s.mask_np = mask
        s.rows = int(np.count_nonzero(mask))
        s.mask = torch.from_numpy(mask).to(dev)
        s.x = x
        s.coords = torch.empty((B * V, 2), dtype=torch.int32, device=dev)
        s.row_of = torch.empty((B, V), dtype=torch.int32, device=dev)
        s.offs = torch.empty((B + 1,), dtype=torch.int32, device=dev)
        s.count = torch.empty((1,), dtype=torch.int32, device=dev)
        s.rb = torch.empty((w.L, B * V), dtype=torch.int32, device=dev)
        s.y = torch.empty((B * V, ly.C_out), dtype=torch.bfloat16, device=dev)
        s.out = torch.zeros((B, V, ly.C_out), dtype=torch.bfloat16, device=dev)
        sets.append(s)
    return sets


def run_ours(args, rank, world, local_rank):
    import torch

    from paper_2608_09388_gb300 import build as hc_build
    from paper_2608_09388_gb300 import hc, inputs

    if rank == 0 or not os.path.exists(os.path.join(ROOT, "paper_2608_09388_gb300", "_build",
                                                    "libhc.so")):
        hc_build.build()
    if world > 1:
        torch.distributed.barrier()
    hc.load_library()
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    props = torch.cuda.get_device_properties(dev)
    l2 = int(getattr(props, "L2_cache_size", 0) or 0) or 126 * 2 ** 20

    w = inputs.make_workload(WORKLOAD)
    ly = w.layers[0]
    B, V, L = w.B, w.V, w.L
    set_bytes = B * V * (1 + 2 * ly.C_in)  # mask + features read by a step
    R = max(4, math.ceil(2.5 * l2 / set_bytes))
    sets = build_sets(torch, w, R, inputs.SEEDS[WORKLOAD] + 1000 * rank, dev)
    spiral = torch.from_numpy(w.spiral).to(dev)
    Wt = torch.from_numpy(ly.W.view(np.int16)).view(torch.bfloat16).to(dev)
    bias = torch.from_numpy(ly.b).to(dev)
    stream = torch.cuda.Stream(device=dev)

    def step(s):
        hc.hc_mask_compact_rulebook(s.mask, spiral, hc.HC_LAYOUT_DENSE, s.coords, s.row_of,
                                    s.offs, s.count, s.rb, stream)
        hc.hc_sparse_conv_rulebook_fwd(s.x, s.rb, s.count, Wt, bias, ly.act, s.y,
                                       coords=s.coords, out=s.out, stream=stream)

    def conv_only(s):
        hc.hc_sparse_conv_rulebook_fwd(s.x, s.rb, s.count, Wt, bias, ly.act, s.y,
                                       coords=s.coords, out=s.out, stream=stream)

    def dense_only(s):
        hc.hc_spiral_conv_fwd(s.x, spiral, Wt, bias, ly.act, s.dense, stream)

    # count pass (+ the tile pre-scan past 1024 tiles), the fused compaction +
    # mapping pass (or the write and mapping kernels past its limits), conv
    fused = V <= 65535
    kernels_per_step = 1 + (1 if (B * V + 4095) // 4096 > 1024 else 0) + (1 if fused else 2) + 1

    # W warm-up steps, then one priming pass over every input set (both
    # eager, untimed; they also set up the library's per-stream workspace).
    with torch.cuda.stream(stream):
        for i in range(args.warmup):
            step(sets[i % R])
        for s in sets:
            step(s)
    torch.cuda.synchronize(dev)
    st = hc.hc_get_device_status(stream)
    if st != hc.HC_OK:
        raise RuntimeError(f"device status {hc.STATUS_NAMES.get(st)} after warm-up")
    for s in sets:
        assert int(s.count.item()) == s.rows, "active-row count differs from the mask"

    def capture(fn, idx):
        # one eager call first: whatever workspace or per-stream state the
        # call needs is allocated before the capture (no allocation inside)
        with torch.cuda.stream(stream):
            fn(sets[idx[0]])
        torch.cuda.synchronize(dev)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for i in idx:
                fn(sets[i])
        return g

    K = args.steps
    g_full = capture(step, range(R))
    g_rem = capture(step, range(K % R)) if K % R else None

    rows_per_round = sum(s.rows for s in sets)
    rows_timed = (K // R) * rows_per_round + sum(sets[i].rows for i in range(K % R))

    def timed_region():
        """Exactly K steps, bracketed by a barrier and a synchronize."""
        if world > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize(dev)
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            e0.record(stream)
            for _ in range(K // R):
                g_full.replay()
            if g_rem is not None:
                g_rem.replay()
            e1.record(stream)
        torch.cuda.synchronize(dev)
        if world > 1:
            torch.distributed.barrier()
        return e0.elapsed_time(e1)

    # The timed region is repeated (at least 3 times, and until a second has
    # passed) while nvidia-smi samples the clocks; ms is the median repeat.
    sampler = ClockSampler(local_rank, args.clocks_csv if rank == 0 else None)
    sampler.start()
    reps_ms = []
    t_start = time.perf_counter()
    while len(reps_ms) < 3 or time.perf_counter() - t_start < 1.0:
        reps_ms.append(timed_region())
        if world > 1 and len(reps_ms) >= 3 and not any_rank(
                time.perf_counter() - t_start < 1.0, world, dev):
            break  # every rank agrees on the number of repeats
    clocks = sampler.stop()
    ms = statistics.median(reps_ms)

    # Dominant kernel alone: the tensor-core conv over the same rotation.
    g_conv = capture(conv_only, range(R))
    reps = max(1, 200 // R)
    with torch.cuda.stream(stream):
        g_conv.replay()
        c0 = torch.cuda.Event(enable_timing=True)
        c1 = torch.cuda.Event(enable_timing=True)
        c0.record(stream)
        for _ in range(reps):
            g_conv.replay()
        c1.record(stream)
    torch.cuda.synchronize(dev)
    conv_ms = c0.elapsed_time(c1) / (reps * R)
    mean_rows = rows_per_round / R
    flops_per_launch = 2.0 * L * ly.C_in * ly.C_out * mean_rows
    pk = peaks()
    achieved = flops_per_launch / (conv_ms * 1e-3) / 1e12
    traffic, khash = ncu_traffic()

    # Dense operator (the speed-up denominator): our dense kernel and torch's
    # gather + matmul, the faster of the two.
    for s in sets:
        s.dense = torch.empty((B, V, ly.C_out), dtype=torch.bfloat16, device=dev)
    g_dense = capture(dense_only, range(R))
    with torch.cuda.stream(stream):
        g_dense.replay()
        d0 = torch.cuda.Event(enable_timing=True)
        d1 = torch.cuda.Event(enable_timing=True)
        d0.record(stream)
        for _ in range(3):
            g_dense.replay()
        d1.record(stream)
    torch.cuda.synchronize(dev)
    dense_ms = d0.elapsed_time(d1) / (3 * R)
    torch_dense_ms = time_torch_dense(torch, sets, w, Wt, bias, stream, dev)
    best_dense = min(dense_ms, torch_dense_ms)
    for s in sets:
        del s.dense
    torch.cuda.empty_cache()

    e2e = None
    if not args.no_e2e:
        e2e = measure_e2e(torch, hc, sets, w, spiral, Wt, bias, stream, dev, args.e2e_steps,
                          args.e2e_in_flight)
        # whole-job end-to-end figure: rows of all ranks over the slowest rank's time
        e2e_rows, e2e_ms = reduce_over_ranks(float(e2e.pop("rows")), e2e.pop("seconds") * 1e3,
                                             world, dev)
        e2e["value"] = e2e_rows / (e2e_ms * 1e-3)
        e2e["ms_per_step"] = e2e_ms / e2e["steps"]
        e2e["ranks"] = world

    # Compaction alone (count pass + fused compaction and Eq. 4 mapping, and
    # the plain compaction without the mapping) over the same rotation; the
    # step is compaction + conv.
    def compact_map(s):
        hc.hc_mask_compact_rulebook(s.mask, spiral, hc.HC_LAYOUT_DENSE, s.coords, s.row_of,
                                    s.offs, s.count, s.rb, stream)

    def compact_only(s):
        hc.hc_mask_compact(s.mask, s.coords, s.row_of, s.offs, s.count, stream)

    comp_us = {}
    for tag, fn in (("compact_map_us", compact_map), ("compact_us", compact_only)):
        g_c = capture(fn, range(R))
        with torch.cuda.stream(stream):
            g_c.replay()
            q0 = torch.cuda.Event(enable_timing=True)
            q1 = torch.cuda.Event(enable_timing=True)
            q0.record(stream)
            for _ in range(reps):
                g_c.replay()
            q1.record(stream)
        torch.cuda.synchronize(dev)
        comp_us[tag] = q0.elapsed_time(q1) / (reps * R) * 1e3
    # bytes a compaction must move: the mask (1 B per vertex), row_of (4 B per
    # vertex), the coordinates (8 B per active row), the frame offsets
    comp_bytes = B * V * (1 + 4) + 8 * mean_rows + 4 * (B + 1)
    # with the mapping: + the slot-major rulebook entries of the active rows
    map_bytes = comp_bytes + 4 * L * mean_rows
    compaction = {
        "compact_us": comp_us["compact_us"],
        "compact_gbs": comp_bytes / (comp_us["compact_us"] * 1e-6) / 1e9,
        "compact_map_us": comp_us["compact_map_us"],
        "compact_map_gbs": map_bytes / (comp_us["compact_map_us"] * 1e-6) / 1e9,
        "conv_us": conv_ms * 1e3,
        "step_us": ms / K * 1e3,
        "peak_gbs": pk["hbm_gbs"],
        "note": "latency-bound: ~1.7 MB per call; the fraction of HBM bandwidth is not its bound",
    }

    sweep = gnorm = mscore = bwd = kap = cfgs = stg = None
    if not args.no_extras and rank == 0:
        want = lambda name: args.extra in ("all", name)  # noqa: E731
        if want("sweep"):
            sweep = run_sweep(torch, hc, dev, stream)
        if want("group_norm"):
            gnorm = run_group_norm(torch, hc, sets, dev, stream, Wt, bias)
        if want("mask_score"):
            mscore = run_mask_score(torch, hc, dev, stream)
        if want("backward"):
            bwd = run_backward(torch, hc, sets[1], w, spiral, Wt, dev, stream)
        if want("kappa"):
            kap = run_kappa(torch, hc, dev, stream)
        if want("configs"):
            cfgs = run_configs(torch, hc, dev, stream)
        if want("stages"):
            stg = run_stages(torch, hc, sets[0], w, dev, stream)

    # Aggregate over ranks: rows summed, time = max over ranks.
    tot_rows, max_ms = reduce_over_ranks(float(rows_timed), ms, world, dev)
    if rank != 0:
        return None

    cpu = cpu_baseline(w)
    value = tot_rows / (max_ms * 1e-3)
    line = {
        "metric": METRIC,
        "value": value,
        "unit": "rows/s",
        "n_gpus": world,
        "steps": K,
        "warmup": args.warmup,
        "ms_per_step": max_ms / K,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic",
        "impl": "ours",
        "config": {
            "workload": WORKLOAD,
            "B": B, "V": V, "L": L, "C_in": ly.C_in, "C_out": ly.C_out, "act": "elu",
            "mask": "clustered, 8 caps per frame, ~5% active",
            "active_rows_per_step": mean_rows,
            "rotation_sets": R,
            "launches_before_timed": (args.warmup + R) * kernels_per_step,
            "step": "hc_mask_compact_rulebook (count pass + fused compaction/Eq. 4 mapping) "
                    "+ hc_sparse_conv_rulebook_fwd (compact rows + scatter to dense "
                    "[B,V,C_out] fused in its epilogue)",
            "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
            "l2": f"{R} rotating input sets of {set_bytes / 2**20:.1f} MiB "
                  f"({R * set_bytes / 2**20:.0f} MiB > 2x L2 {l2 / 2**20:.0f} MiB)",
            "timing": f"CUDA events around CUDA-graph replays on the bench stream; median of "
                      f"{len(reps_ms)} repeats of exactly {K} steps",
        },
        "roofline": {
            "kernel": "conv_tc_kernel<128> (sparse spiral conv, tcgen05)",
            "bound": "tensor",
            "achieved": achieved,
            "peak": pk["bf16_tflops"],
            "unit": "TFLOP/s",
            "frac": achieved / pk["bf16_tflops"],
            "peak_source": f"{pk['source']} bf16 burst",
            "traffic": traffic,
            "flops_per_launch": flops_per_launch,
            "launch_us": conv_ms * 1e3,
            "kernel_source_hash": khash if traffic is not None else kernel_source_hash(),
        },
        "dense": {
            "hc_spiral_conv_fwd_us": dense_ms * 1e3,
            "torch_gather_matmul_us": torch_dense_ms * 1e3,
            "sparse_conv_us": conv_ms * 1e3,
            "sparse_step_us": max_ms / K * 1e3,
            "speedup_conv_vs_dense": best_dense / conv_ms,
            "speedup_step_vs_dense": best_dense / (max_ms / K),
            "dense_tflops": 2.0 * L * ly.C_in * ly.C_out * B * V / (dense_ms * 1e-3) / 1e12,
        },
        "cpu_baseline": cpu,
        "e2e": e2e,
        "gpu_launches": K * kernels_per_step,
        "clocks": clocks,
    }
    if sweep is not None:
        line["sweep"] = sweep
    if gnorm is not None:
        line["group_norm"] = gnorm
    if mscore is not None:
        line["mask_score"] = mscore
    if bwd is not None:
        line["backward"] = bwd
    if kap is not None:
        line["kappa_inference"] = kap
    if cfgs is not None:
        line["configs"] = cfgs
    if stg is not None:
        line["stages"] = stg
    line["compaction"] = compaction
    return line


def time_torch_dense(torch, sets, w, Wt, bias, stream, dev):
    """torch reference of the dense layer: gather the spiral rows
    (index_select), one bf16 matmul, bias, ELU."""
    ly = w.layers[0]
    B, V, L = w.B, w.V, w.L
    idx = torch.from_numpy(w.spiral.astype(np.int64).ravel()).to(dev)

    def run(s):
        g = s.x.index_select(1, idx).view(B * V, L * ly.C_in)
        return torch.nn.functional.elu(torch.addmm(bias.to(torch.bfloat16), g, Wt))

    with torch.cuda.stream(stream):
        for s in sets[:2]:
            run(s)
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        t0.record(stream)
        for s in sets:
            run(s)
        t1.record(stream)
    torch.cuda.synchronize(dev)
    return t0.elapsed_time(t1) / len(sets)


def measure_e2e(torch, hc, sets, w, spiral, Wt, bias, stream, dev, steps, in_flight):
    """Same metric through the C-ABI with host inputs and outputs: every step
    copies its mask from pinned host memory, compacts it and builds the Eq. 4
    mapping (compact layout), gathers the active rows of its dense features
    straight from the pinned host buffer (hc_gather_rows reading host memory:
    only the active rows cross the host link), runs the conv on those compact
    rows (with the fused scatter), and writes its results to pinned host
    memory: the count (a copy), the coordinates and the compact output rows
    (hc_gather_rows in row order, the copy sized by the count on the device,
    so the host never waits for N' inside the loop). A step is one CUDA graph
    per buffer set: step i runs on buffer set i % in_flight, which always
    takes input set (i % in_flight) % len(sets), each buffer set with its own
    stream (and so its own library workspace), as a serving loop with that
    many requests in flight would run them. Every step moves the inputs it
    uses and all of its results."""
    ly = w.layers[0]
    B, V = w.B, w.V
    host = []
    for s in sets:
        host.append((s.mask.cpu().pin_memory(), s.x.cpu().pin_memory()))
    nb = max(1, in_flight)
    streams = [stream] + [torch.cuda.Stream(device=dev) for _ in range(nb - 1)]
    mask_d = [torch.empty_like(sets[0].mask) for _ in range(nb)]
    outs = []  # device buffers of buffer set b (the input sets' own buffers stay as they are)
    for _ in range(nb):
        o = LayerSet()
        o.coords = torch.empty((B * V, 2), dtype=torch.int32, device=dev)
        o.row_of = torch.empty((B, V), dtype=torch.int32, device=dev)
        o.offs = torch.empty((B + 1,), dtype=torch.int32, device=dev)
        o.count = torch.empty((1,), dtype=torch.int32, device=dev)
        o.rb = torch.empty((w.L, B * V), dtype=torch.int32, device=dev)
        o.xc = torch.empty((B * V, ly.C_in), dtype=torch.bfloat16, device=dev)
        o.y = torch.empty((B * V, ly.C_out), dtype=torch.bfloat16, device=dev)
        o.out = torch.zeros((B, V, ly.C_out), dtype=torch.bfloat16, device=dev)
        outs.append(o)
    cnt_h = [torch.empty((1,), dtype=torch.int32).pin_memory() for _ in range(nb)]
    y_h = [torch.empty((B * V, ly.C_out), dtype=torch.bfloat16).pin_memory() for _ in range(nb)]
    c_h = [torch.empty((B * V, 2), dtype=torch.int32).pin_memory() for _ in range(nb)]

    def step(b):
        mh, xh = host[b % len(host)]
        o = outs[b]
        st = streams[b]
        mask_d[b].copy_(mh, non_blocking=True)
        hc.hc_mask_compact_rulebook(mask_d[b], spiral, hc.HC_LAYOUT_COMPACT, o.coords,
                                    o.row_of, o.offs, o.count, o.rb, st)
        hc.hc_gather_rows(xh, o.coords, o.count, 1, o.xc, st)  # rows from host memory
        hc.hc_sparse_conv_rulebook_fwd(o.xc, o.rb, o.count, Wt, bias, ly.act, o.y,
                                       coords=o.coords, out=o.out, stream=st)
        cnt_h[b].copy_(o.count, non_blocking=True)
        # the first N' coordinates and rows, into pinned host memory
        hc.hc_gather_rows(o.coords.view(torch.float32).view(1, B * V, 2), None, o.count, 1,
                          c_h[b].view(torch.float32), st)
        hc.hc_gather_rows(o.y.view(1, B * V, ly.C_out), None, o.count, 1, y_h[b], st)

    # one CUDA graph per buffer set, captured on its stream
    for b in range(nb):
        with torch.cuda.stream(streams[b]):
            step(b)
    torch.cuda.synchronize(dev)
    graphs = []
    for b in range(nb):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=streams[b]):
            step(b)
        graphs.append(g)
    acc = {"h2d": 0, "d2h": 0, "rows": 0}

    def run(k):
        for i in range(k):
            b = i % nb
            with torch.cuda.stream(streams[b]):
                graphs[b].replay()
            j = b % len(host)
            n = sets[j].rows  # the count this input set's mask gives (checked below)
            acc["h2d"] += host[j][0].numel() + n * ly.C_in * 2  # mask + active feature rows
            acc["d2h"] += 4 + n * 8 + n * ly.C_out * 2
            acc["rows"] += n
        torch.cuda.synchronize(dev)

    run(4)  # warm-up
    for key in acc:
        acc[key] = 0
    torch.cuda.synchronize(dev)
    t0 = time.perf_counter()
    run(steps)
    dt = time.perf_counter() - t0
    # the last step's results as written to host memory, against the same
    # input set's from the device-resident step timed above
    b = (steps - 1) % nb
    s_ref = sets[b % len(host)]
    n = int(cnt_h[b][0])
    same = (n == s_ref.rows and
            torch.equal(y_h[b][:n], s_ref.y[:n].cpu()) and
            torch.equal(c_h[b][:n], s_ref.coords[:n].cpu()))
    return {"value": acc["rows"] / dt, "unit": "rows/s", "steps": steps,
            "rows": acc["rows"], "seconds": dt,
            "rows_match_device_step": bool(same),
            "h2d_bytes_per_step": acc["h2d"] // steps, "d2h_bytes_per_step": acc["d2h"] // steps,
            "ms_per_step": dt / steps * 1e3,
            "path": "pinned host mask (copied) + pinned host features (active rows gathered "
                    "by hc_gather_rows over the host link) -> hc_mask_compact_rulebook, "
                    "hc_gather_rows, hc_sparse_conv_rulebook_fwd -> count (copied), coords "
                    "and rows (hc_gather_rows in row order, sized on the device) into pinned "
                    f"host memory; one CUDA graph per step, {nb} buffer sets on {nb} streams, "
                    "no host wait inside the loop"}


def run_sweep(torch, hc, dev, stream):
    """Mask-density sweep at V = 10475, L = 9, B = 64, 128 -> 128 channels:
    sparse conv (compaction and Eq. 4 mapping done beforehand) against the
    dense layer. tensor_frac counts the work the kernel issues (every tap of
    every active row, absent taps as zero rows: the dense-K formulation);
    tensor_frac_present only the present taps' work (Eq. 5's sum). The
    *_hinted fields time hc_sparse_conv_rulebook_fwd_hint with the mask's
    row count (known here on the host, where the mask was made) as the
    estimate: same results, the tiling chosen for that many rows."""
    from paper_2608_09388_gb300 import inputs
    w = inputs.make_workload("sweep10475_bf16")
    ly = w.layers[0]
    B, V, L = w.B, w.V, w.L
    x = torch.from_numpy(w.x.view(np.int16)).view(torch.bfloat16).to(dev)
    spiral = torch.from_numpy(w.spiral).to(dev)
    Wt = torch.from_numpy(ly.W.view(np.int16)).view(torch.bfloat16).to(dev)
    bias = torch.from_numpy(ly.b).to(dev)
    y = torch.empty((B * V, ly.C_out), dtype=torch.bfloat16, device=dev)
    coords = torch.empty((B * V, 2), dtype=torch.int32, device=dev)
    row_of = torch.empty((B, V), dtype=torch.int32, device=dev)
    offs = torch.empty((B + 1,), dtype=torch.int32, device=dev)
    count = torch.empty((1,), dtype=torch.int32, device=dev)
    rb = torch.empty((L, B * V), dtype=torch.int32, device=dev)
    pk = peaks()

    def timeit(fn, reps=20):
        with torch.cuda.stream(stream):
            fn()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                for _ in range(reps):
                    fn()
            g.replay()
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record(stream)
            g.replay()
            b.record(stream)
        torch.cuda.synchronize(dev)
        return a.elapsed_time(b) / reps

    yd = torch.empty((B, V, ly.C_out), dtype=torch.bfloat16, device=dev)
    dense_ms = timeit(lambda: hc.hc_spiral_conv_fwd(x, spiral, Wt, bias, ly.act, yd, stream), 5)
    out = []
    for d, m in zip(w.densities, w.masks):
        mt = torch.from_numpy(m).to(dev)
        with torch.cuda.stream(stream):
            hc.hc_mask_compact_rulebook(mt, spiral, hc.HC_LAYOUT_DENSE, coords, row_of, offs,
                                        count, rb, stream)
        n = int(np.count_nonzero(m))
        ms = timeit(lambda: hc.hc_sparse_conv_rulebook_fwd(x, rb, count, Wt, bias, ly.act, y,
                                                           stream=stream))
        ms_h = timeit(lambda: hc.hc_sparse_conv_rulebook_fwd_hint(x, rb, count, Wt, bias, ly.act,
                                                                  y, n, stream=stream))
        per_tap = 2.0 * ly.C_in * ly.C_out
        fl = per_tap * L * n
        present = per_tap * float((rb[:, :n] >= 0).sum().item())
        tf = lambda f, t: f / (t * 1e-3) / 1e12 / pk["bf16_tflops"]  # noqa: E731
        out.append({"density": d, "active_rows": n, "sparse_us": ms * 1e3,
                    "dense_us": dense_ms * 1e3, "speedup": dense_ms / ms,
                    "rows_per_s": n / (ms * 1e-3),
                    "work_present_of_issued": present / fl,
                    "tensor_frac": tf(fl, ms),
                    "tensor_frac_present": tf(present, ms),
                    "sparse_hinted_us": ms_h * 1e3, "speedup_hinted": dense_ms / ms_h,
                    "tensor_frac_hinted": tf(fl, ms_h)})
    st = hc.hc_get_device_status(stream)
    if st != hc.HC_OK:
        raise RuntimeError(f"device status {hc.STATUS_NAMES.get(st)} in the sweep")
    return out


def run_group_norm(torch, hc, sets, dev, stream, Wt, bias, G=8):
    """Sparse group norm (Eqs. 7-9), G = 8, affine + ELU, on two inputs:
    the bench layer's compact conv outputs (rotating over the input sets;
    they sit in L2 as they would right after the conv) and a fully active
    64 x 10475 x 128 bf16 activation (171 MB, larger than L2). Algorithmic
    bytes: every active element read once and written once. Then the whole
    layer conv -> group norm -> ELU on the rotating sets: the convolution
    alone (no activation), the two calls, and hc_sparse_conv_gn_fwd (group
    statistics from the convolution's epilogue)."""
    pk = peaks()
    C = sets[0].y.shape[1]
    gamma = torch.linspace(0.5, 1.5, C, device=dev)
    beta = torch.linspace(-0.1, 0.1, C, device=dev)
    with torch.cuda.stream(stream):  # each set's compaction buffers from its own mask
        for s in sets:
            hc.hc_mask_compact(s.mask, s.coords, s.row_of, s.offs, s.count, stream)
    torch.cuda.synchronize(dev)
    for s in sets:
        assert int(s.count.item()) == s.rows
        s.gn = torch.empty_like(s.y)

    def timeit(fns, reps):
        with torch.cuda.stream(stream):
            for f in fns:
                f()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                for _ in range(reps):
                    for f in fns:
                        f()
            g.replay()
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record(stream)
            g.replay()
            b.record(stream)
        torch.cuda.synchronize(dev)
        return a.elapsed_time(b) / (reps * len(fns))

    def gn(x, offs, y):
        return lambda: hc.hc_sparse_group_norm_fwd(x, offs, G, 1e-5, gamma, beta, hc.HC_ACT_ELU,
                                                   y, stream)

    out = {"G": G, "act": "elu", "affine": True}
    ms = timeit([gn(s.y[:s.rows], s.offs, s.gn[:s.rows]) for s in sets], 10)
    rows = sum(s.rows for s in sets) / len(sets)
    nbytes = 2 * rows * C * 2
    out["layer_output"] = {"rows": rows, "C": C, "us": ms * 1e3,
                           "gbs": nbytes / (ms * 1e-3) / 1e9,
                           "hbm_frac": nbytes / (ms * 1e-3) / 1e9 / pk["hbm_gbs"],
                           "kernels": "group_norm_slice_kernel (one block per frame and group)",
                           "note": "compact conv outputs of the bench layer, L2-resident"}
    def conv(s):
        return lambda: hc.hc_sparse_conv_rulebook_fwd(s.x, s.rb, s.count, Wt, bias,
                                                      hc.HC_ACT_NONE, s.gn, stream=stream)

    def fused(s):
        return lambda: hc.hc_sparse_conv_gn_fwd(s.x, s.rb, s.count, Wt, bias, s.coords, s.offs,
                                                G, 1e-5, gamma, beta, hc.HC_ACT_ELU, s.gn,
                                                stream)

    layer = {"rows": rows, "C_out": C,
             "note": "rotating input sets, inputs larger than L2 over a rotation"}
    layer["conv_us"] = timeit([conv(s) for s in sets], 10) * 1e3
    # conv then group norm in place: two calls, three launches
    layer["two_calls_us"] = timeit([f for s in sets for f in (conv(s), gn(s.gn[:s.rows], s.offs,
                                                                         s.gn[:s.rows]))],
                                   10) * 2e3
    layer["fused_us"] = timeit([fused(s) for s in sets], 10) * 1e3
    layer["gn_added_us"] = {"two_calls": layer["two_calls_us"] - layer["conv_us"],
                            "fused": layer["fused_us"] - layer["conv_us"]}
    layer["kernels"] = "conv_tc_kernel (statistics in the epilogue) + gn_apply_kernel"
    out["conv_layer"] = layer
    for s in sets:
        del s.gn
    Bl, Vl = 64, 10475
    x = torch.randn((Bl * Vl, C), device=dev).to(torch.bfloat16)
    y = torch.empty_like(x)
    offs = (torch.arange(Bl + 1, device=dev, dtype=torch.int32) * Vl).contiguous()
    ms = timeit([gn(x, offs, y)], 10)
    nbytes = 2 * x.numel() * 2
    gbs = nbytes / (ms * 1e-3) / 1e9
    out["large"] = {"rows": Bl * Vl, "C": C, "bytes": nbytes, "us": ms * 1e3, "gbs": gbs,
                    "kernels": "gn_stats_kernel + gn_apply_kernel (contiguous row ranges)",
                    "hbm_frac": gbs / pk["hbm_gbs"],
                    "peak": f"{pk['hbm_gbs']} GB/s ({pk['source']} copy)"}
    st = hc.hc_get_device_status(stream)
    if st != hc.HC_OK:
        raise RuntimeError(f"device status {hc.STATUS_NAMES.get(st)} in group norm")
    del x, y
    torch.cuda.empty_cache()
    return out


def run_mask_score(torch, hc, dev, stream, K=10):
    """Mask-score update (Eq. 3) for K = 10 masks, bf16 outputs, on the
    4-layer encoder's output rows (64 frames x 655 vertices, 64 features)
    and on a large layer's (32 frames x 10475 vertices, 128 features).
    Algorithmic work: the symmetric Gram matrix of the [N, K*D] outputs,
    N * KD * (KD + 1) flops (its upper triangle and diagonal)."""
    pk = peaks()
    out = {"K": K, "dtype": "bf16",
           "kernels": "gram_tc_kernel (tcgen05 split-K Gram tiles) + pair_kernel + alpha_kernel"}
    for name, N, D in (("encoder_outputs", 64 * 655, 64), ("large_layer", 32 * 10475, 128)):
        g = torch.Generator(device=dev)
        g.manual_seed(1234 + D)
        O = torch.randn((K, N, D), generator=g, device=dev).to(torch.bfloat16)
        a_in = torch.zeros(K, device=dev)
        a_out = torch.empty(K, device=dev)
        fn = lambda: hc.hc_mask_score_update(O, a_in, a_out, None, stream)  # noqa: E731
        reps = 20 if N < 100000 else 5
        with torch.cuda.stream(stream):
            fn()
            gr = torch.cuda.CUDAGraph()
            with torch.cuda.graph(gr, stream=stream):
                for _ in range(reps):
                    fn()
            gr.replay()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            gr.replay()
            e1.record(stream)
        torch.cuda.synchronize(dev)
        ms = e0.elapsed_time(e1) / reps
        KD = K * D
        flops = float(N) * KD * (KD + 1)
        tf = flops / (ms * 1e-3) / 1e12
        out[name] = {"N": N, "D": D, "us": ms * 1e3, "tflops": tf,
                     "tensor_frac": tf / pk["bf16_tflops"],
                     "input_bytes": O.numel() * 2,
                     "peak": f"{pk['bf16_tflops']} TFLOP/s ({pk['source']} bf16 burst)"}
        del O
    st = hc.hc_get_device_status(stream)
    if st != hc.HC_OK:
        raise RuntimeError(f"device status {hc.STATUS_NAMES.get(st)} in the mask score")
    torch.cuda.empty_cache()
    return out


def run_backward(torch, hc, s, w, spiral, Wt, dev, stream):
    """Backward of the bench layer (one input set: its mask, rulebook and
    forward output), with an upstream gradient drawn on the device:
    the transposed mapping (once per mask), then the full backward (input,
    weight and bias gradients), and its weight-gradient and input-gradient
    parts alone. Weight-gradient roofline: 2 * N' * L*C_in * C_out flops."""
    pk = peaks()
    ly = w.layers[0]
    B, V, L = w.B, w.V, w.L
    cap = B * V
    K = L * ly.C_in
    g = torch.Generator(device=dev)
    g.manual_seed(4321)
    dy = torch.randn((cap, ly.C_out), generator=g, device=dev).to(torch.bfloat16)
    x = s.x.view(cap, ly.C_in)
    row_ptr = torch.empty(cap + 1, dtype=torch.int32, device=dev)
    taps = torch.empty(L * cap, dtype=torch.int32, device=dev)
    dx = torch.empty_like(x)
    dW = torch.empty((K, ly.C_out), device=dev)
    db = torch.empty(ly.C_out, device=dev)

    def transpose():
        hc.hc_conv_rulebook_transpose(s.rb, s.count, cap, row_ptr, taps, stream)

    def bwd(dx_, dW_, db_):
        return lambda: hc.hc_sparse_conv_rulebook_bwd(x, s.rb, s.count, Wt, s.y, dy, ly.act,
                                                      row_ptr, taps, dx_, dW_, db_, stream)

    def timeit(fn, reps=20):
        with torch.cuda.stream(stream):
            fn()
            gr = torch.cuda.CUDAGraph()
            with torch.cuda.graph(gr, stream=stream):
                for _ in range(reps):
                    fn()
            gr.replay()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            gr.replay()
            e1.record(stream)
        torch.cuda.synchronize(dev)
        return e0.elapsed_time(e1) / reps * 1e3

    t_tr = timeit(transpose)
    t_all = timeit(bwd(dx, dW, db))
    t_w = timeit(bwd(None, dW, None))
    t_x = timeit(bwd(dx, None, None))
    st = hc.hc_get_device_status(stream)
    if st != hc.HC_OK:
        raise RuntimeError(f"device status {hc.STATUS_NAMES.get(st)} in the backward")
    flops = 2.0 * s.rows * K * ly.C_out
    tf = flops / (t_w * 1e-6) / 1e12
    return {"workload": WORKLOAD, "active_rows": s.rows, "dtype": "bf16",
            "transpose_us": t_tr, "bwd_us": t_all, "wgrad_part_us": t_w, "dgrad_part_us": t_x,
            "wgrad_tflops": tf, "wgrad_tensor_frac": tf / pk["bf16_tflops"],
            "kernels": "act_bwd + wgrad_tc_kernel (tcgen05 split-K) + wgrad_reduce; "
                       "W^T + linear conv (dz W^T) + dgrad gather-sum",
            "peak": f"{pk['bf16_tflops']} TFLOP/s ({pk['source']} bf16 burst)"}


def run_kappa(torch, hc, dev, stream, K=10, kappa=3, density=0.1):
    """Inference with kappa kept masks (Sec. 3.1; kappa = 3 of K = 10 as in
    Sec. 4) on the 4-layer bf16 encoder (64 samples of the 655-vertex sphere,
    16 -> 64 -> 64 -> 64 -> 64 + linear 64 -> 42): top-kappa by the mask
    score, every kept mask on every sample (192 frames), compaction, the Eq. 4
    mapping, the S' rows of Eq. 2 gathered from the samples, the four sparse
    conv layers and the head, all on compact rows. Against the same encoder
    run densely on every vertex of the 64 samples."""
    from paper_2608_09388_gb300 import inputs
    w = inputs.make_workload("encoder655_bf16")
    B, V, L = w.B, w.V, w.L
    F = B * kappa
    rng = np.random.default_rng(inputs.SEEDS["encoder655_bf16"] + 77)
    masks = torch.from_numpy(inputs.uniform_mask(rng, K, V, density)).to(dev)
    alpha = torch.from_numpy(rng.standard_normal(K).astype(np.float32)).to(dev)
    x = torch.from_numpy(w.x.view(np.int16)).view(torch.bfloat16).to(dev)
    sp = torch.from_numpy(w.spiral).to(dev)
    Ws = [torch.from_numpy(ly.W.view(np.int16)).view(torch.bfloat16).to(dev) for ly in w.layers]
    bs = [torch.from_numpy(ly.b).to(dev) for ly in w.layers]
    sel = torch.empty(kappa, dtype=torch.int32, device=dev)
    fm = torch.empty((F, V), dtype=torch.uint8, device=dev)
    coords = torch.empty((F * V, 2), dtype=torch.int32, device=dev)
    row_of = torch.empty((F, V), dtype=torch.int32, device=dev)
    offs = torch.empty(F + 1, dtype=torch.int32, device=dev)
    count = torch.empty(1, dtype=torch.int32, device=dev)
    rb = torch.empty((L, F * V), dtype=torch.int32, device=dev)
    hs = [torch.empty((F * V, ly.C_in), dtype=torch.bfloat16, device=dev) for ly in w.layers]
    out = torch.empty((F * V, w.layers[-1].C_out), dtype=torch.bfloat16, device=dev)
    dense_h = [torch.empty((B, V, ly.C_out), dtype=torch.bfloat16, device=dev) for ly in w.layers]

    def sparse():
        hc.hc_mask_select_topk(alpha, kappa, sel, stream)
        hc.hc_kappa_masks(masks, sel, B, fm, stream)
        hc.hc_mask_compact_rulebook(fm, sp, hc.HC_LAYOUT_COMPACT, coords, row_of, offs, count,
                                    rb, stream)
        hc.hc_gather_rows(x, coords, count, kappa, hs[0], stream)
        for i, ly in enumerate(w.layers):
            dst = hs[i + 1] if i + 1 < len(w.layers) else out
            if ly.kind == "conv":
                hc.hc_sparse_conv_rulebook_fwd(hs[i], rb, count, Ws[i], bs[i], ly.act, dst,
                                               stream=stream)
            else:
                hc.hc_sparse_linear_fwd(hs[i], count, Ws[i], bs[i], ly.act, dst, stream)

    def dense():
        h = x
        for i, ly in enumerate(w.layers):
            if ly.kind == "conv":
                hc.hc_spiral_conv_fwd(h, sp, Ws[i], bs[i], ly.act, dense_h[i], stream)
            else:
                hc.hc_sparse_linear_fwd(h.view(B * V, -1), full, Ws[i], bs[i], ly.act,
                                        dense_h[i].view(B * V, -1), stream)
            h = dense_h[i]

    full = torch.tensor([B * V], dtype=torch.int32, device=dev)

    def timeit(fn, reps=20):
        with torch.cuda.stream(stream):
            fn()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                for _ in range(reps):
                    fn()
            g.replay()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            g.replay()
            e1.record(stream)
        torch.cuda.synchronize(dev)
        return e0.elapsed_time(e1) / reps * 1e3

    t_sparse = timeit(sparse)
    t_dense = timeit(dense)
    st = hc.hc_get_device_status(stream)
    if st != hc.HC_OK:
        raise RuntimeError(f"device status {hc.STATUS_NAMES.get(st)} in the kappa inference")
    n = int(count.item())
    return {"K": K, "kappa": kappa, "samples": B, "frames": F, "V": V, "mask_density": density,
            "active_rows": n, "layers": "4 sparse spiral convs 16-64-64-64-64 + linear 64->42",
            "us": t_sparse, "rows_per_s": n / (t_sparse * 1e-6),
            "dense_encoder_us": t_dense, "speedup_vs_dense": t_dense / t_sparse,
            "chain": "topk + kappa masks + compaction + Eq. 4 mapping + S' gather + 4 convs + "
                     "linear head (compact rows throughout)"}


def run_stages(torch, hc, s, w, dev, stream):
    """The HBM-bound stages of the path on one input set of the bench layer,
    each timed alone (CUDA-graph replays): the S' row gather (Eq. 2) from the
    dense features, the scatter of the conv's compact rows back to the dense
    tensor (Eq. 2 inverse) without and with the zero fill, and the
    compaction (in the "compaction" block). Achieved GB/s = the bytes each
    must move / time, against the measured HBM copy bandwidth."""
    B, V = w.B, w.V
    C_in = w.layers[0].C_in
    C_out = w.layers[0].C_out
    n = s.rows
    pk = peaks()
    rows_x = torch.empty((B * V, C_in), dtype=torch.bfloat16, device=dev)
    dense = torch.empty((B, V, C_out), dtype=torch.bfloat16, device=dev)
    with torch.cuda.stream(stream):
        hc.hc_mask_compact(s.mask, s.coords, s.row_of, s.offs, s.count, stream)
    cases = {
        "gather_rows": (lambda: hc.hc_gather_rows(s.x, s.coords, s.count, 1, rows_x, stream),
                        n * (2 * C_in * 2 + 8)),
        "scatter": (lambda: hc.hc_scatter_dense(s.y, s.coords, None, s.count, B, V, 0, dense,
                                                stream),
                    n * (2 * C_out * 2 + 8)),
        "scatter_zero_fill": (lambda: hc.hc_scatter_dense(s.y, s.coords, s.row_of, s.count, B, V,
                                                          1, dense, stream),
                              B * V * (C_out * 2 + 4) + n * C_out * 2),
    }
    out = {"workload": WORKLOAD, "active_rows": n, "peak_gbs": pk["hbm_gbs"]}
    for name, (fn, nbytes) in cases.items():
        us = _graph_time_us(torch, fn, stream, dev)
        out[name] = {"us": us, "bytes": nbytes, "gbs": nbytes / (us * 1e-6) / 1e9,
                     "hbm_frac": nbytes / (us * 1e-6) / 1e9 / pk["hbm_gbs"]}
    st = hc.hc_get_device_status(stream)
    if st != hc.HC_OK:
        raise RuntimeError(f"device status {hc.STATUS_NAMES.get(st)} in the stage timings")
    return out


def _graph_time_us(torch, fn, stream, dev, reps=20):
    """Mean time of fn over `reps` calls replayed from one CUDA graph (after
    an eager call and one replay), CUDA events on the stream."""
    with torch.cuda.stream(stream):
        fn()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for _ in range(reps):
                fn()
        g.replay()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        g.replay()
        e1.record(stream)
    torch.cuda.synchronize(dev)
    return e0.elapsed_time(e1) / reps * 1e3


def _oracle_rows_per_s(w, threads, budget_s):
    """The oracle's whole stack (compaction, every layer on the compact rows)
    on the first k frames of the workload, k chosen so that the run takes
    about budget_s; returns (active rows per second, frames, rows)."""
    import oracle

    def run(k):
        t0 = time.perf_counter()
        _, _, _, n, _ = oracle.encoder(w.x[:k], w.masks[0][:k], w.spiral, w.layers,
                                       n_threads=threads)
        return time.perf_counter() - t0, n

    t1, n1 = run(1)
    k = max(1, min(w.B, int(budget_s / max(t1, 1e-4))))
    t, n = (t1, n1) if k == 1 else run(k)
    return n / t, k, n


def run_configs(torch, hc, dev, stream, cpu_budget_s=3.0):
    """The other workloads of the scope (655-vertex mesh): the single fp32
    layer, the 4-layer bf16 encoder + 64 -> 42 head, and the 256-frame motion
    encoder + 64 -> 1 head. Each runs as the paper's network would: compact
    once (compaction + Eq. 4 mapping in the compact layout), gather S'
    (Eq. 2), every layer on the compact rows, one CUDA graph; against the
    same network run densely on every vertex, and against the oracle on 1
    thread and on every host core (bounded frame samples).
    Chains: "compact" (compaction + mapping in the compact layout, the S'
    gather, every layer on compact rows) and "dense_layout" (the mapping in
    the dense layout, every conv reading the previous layer's dense rows and
    writing only its active rows back into a dense tensor by the fused
    scatter, the per-vertex head as the rulebook conv on the centre slot:
    no gather launch); the line reports the faster."""
    from paper_2608_09388_gb300 import inputs
    pk = peaks()
    props = torch.cuda.get_device_properties(dev)
    # fp32 FFMA peak: SMs x 128 lanes x 2 flops at the maximum SM clock
    ffma_tflops = props.multi_processor_count * 128 * 2 * 2.07e9 / 1e12
    cores = len(os.sched_getaffinity(0))
    res = {}
    for name in ("layer655_f32", "encoder655_bf16", "motion655_bf16"):
        w = inputs.make_workload(name)
        B, V, L = w.B, w.V, w.L

        def T(a):
            if a.dtype == np.uint16:
                return torch.from_numpy(a.view(np.int16)).view(torch.bfloat16).to(dev)
            return torch.from_numpy(np.ascontiguousarray(a)).to(dev)

        dt = torch.float32 if w.dtype == "f32" else torch.bfloat16
        mask, x, sp = T(w.masks[0]), T(w.x), T(w.spiral)
        Ws = [T(ly.W) for ly in w.layers]
        bs = [T(ly.b) for ly in w.layers]
        coords = torch.empty((B * V, 2), dtype=torch.int32, device=dev)
        row_of = torch.empty((B, V), dtype=torch.int32, device=dev)
        offs = torch.empty(B + 1, dtype=torch.int32, device=dev)
        count = torch.empty(1, dtype=torch.int32, device=dev)
        rb = torch.empty((L, B * V), dtype=torch.int32, device=dev)
        hs = [torch.empty((B * V, ly.C_in), dtype=dt, device=dev) for ly in w.layers]
        out = torch.empty((B * V, w.layers[-1].C_out), dtype=dt, device=dev)
        dense_h = [torch.empty((B, V, ly.C_out), dtype=dt, device=dev) for ly in w.layers]
        full = torch.tensor([B * V], dtype=torch.int32, device=dev)

        def sparse():
            hc.hc_mask_compact_rulebook(mask, sp, hc.HC_LAYOUT_COMPACT, coords, row_of, offs,
                                        count, rb, stream)
            hc.hc_gather_rows(x, coords, count, 1, hs[0], stream)
            for i, ly in enumerate(w.layers):
                dst = hs[i + 1] if i + 1 < len(w.layers) else out
                if ly.kind == "conv":
                    hc.hc_sparse_conv_rulebook_fwd(hs[i], rb, count, Ws[i], bs[i], ly.act, dst,
                                                   stream=stream)
                else:
                    hc.hc_sparse_linear_fwd(hs[i], count, Ws[i], bs[i], ly.act, dst, stream)

        # the dense-layout chain: inactive rows of the dense tensors are never
        # read (their taps are absent in the rulebook)
        rb_d = torch.empty((L, B * V), dtype=torch.int32, device=dev)
        dense_a = [torch.empty((B, V, ly.C_out), dtype=dt, device=dev) for ly in w.layers]

        def sparse_dense_layout():
            hc.hc_mask_compact_rulebook(mask, sp, hc.HC_LAYOUT_DENSE, coords, row_of, offs,
                                        count, rb_d, stream)
            h = x
            for i, ly in enumerate(w.layers):
                last = i + 1 == len(w.layers)
                taps = rb_d if ly.kind == "conv" else rb_d[0:1]  # centre slot: a 1x1 layer
                if last:
                    hc.hc_sparse_conv_rulebook_fwd(h, taps, count, Ws[i], bs[i], ly.act, out,
                                                   stream=stream)
                else:
                    hc.hc_sparse_conv_rulebook_fwd(h, taps, count, Ws[i], bs[i], ly.act, None,
                                                   coords=coords, out=dense_a[i], stream=stream)
                h = dense_a[i]

        def dense():
            h = x
            for i, ly in enumerate(w.layers):
                if ly.kind == "conv":
                    hc.hc_spiral_conv_fwd(h, sp, Ws[i], bs[i], ly.act, dense_h[i], stream)
                else:
                    hc.hc_sparse_linear_fwd(h.view(B * V, -1), full, Ws[i], bs[i], ly.act,
                                            dense_h[i].view(B * V, -1), stream)
                h = dense_h[i]

        t_compact = _graph_time_us(torch, sparse, stream, dev)
        y_compact = out[:int(count.item())].clone()
        t_dl = _graph_time_us(torch, sparse_dense_layout, stream, dev)
        same = bool(torch.equal(out[:int(count.item())], y_compact))
        t_sparse = min(t_compact, t_dl)
        t_dense = _graph_time_us(torch, dense, stream, dev)
        st = hc.hc_get_device_status(stream)
        if st != hc.HC_OK:
            raise RuntimeError(f"device status {hc.STATUS_NAMES.get(st)} in {name}")
        n = int(count.item())
        flops = sum(2.0 * (L if ly.kind == "conv" else 1) * ly.C_in * ly.C_out * n
                    for ly in w.layers)
        peak = pk["bf16_tflops"] if w.dtype == "bf16" else ffma_tflops
        achieved = flops / (t_sparse * 1e-6) / 1e12
        o1, k1, n1 = _oracle_rows_per_s(w, 1, cpu_budget_s)
        on, kn, nn = _oracle_rows_per_s(w, cores, cpu_budget_s)
        res[name] = {
            "B": B, "V": V, "L": L, "dtype": w.dtype, "active_rows": n,
            "layers": " -> ".join([str(w.layers[0].C_in)] + [str(ly.C_out) for ly in w.layers]),
            "us": t_sparse, "rows_per_s": n / (t_sparse * 1e-6),
            "gflops": flops / (t_sparse * 1e-6) / 1e9,
            "roofline": {"bound": "tensor" if w.dtype == "bf16" else "alu", "achieved": achieved,
                         "peak": peak, "unit": "TFLOP/s", "frac": achieved / peak,
                         "peak_source": "measured bf16 burst" if w.dtype == "bf16" else
                         "FFMA: SMs x 128 x 2 x 2.07 GHz",
                         "note": "latency-bound: a few thousand rows per launch"},
            "dense_us": t_dense, "speedup_vs_dense": t_dense / t_sparse,
            "oracle_1_thread": {"rows_per_s": o1, "frames": k1, "rows": n1, "cores": 1},
            "oracle_all_cores": {"rows_per_s": on, "frames": kn, "rows": nn, "cores": cores},
            "chain": ("dense_layout" if t_dl < t_compact else "compact") + " (one CUDA graph)",
            "chains_us": {"compact": t_compact, "dense_layout": t_dl},
            "chains_same_output": same,
        }
    return res


def run_case(args):
    """One call, args.steps times in a row, each timed with CUDA events: a
    small, fixed launch sequence for a profiler to capture. A layer of the
    density sweep's workload (V = 10475, L = 9, B = 64, 128 -> 128), or the
    mask-score update on the encoder outputs."""
    import torch

    from paper_2608_09388_gb300 import build as hc_build
    from paper_2608_09388_gb300 import hc, inputs
    hc_build.build()
    hc.load_library()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    stream = torch.cuda.Stream(device=dev)
    w = inputs.make_workload("sweep10475_bf16")
    ly = w.layers[0]
    B, V, L = w.B, w.V, w.L
    x = torch.from_numpy(w.x.view(np.int16)).view(torch.bfloat16).to(dev)
    spiral = torch.from_numpy(w.spiral).to(dev)
    Wt = torch.from_numpy(ly.W.view(np.int16)).view(torch.bfloat16).to(dev)
    bias = torch.from_numpy(ly.b).to(dev)
    if args.case == "mask-score":
        g = torch.Generator(device=dev)
        g.manual_seed(1234 + 64)
        O = torch.randn((10, 64 * 655, 64), generator=g, device=dev).to(torch.bfloat16)
        a_in = torch.zeros(10, device=dev)
        a_out = torch.empty(10, device=dev)
        fn = lambda: hc.hc_mask_score_update(O, a_in, a_out, None, stream)  # noqa: E731
        rows = 64 * 655
    elif args.case == "sweep-dense":
        yd = torch.empty((B, V, ly.C_out), dtype=torch.bfloat16, device=dev)
        fn = lambda: hc.hc_spiral_conv_fwd(x, spiral, Wt, bias, ly.act, yd, stream)  # noqa: E731
        rows = B * V
    elif args.case.startswith("sweep:"):
        d = float(args.case.split(":", 1)[1])
        if d not in w.densities:
            raise SystemExit(f"--case {args.case}: density not in {list(w.densities)}")
        m = torch.from_numpy(w.masks[list(w.densities).index(d)]).to(dev)
        coords = torch.empty((B * V, 2), dtype=torch.int32, device=dev)
        row_of = torch.empty((B, V), dtype=torch.int32, device=dev)
        offs = torch.empty((B + 1,), dtype=torch.int32, device=dev)
        count = torch.empty((1,), dtype=torch.int32, device=dev)
        rb = torch.empty((L, B * V), dtype=torch.int32, device=dev)
        y = torch.empty((B * V, ly.C_out), dtype=torch.bfloat16, device=dev)
        with torch.cuda.stream(stream):
            hc.hc_mask_compact_rulebook(m, spiral, hc.HC_LAYOUT_DENSE, coords, row_of, offs, count,
                                        rb, stream)
        torch.cuda.synchronize(dev)
        rows = int(count.item())
        fn = lambda: hc.hc_sparse_conv_rulebook_fwd(x, rb, count, Wt, bias, ly.act, y,  # noqa: E731
                                                    stream=stream)
    else:
        raise SystemExit(f"--case {args.case}: expected sweep:D, sweep-dense or mask-score")
    times = []
    for _ in range(args.steps):
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            a.record(stream)
            fn()
            b.record(stream)
        torch.cuda.synchronize(dev)
        times.append(a.elapsed_time(b) * 1e3)
    status = hc.hc_get_device_status()
    print(json.dumps({"case": args.case, "rows": rows, "us": times, "status": status}), flush=True)
    if status != hc.HC_OK:
        raise SystemExit(1)


def cpu_baseline(w, budget_s=20.0):
    """The CPU oracle as it stands on this host's cores: compaction, sparse
    conv and scatter of batch 0 of the workload (all of its active rows when
    that fits the time budget, else a prefix of them, scaled to rows/s)."""
    import oracle
    ly = w.layers[0]
    cores = len(os.sched_getaffinity(0))
    t0 = time.perf_counter()
    coords, row_of, offs, n = oracle.mask_compact(w.masks[0])
    t_compact = time.perf_counter() - t0
    probe = np.arange(min(n, 256), dtype=np.int64)
    t0 = time.perf_counter()
    oracle.sparse_spiral_conv(w.x, oracle.LAYOUT_DENSE, coords, row_of, w.spiral, ly.W, ly.b,
                              ly.act, rows=probe, n_threads=cores)
    per_row = (time.perf_counter() - t0) / max(1, len(probe))
    k = n if per_row * n <= budget_s else max(256, int(budget_s / per_row))
    rows = np.arange(k, dtype=np.int64)
    t0 = time.perf_counter()
    _, y = oracle.sparse_spiral_conv(w.x, oracle.LAYOUT_DENSE, coords, row_of, w.spiral, ly.W,
                                     ly.b, ly.act, rows=rows, n_threads=cores)
    t_conv = time.perf_counter() - t0
    t0 = time.perf_counter()
    oracle.scatter_dense(y, coords[:k], w.B, w.V, False)
    t_scatter = time.perf_counter() - t0
    secs = t_compact * k / max(n, 1) + t_conv + t_scatter
    # the same on one thread, on a prefix of the rows sized to ~budget_s / 4
    t0 = time.perf_counter()
    oracle.sparse_spiral_conv(w.x, oracle.LAYOUT_DENSE, coords, row_of, w.spiral, ly.W, ly.b,
                              ly.act, rows=probe[:64], n_threads=1)
    per_row1 = (time.perf_counter() - t0) / max(1, min(64, len(probe)))
    k1 = max(64, min(n, int(budget_s / 4 / max(per_row1, 1e-7))))
    rows1 = np.arange(k1, dtype=np.int64)
    t0 = time.perf_counter()
    _, y1 = oracle.sparse_spiral_conv(w.x, oracle.LAYOUT_DENSE, coords, row_of, w.spiral, ly.W,
                                      ly.b, ly.act, rows=rows1, n_threads=1)
    t_conv1 = time.perf_counter() - t0
    t0 = time.perf_counter()
    oracle.scatter_dense(y1, coords[:k1], w.B, w.V, False)
    secs1 = t_compact * k1 / max(n, 1) + t_conv1 + time.perf_counter() - t0
    return {"value": k / secs, "unit": "rows/s", "cores": cores, "kind": "oracle",
            "sample": f"batch 0 of {WORKLOAD}: compaction, sparse conv and scatter of "
                      f"{k} of its {n} active rows (fp64 C oracle, OpenMP over rows)",
            "single_thread": {"value": k1 / secs1, "unit": "rows/s", "cores": 1,
                              "sample": f"the first {k1} active rows of batch 0"}}


# ----------------------------------------------------------------- reference arm

def run_reference(args, rank):
    """The CPU oracle, as it stands, timed on this host's cores on bounded
    samples of the same workload: each step computes 512 consecutive active
    rows (compaction pro rata, conv, scatter)."""
    if rank != 0:
        return None
    import oracle
    from paper_2608_09388_gb300 import inputs
    w = inputs.make_workload(WORKLOAD)
    ly = w.layers[0]
    cores = len(os.sched_getaffinity(0))
    t0 = time.perf_counter()
    coords, row_of, offs, n = oracle.mask_compact(w.masks[0])
    t_compact_row = (time.perf_counter() - t0) / max(n, 1)
    per = 512

    def step(i):
        s = (i * per) % max(1, n - per)
        rows = np.arange(s, min(n, s + per), dtype=np.int64)
        _, y = oracle.sparse_spiral_conv(w.x, oracle.LAYOUT_DENSE, coords, row_of, w.spiral, ly.W,
                                         ly.b, ly.act, rows=rows, n_threads=cores)
        oracle.scatter_dense(y, coords[rows], w.B, w.V, False)
        return len(rows)

    for i in range(args.warmup):
        step(i)
    t0 = time.perf_counter()
    done = 0
    for i in range(args.steps):
        done += step(i)
    secs = time.perf_counter() - t0 + t_compact_row * done
    value = done / secs
    return {
        "metric": METRIC, "value": value, "unit": "rows/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": secs / args.steps * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "impl": "reference",
        "config": {"workload": WORKLOAD, "B": w.B, "V": w.V, "L": w.L, "C_in": ly.C_in,
                   "C_out": ly.C_out, "rows_per_step": per},
        "cpu_baseline": {"value": value, "unit": "rows/s", "cores": cores, "kind": "oracle",
                         "sample": f"{per} consecutive active rows of batch 0 per step"},
        "e2e": {"value": value, "unit": "rows/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }


def main():
    args = parse_args()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        line = run_reference(args, rank)
        if line is not None:
            print(json.dumps(line), flush=True)
        return
    if args.case:
        run_case(args)
        return
    import torch
    if world > 1:
        torch.cuda.set_device(local_rank)
        torch.distributed.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    try:
        line = run_ours(args, rank, world, local_rank)
    finally:
        if world > 1:
            torch.distributed.destroy_process_group()
    if line is not None:
        print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
