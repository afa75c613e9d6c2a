#!/usr/bin/env python3
"""Benchmark of the error-feedback sparsification step (arXiv:2108.00951).

One step = one error-feedback iteration of the n simulated workers of a
workload, through the whole hot path:
  - n x ef_hard_threshold (EF accumulate + hard-threshold + compaction +
    residual), then sparse_aggregate of their n messages;
  - n x ef_topk on the same gradients (separate error memories), then
    sparse_aggregate of those messages;
  - n x ef_topk_layerwise (Top-k on each parameter tensor separately, the
    same fraction of every tensor) on the same gradients, then
    sparse_aggregate of those messages;
  - sparse_aggregate_apply of the hard-threshold messages into a model and
    momentum state (the momentum EF SGD update, fused with the exchange);
  - n x ef_scaled_round (scaled integer rounding, another absolute
    compressor: dense int32 messages) on the same gradients, then
    int_aggregate of those messages (exact integer sum).
  - n x ef_hard_threshold_bf16 on the same gradients rounded to bfloat16
    (the bf16-gradient variant, widened exactly in the kernel).
Gradients come from two pre-generated synthetic batches (alternating), so
every step compresses different data; each step's working set (n workers x
(g, e_ht, e_topk)) is far larger than the 126 MB L2.

The default workload is the VGG-16-shaped vector (d = 138,357,544, 8
workers), the largest one that fits one GPU. After the timed steps, further
legs time the rest of the d >= 25 M regime on the same GPU: hard-threshold
and Top-k on the LSTM-shaped vector and on the ResNet-50-shaped vector at
each of its thresholds and Top-k fractions; a cold-L2 variant of the
headline call (L2 flushed before every call); and the latency of the
logistic-regression-sized case (d = 100,000, which fits in L2).

Headline (`value`): hard-threshold compress throughput in GB/s of
algorithmic traffic, 12 B/coordinate (read g, read e, write e) + 8 B per sent
pair, summed over all compress calls of the K timed steps and divided by
their device time (CUDA events on the launching stream). Top-k and
aggregation are reported as ms per iteration and as fractions of the same
HBM roofline. `e2e` repeats the hard-threshold iteration through the public
API with the n gradients copied host->device from pinned memory and the
dense aggregate copied back, every step.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload vgg16]
  python bench.py --harness ht --workload vgg16 --steps 3 --warmup 3
      # one worker's calls only (a few GB on the device), for ncu captures
  python bench.py --impl reference ...   # the CPU oracle as the reference arm

For N > 1 (one process per GPU under torch.distributed.run) every rank runs
its own replica of the workload (weak scaling); ranks only meet in a barrier
and in the max/sum reductions of the timing.
"""
from __future__ import annotations

import argparse
import ctypes
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

PEAK_FALLBACK_GBS = 6800.0
NOMINAL_HBM_GBS = 8000.0
METRIC = "EF hard-threshold compress GB/s & elem/s vs HBM peak; Top-k and aggregate ms/iter"
HT_KERNEL_SOURCES = ["paper_2108_00951_gb300/csrc/ht.cu",
                     "paper_2108_00951_gb300/csrc/stream_compact.cuh",
                     "paper_2108_00951_gb300/csrc/stream_lookback.cuh",
                     "paper_2108_00951_gb300/csrc/tma.cuh",
                     "paper_2108_00951_gb300/csrc/compact.cuh",
                     "paper_2108_00951_gb300/csrc/common.cuh",
                     "paper_2108_00951_gb300/csrc/gradient.cuh"]


def parse_args(argv=None):
    p = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=200)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--workload", default="vgg16")
    p.add_argument("--harness", choices=["ht", "ht_bf16", "topk", "topk_layerwise", "aggregate"],
                   default=None,
                   help="run only one kind of call, for one worker (aggregate: the n workers' "
                        "hard-threshold messages), and print a short summary")
    p.add_argument("--lam-index", type=int, default=0,
                   help="which of the workload's fixed lambdas (or Top-k fractions) to use")
    p.add_argument("--no-extra-legs", action="store_true",
                   help="skip the d >= 25 M regime, cold-L2 and latency legs")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--error-norm", action="store_true",
                   help="every compress call also returns ||e'||^2 (the _ex entries)")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--cpu-seconds", type=float, default=10.0,
                   help="bound on the CPU-oracle sample of the cpu_baseline leg")
    return p.parse_args(argv)


# ------------------------------------------------------------ distributed
def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def dist_init(backend):
    import torch.distributed as dist
    rank, world, _ = dist_env()
    if world > 1 and not dist.is_initialized():
        dist.init_process_group(backend=backend, rank=rank, world_size=world)
    return dist if world > 1 else None


def reduce_timing(dist, seconds: float, units: float, device=None):
    """(max seconds over ranks, sum of units over ranks)."""
    if dist is None:
        return seconds, units
    import torch
    t = torch.tensor([seconds], dtype=torch.float64, device=device)
    u = torch.tensor([units], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    dist.all_reduce(u, op=dist.ReduceOp.SUM)
    return float(t.item()), float(u.item())


def replica_workload(w, rank: int):
    """The workload a rank simulates: every rank runs its own n workers (a
    replica), on gradients drawn from a seed of its own."""
    from paper_2108_00951_gb300 import workloads
    return workloads.Workload(**{**w.__dict__, "seed": w.seed + 1000 * rank})


def barrier(dist, device=None):
    if dist is not None:
        if device is not None and device.type == "cuda":
            dist.barrier(device_ids=[device.index])
        else:
            dist.barrier()


# ------------------------------------------------------------ peaks, clocks
def measured_peak_gbs():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            v = float(json.load(f)["hbm_gbs"])
        return v, "measured"
    except Exception:
        return PEAK_FALLBACK_GBS, "fallback"


class ClockSampler:
    """Samples the SM clock and clock-event reasons of one GPU every ~10 ms
    through NVML (read-only queries), falling back to nvidia-smi."""

    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown",
               0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown"}

    def __init__(self, cuda_index: int):
        self.samples = []
        self.reasons = set()
        self.max_mhz = None
        self._stop = threading.Event()
        self._thread = None
        self._nvml = None
        self._handle = None
        self._smi_index = cuda_index
        try:
            import torch
            lib = ctypes.CDLL("libnvidia-ml.so.1")
            if lib.nvmlInit_v2() != 0:
                raise OSError("nvmlInit failed")
            handle = ctypes.c_void_p()
            uuid = "GPU-" + str(torch.cuda.get_device_properties(cuda_index).uuid)
            if lib.nvmlDeviceGetHandleByUUID(uuid.encode(), ctypes.byref(handle)) != 0:
                raise OSError("no NVML handle")
            mx = ctypes.c_uint()
            if lib.nvmlDeviceGetMaxClockInfo(handle, 1, ctypes.byref(mx)) == 0:
                self.max_mhz = mx.value
            self._nvml, self._handle = lib, handle
        except Exception:
            self._nvml = None

    def _poll_nvml(self):
        clk = ctypes.c_uint()
        rs = ctypes.c_ulonglong()
        get_reasons = getattr(self._nvml, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
            getattr(self._nvml, "nvmlDeviceGetCurrentClocksThrottleReasons")
        while not self._stop.is_set():
            if self._nvml.nvmlDeviceGetClockInfo(self._handle, 1, ctypes.byref(clk)) == 0:
                self.samples.append(clk.value)
            if get_reasons(self._handle, ctypes.byref(rs)) == 0:
                for bit, name in self.REASONS.items():
                    if rs.value & bit:
                        self.reasons.add(name)
            time.sleep(0.01)

    def _poll_smi(self):
        q = ("clocks.sm,clocks.max.sm,clocks_event_reasons.hw_slowdown,"
             "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
             "clocks_event_reasons.sw_power_cap")
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        while not self._stop.is_set():
            try:
                out = subprocess.run(["nvidia-smi", "-i", str(self._smi_index),
                                      "--query-gpu=" + q, "--format=csv,noheader,nounits"],
                                     capture_output=True, text=True, timeout=5).stdout
                f = [x.strip() for x in out.strip().split(",")]
                self.samples.append(float(f[0]))
                self.max_mhz = float(f[1])
                for name, v in zip(names, f[2:]):
                    if v.lower() == "active":
                        self.reasons.add(name)
            except Exception:
                pass
            time.sleep(0.05)

    def start(self):
        self._thread = threading.Thread(target=self._poll_nvml if self._nvml else self._poll_smi,
                                        daemon=True)
        self._thread.start()

    def stop(self):
        self._stop.set()
        if self._thread:
            self._thread.join()
        return {"sm_mhz": statistics.median(self.samples) if self.samples else None,
                "sm_max_mhz": self.max_mhz, "reasons": sorted(self.reasons),
                "samples": len(self.samples), "source": "nvml" if self._nvml else "nvidia-smi"}


def sources_hash(paths):
    h = hashlib.sha256()
    for p in paths:
        with open(os.path.join(ROOT, p), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def profiled_traffic(kernel_tag: str, workload: str):
    """DRAM bytes per launch from the committed ncu summary, if it was taken
    on the current sources of the captured kernel (the entry's own source
    list: the static-chunk and the claimed-group kernels differ); else None."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            entry = json.load(f)[kernel_tag][workload]
        sources = entry.get("sources", HT_KERNEL_SOURCES)
        if entry.get("sources_sha256_16") != sources_hash(sources):
            return None
    except Exception:
        return None
    return entry.get("dram_bytes_per_launch")


# ------------------------------------------------------------ our arm
def percentiles(xs):
    """[p10, p50, p90] of a list, rounded."""
    xs = sorted(xs)
    pick = lambda q: xs[min(len(xs) - 1, int(q * (len(xs) - 1) + 0.5))]  # noqa: E731
    return [round(pick(0.1), 2), round(pick(0.5), 2), round(pick(0.9), 2)]


def ht_bytes(d, count, g_bytes=4):
    return (g_bytes + 8) * d + 8 * count


def run_ours(args):
    import torch
    import paper_2108_00951_gb300 as efs
    from paper_2108_00951_gb300 import workloads

    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    dist = dist_init("nccl")
    efs.load_library()

    w = workloads.BY_NAME[args.workload]
    d, n, gamma = w.d, w.n, w.gamma
    ks = w.topk_values()
    k = ks[min(args.lam_index, len(ks) - 1)]
    frac = k / d if not w.topk_fracs else w.topk_fracs[min(args.lam_index, len(w.topk_fracs) - 1)]
    seg_end = workloads.segment_ends(w)
    seg_k = workloads.layerwise_k(w, frac)
    k_lw = sum(seg_k)
    wr = replica_workload(w, rank)
    batches = [[workloads.gradient(wr, i, b, device=dev) for i in range(n)] for b in range(2)]
    lam = (workloads.density_lambda(wr, batches[0][0], w.density) if w.density is not None
           else w.lambdas[args.lam_index])

    def outputs(cap):
        return ([torch.empty(cap, dtype=torch.int32, device=dev) for _ in range(n)],
                [torch.empty(cap, dtype=torch.float32, device=dev) for _ in range(n)])

    e_ht = [torch.zeros(d, device=dev) for _ in range(n)]
    e_tk = [torch.zeros(d, device=dev) for _ in range(n)]
    e_lw = [torch.zeros(d, device=dev) for _ in range(n)]
    idx_ht, val_ht = outputs(d)
    # the hard-threshold messages' tile indexes, written by the compress calls
    # and read by the aggregations of those messages
    tiles_ht = [torch.empty(efs.tiles_for(d), dtype=torch.int32, device=dev) for _ in range(n)]
    idx_tk, val_tk = outputs(k)
    idx_lw, val_lw = outputs(k_lw)
    dense_ht = torch.empty(d, device=dev)
    dense_tk = torch.empty(d, device=dev)
    dense_lw = torch.empty(d, device=dev)
    x_model = torch.zeros(d, device=dev)
    m_model = torch.zeros(d, device=dev)
    e_rd = [torch.zeros(d, device=dev) for _ in range(n)]
    # the bf16-gradient variant: the same gradients rounded to bfloat16
    batches_bf = [[g.to(torch.bfloat16) for g in b] for b in batches]
    e_bf = [torch.zeros(d, device=dev) for _ in range(n)]
    idx_bf, val_bf = outputs(d)
    q_rd = [torch.empty(d, dtype=torch.int32, device=dev) for _ in range(n)]
    unsent_rd = torch.zeros(n, dtype=torch.int32, device=dev)
    dense_rd = torch.empty(d, device=dev)
    scale_log2 = 20  # grid 2^-20 for the rounding compressor
    total = args.warmup + args.steps
    cnt_ht = torch.zeros(total, n, dtype=torch.int32, device=dev)
    cnt_tk = torch.zeros(total, n, dtype=torch.int32, device=dev)
    cnt_lw = torch.zeros(total, n, dtype=torch.int32, device=dev)
    cnt_bf = torch.zeros(total, n, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream()

    ev = lambda: torch.cuda.Event(enable_timing=True)  # noqa: E731
    marks = [[ev() for _ in range(11)] for _ in range(args.steps)]

    err_sq = torch.zeros(3, n, dtype=torch.float64, device=dev)

    def errkw(leg, i):
        return {"err_sq_out": err_sq[leg, i:i + 1]} if args.error_norm else {}

    def step(s, timed):
        g = batches[s % 2]
        m = marks[s - args.warmup] if timed else None
        if m: m[0].record(stream)
        for i in range(n):
            efs.ef_hard_threshold(g[i], e_ht[i], gamma, lam, idx_ht[i], val_ht[i],
                                  cnt_ht[s, i:i + 1], tiles_out=tiles_ht[i], **errkw(0, i))
        if m: m[1].record(stream)
        efs.sparse_aggregate(idx_ht, val_ht, cnt_ht[s], d, dense_ht, tiles=tiles_ht)
        if m: m[2].record(stream)
        for i in range(n):
            efs.ef_topk(g[i], e_tk[i], gamma, k, idx_tk[i], val_tk[i], cnt_tk[s, i:i + 1],
                        **errkw(1, i))
        if m: m[3].record(stream)
        efs.sparse_aggregate(idx_tk, val_tk, cnt_tk[s], d, dense_tk)
        if m: m[4].record(stream)
        for i in range(n):
            efs.ef_topk_layerwise(g[i], e_lw[i], gamma, seg_end, seg_k, idx_lw[i], val_lw[i],
                                  cnt_lw[s, i:i + 1], **errkw(2, i))
        if m: m[5].record(stream)
        efs.sparse_aggregate(idx_lw, val_lw, cnt_lw[s], d, dense_lw)
        if m: m[6].record(stream)
        efs.sparse_aggregate_apply(idx_ht, val_ht, cnt_ht[s], d, 1.0 / n, x_model, m_model, 0.9,
                                   gamma, tiles=tiles_ht)
        if m: m[7].record(stream)
        for i in range(n):
            efs.ef_scaled_round(g[i], e_rd[i], gamma, scale_log2, q_rd[i], unsent_rd[i:i + 1])
        if m: m[8].record(stream)
        efs.int_aggregate(q_rd, d, scale_log2, dense_rd)
        if m: m[9].record(stream)
        gb = batches_bf[s % 2]
        for i in range(n):
            efs.ef_hard_threshold(gb[i], e_bf[i], gamma, lam, idx_bf[i], val_bf[i],
                                  cnt_bf[s, i:i + 1])
        if m: m[10].record(stream)

    for s in range(args.warmup):
        step(s, False)
    torch.cuda.synchronize()
    if efs.ef_check_status() != efs.EF_OK:
        raise RuntimeError("device error during warm-up")

    sampler = ClockSampler(local)
    sampler.start()
    launches0 = efs.ef_kernel_launches()
    barrier(dist, dev)
    torch.cuda.synchronize()
    t0, t1 = ev(), ev()
    t0.record(stream)
    for s in range(args.warmup, total):
        step(s, True)
    t1.record(stream)
    torch.cuda.synchronize()
    barrier(dist, dev)
    launches = efs.ef_kernel_launches() - launches0
    clocks = sampler.stop()
    if efs.ef_check_status() != efs.EF_OK:
        raise RuntimeError("device error during the timed steps")

    step_s = t0.elapsed_time(t1) / 1e3
    # per-iteration segment times (µs per call: the segment of n calls / n)
    seg_us = [[m[a].elapsed_time(m[a + 1]) * 1e3 for m in marks] for a in range(10)]
    ht_s = sum(m[0].elapsed_time(m[1]) for m in marks) / 1e3
    agg_ht_s = sum(m[1].elapsed_time(m[2]) for m in marks) / 1e3
    tk_s = sum(m[2].elapsed_time(m[3]) for m in marks) / 1e3
    agg_tk_s = sum(m[3].elapsed_time(m[4]) for m in marks) / 1e3
    lw_s = sum(m[4].elapsed_time(m[5]) for m in marks) / 1e3
    agg_lw_s = sum(m[5].elapsed_time(m[6]) for m in marks) / 1e3
    upd_s = sum(m[6].elapsed_time(m[7]) for m in marks) / 1e3
    rd_s = sum(m[7].elapsed_time(m[8]) for m in marks) / 1e3
    iagg_s = sum(m[8].elapsed_time(m[9]) for m in marks) / 1e3
    bf_s = sum(m[9].elapsed_time(m[10]) for m in marks) / 1e3
    counts_bf = cnt_bf[args.warmup:].double()
    bytes_bf = float(ht_bytes(d, 0, 2) * n * args.steps + 8 * counts_bf.sum().item())
    counts_ht = cnt_ht[args.warmup:].double()
    counts_tk = cnt_tk[args.warmup:].double()
    bytes_ht = float(ht_bytes(d, 0) * n * args.steps + 8 * counts_ht.sum().item())
    bytes_tk = float((12 * d + 8 * k) * n * args.steps)
    bytes_lw = float((12 * d + 8 * k_lw) * n * args.steps)
    bytes_agg_ht = float(8 * counts_ht.sum().item() + 4 * d * args.steps)
    bytes_agg_tk = float(8 * counts_tk.sum().item() + 4 * d * args.steps)
    bytes_upd = float(8 * counts_ht.sum().item() + 16 * d * args.steps)
    bytes_rd = float(16 * d * n * args.steps)
    bytes_iagg = float((4 * n + 4) * d * args.steps)

    ht_s_max, bytes_ht_all = reduce_timing(dist, ht_s, bytes_ht, dev)
    step_s_max, _ = reduce_timing(dist, step_s, 0.0, dev)
    value = bytes_ht_all / ht_s_max / 1e9
    peak, peak_kind = measured_peak_gbs()
    # the n compress calls of a step run back to back on the stream (one
    # kernel launch each), so the segment time / n is the average launch
    # duration including the gaps between launches
    avg_launch = ht_s / (n * args.steps)
    achieved = (ht_bytes(d, 0) + 8 * counts_ht.mean().item()) / avg_launch / 1e9

    # free the main legs' buffers before the extra legs allocate theirs
    del batches, batches_bf, e_ht, e_tk, e_lw, e_rd, e_bf, idx_ht, val_ht, idx_tk, val_tk
    del idx_lw, val_lw, idx_bf, val_bf, q_rd, dense_tk, dense_lw, dense_rd, x_model, m_model
    torch.cuda.empty_cache()
    extra = None
    if not args.no_extra_legs:
        extra = extra_legs(args, efs, torch, dev, dist, rank, w, peak)

    e2e = None
    if not args.no_e2e:
        grads0 = [workloads.gradient(wr, i, 0, device=dev) for i in range(n)]
        e2e = run_e2e(args, efs, torch, dev, dist, grads0, d, n, gamma, lam, stream)
        del grads0

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(args, [workloads.gradient(wr, i, 0, device=dev).cpu().numpy()
                                  for i in range(2)], d, gamma, lam, k)

    if rank != 0:
        return None
    density = counts_ht.mean().item() / d
    return {
        "metric": METRIC,
        "value": round(value, 2),
        "unit": "GB/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(step_s_max / args.steps * 1e3, 4),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "f32",
        "data": "synthetic (seeded %s-shaped gradients; no dataset or trained model)" % w.name,
        "config": {
            "workload": "%s: d=%d in %d segments, n=%d simulated workers, gamma=%g, "
                        "hard-threshold lambda=%.6g (first-iteration density %.4g%%), "
                        "Top-k k=%d" % (w.name, d, len(w.segments), n, gamma, lam,
                                        100 * (w.density or 0), k),
            "global_batch": n,
            "seq_len": None,
            "parallelism": "replicas x%d (simulated workers on each GPU)" % world,
            "l2": "inputs larger than L2: %.2f GB touched per step vs 126 MB L2"
                  % (n * 12 * d / 1e9),
            "value_scope": "n hard-threshold compress calls per step, device time",
        },
        "elem_per_s": round(n * d * args.steps * world / ht_s_max, 1),
        "ht_density": round(density, 6),
        "ht_ms_per_iter": round(ht_s / args.steps * 1e3, 4),
        "topk_ms_per_iter": round(tk_s / args.steps * 1e3, 4),
        "topk_gbs": round(bytes_tk / tk_s / 1e9, 2),
        "topk_frac_of_peak": round(bytes_tk / tk_s / 1e9 / peak, 4),
        "aggregate_ms_per_iter": round(agg_ht_s / args.steps * 1e3, 4),
        "aggregate_tile_index": "hard-threshold messages: from the compress calls; Top-k: searched",
        "aggregate_gbs": round(bytes_agg_ht / agg_ht_s / 1e9, 2),
        "aggregate_frac_of_peak": round(bytes_agg_ht / agg_ht_s / 1e9 / peak, 4),
        "aggregate_topk_ms_per_iter": round(agg_tk_s / args.steps * 1e3, 4),
        "topk_layerwise": {
            "segments": len(seg_end),
            "k_total": k_lw,
            "k_rule": "k_s = max(1, floor(%g d_s))" % frac,
            "ms_per_iter": round(lw_s / args.steps * 1e3, 4),
            "gbs": round(bytes_lw / lw_s / 1e9, 2),
            "frac_of_peak": round(bytes_lw / lw_s / 1e9 / peak, 4),
            "aggregate_ms_per_iter": round(agg_lw_s / args.steps * 1e3, 4),
        },
        "aggregate_apply_momentum": {
            "ms_per_iter": round(upd_s / args.steps * 1e3, 4),
            "gbs": round(bytes_upd / upd_s / 1e9, 2),
            "frac_of_peak": round(bytes_upd / upd_s / 1e9 / peak, 4),
            "bytes": "8 per hard-threshold pair + 16 per coordinate (x, m read and written)",
            "tile_index": "the messages' tile indexes written by the compress calls",
        },
        "scaled_round": {
            "scale_log2": scale_log2,
            "ms_per_iter": round(rd_s / args.steps * 1e3, 4),
            "gbs": round(bytes_rd / rd_s / 1e9, 2),
            "frac_of_peak": round(bytes_rd / rd_s / 1e9 / peak, 4),
            "int_aggregate_ms_per_iter": round(iagg_s / args.steps * 1e3, 4),
            "int_aggregate_gbs": round(bytes_iagg / iagg_s / 1e9, 2),
            "int_aggregate_frac_of_peak": round(bytes_iagg / iagg_s / 1e9 / peak, 4),
            "bytes": "compress 16 per coordinate; exchange 4 n + 4 per coordinate",
        },
        "ht_bf16": {
            "ms_per_iter": round(bf_s / args.steps * 1e3, 4),
            "gbs": round(bytes_bf / bf_s / 1e9, 2),
            "frac_of_peak": round(bytes_bf / bf_s / 1e9 / peak, 4),
            "density": round(counts_bf.mean().item() / d, 6),
            "bytes": "10 per coordinate (bf16 g, fp32 e read and written) + 8 per sent pair",
        },
        "per_call_us_p10_p50_p90": {
            "ht": percentiles([v / n for v in seg_us[0]]),
            "topk": percentiles([v / n for v in seg_us[2]]),
            "topk_layerwise": percentiles([v / n for v in seg_us[4]]),
            "aggregate_ht": percentiles(seg_us[1]),
            "aggregate_topk": percentiles(seg_us[3]),
            "aggregate_topk_layerwise": percentiles(seg_us[5]),
            "aggregate_apply_momentum": percentiles(seg_us[6]),
            "scaled_round": percentiles([v / n for v in seg_us[7]]),
            "int_aggregate": percentiles(seg_us[8]),
            "ht_bf16": percentiles([v / n for v in seg_us[9]]),
        },
        "frac_of_nominal_8tbs": round(value / NOMINAL_HBM_GBS, 4),
        "roofline": {
            "bound": "hbm",
            "kernel": (("lookback_stream_kernel<HtOp> (claimed tile groups, decoupled look-back)"
                        if (d + 4095) // 4096 >= 4096 else
                        "stream_compact_kernel<HtOp> (static chunks)") +
                       ": fused EF accumulate + hard-threshold + compaction + residual"),
            "achieved": round(achieved, 2),
            "peak": peak,
            "peak_kind": peak_kind,
            "unit": "GB/s",
            "frac": round(achieved / peak, 4),
            "avg_launch_us": round(avg_launch * 1e6, 3),
            "algorithmic_bytes_per_launch": int(ht_bytes(d, 0) + 8 * counts_ht.mean().item()),
            "traffic": profiled_traffic("ht_kernel", w.name),
        },
        "error_norm": ({"requested": True,
                        "last_step_sq_norms_worker0": {
                            "ht": float(err_sq[0, 0]), "topk": float(err_sq[1, 0]),
                            "topk_layerwise": float(err_sq[2, 0])}}
                       if args.error_norm else {"requested": False}),
        "extra_legs": extra,
        "gpu_launches": int(launches),
        "clocks": clocks,
        "e2e": e2e,
        "cpu_baseline": cpu,
    }


def compress_leg(efs, torch, dev, dist, w, method, param, steps, warmup, peak, flush=None):
    """Time an EF loop of workload w's n workers through one compress method
    ("ht": param = lambda; "topk": param = k): `warmup` untimed iterations,
    then `steps` timed ones (CUDA events around each iteration's n calls on
    the launching stream). With `flush` (a device buffer larger than L2) the
    buffer is rewritten before every call and each call is timed alone: the
    cold-L2 variant."""
    n, d = w.n, w.d
    batches = [[workloads_gradient(w, i, b, dev) for i in range(n)] for b in range(2)]
    e = [torch.zeros(d, device=dev) for _ in range(n)]
    cap = d if method == "ht" else param
    idx = [torch.empty(cap, dtype=torch.int32, device=dev) for _ in range(n)]
    val = [torch.empty(cap, dtype=torch.float32, device=dev) for _ in range(n)]
    cnt = torch.zeros(warmup + steps, n, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream()
    ev = lambda: torch.cuda.Event(enable_timing=True)  # noqa: E731
    per = n if flush is not None else 1
    marks = [[(ev(), ev()) for _ in range(per)] for _ in range(steps)]

    def call(s, i):
        g = batches[s % 2][i]
        if method == "ht":
            efs.ef_hard_threshold(g, e[i], w.gamma, param, idx[i], val[i], cnt[s, i:i + 1])
        else:
            efs.ef_topk(g, e[i], w.gamma, param, idx[i], val[i], cnt[s, i:i + 1])

    for s in range(warmup + steps):
        m = marks[s - warmup] if s >= warmup else None
        if flush is None:
            if m: m[0][0].record(stream)
            for i in range(n):
                call(s, i)
            if m: m[0][1].record(stream)
        else:
            for i in range(n):
                flush.add_(1.0)
                if m: m[i][0].record(stream)
                call(s, i)
                if m: m[i][1].record(stream)
    torch.cuda.synchronize()
    if efs.ef_check_status() != efs.EF_OK:
        raise RuntimeError("device error in the %s leg of %s" % (method, w.name))
    secs = sum(a.elapsed_time(b) for m in marks for a, b in m) / 1e3
    calls_us = ([a.elapsed_time(b) * 1e3 / n for m in marks for a, b in m] if flush is None else
                [a.elapsed_time(b) * 1e3 for m in marks for a, b in m])
    counts = cnt[warmup:].double()
    byts = float(12 * d * n * steps + 8 * counts.sum().item())
    secs_max, byts_all = reduce_timing(dist, secs, byts, dev)
    gbs = byts_all / secs_max / 1e9 if dist is None else byts / secs / 1e9
    return {"workload": w.name, "d": d, "n": n,
            ("lambda" if method == "ht" else "k"): param,
            "density": round(counts.mean().item() / d, 6),
            "us_per_call_p10_p50_p90": percentiles(calls_us),
            "gbs": round(gbs, 2), "frac_of_peak": round(gbs / peak, 4),
            "iterations": steps, "warmup": warmup}


def workloads_gradient(w, i, t, dev):
    from paper_2108_00951_gb300 import workloads
    return workloads.gradient(w, i, t, device=dev)


def extra_legs(args, efs, torch, dev, dist, rank, w_main, peak):
    """The rest of the d >= 25 M regime (LSTM-shaped at its threshold and
    Top-k fraction, ResNet-50-shaped at each threshold and Top-k fraction),
    the cold-L2 variant of the headline call, and the latency of the
    L2-resident logistic-regression-sized case."""
    from paper_2108_00951_gb300 import workloads
    steps, warmup = max(3, min(args.steps, 20)), max(3, args.warmup)
    out = {"regime_d_ge_25M": [], "bytes": "12 per coordinate + 8 per sent pair"}
    for name in ("lstm", "resnet50"):
        if name == w_main.name:
            continue
        w = replica_workload(workloads.BY_NAME[name], rank)
        if w.density is not None:
            lams = [workloads.density_lambda(w, workloads_gradient(w, 0, 0, dev), w.density)]
        else:
            lams = list(w.lambdas)
        for lam in lams:
            out["regime_d_ge_25M"].append(
                {"method": "hard_threshold",
                 **compress_leg(efs, torch, dev, dist, w, "ht", lam, steps, warmup, peak)})
            torch.cuda.empty_cache()
        for k in w.topk_values():
            out["regime_d_ge_25M"].append(
                {"method": "topk",
                 **compress_leg(efs, torch, dev, dist, w, "topk", k, steps, warmup, peak)})
            torch.cuda.empty_cache()
    # cold L2: a 512 MB buffer (4x the L2) rewritten before every call
    flush = torch.zeros(128 << 20, device=dev)
    w = replica_workload(w_main, rank)
    lam = (workloads.density_lambda(w, workloads_gradient(w, 0, 0, dev), w.density)
           if w.density is not None else w.lambdas[args.lam_index])
    out["cold_l2_ht"] = compress_leg(efs, torch, dev, dist, w, "ht", lam, 3, warmup, peak,
                                     flush=flush)
    del flush
    torch.cuda.empty_cache()
    # latency of the L2-resident case (d = 100,000, 4 workers)
    w = replica_workload(workloads.BY_NAME["lr"], rank)
    lat = {}
    for method, param in (("ht", w.lambdas[0]), ("topk", w.topk_k[0])):
        r = compress_leg(efs, torch, dev, dist, w, method, param, 50, warmup, peak)
        lat[method + "_us_per_call_p10_p50_p90"] = r["us_per_call_p10_p50_p90"]
    out["latency_lr"] = {"d": w.d, "n": w.n, **lat,
                         "note": "the working set fits in L2: reported as latency"}
    return out


def run_harness(args):
    """One kind of call on one worker of the workload (a few GB on the
    device), for profiler captures: `--warmup` then `--steps` calls on
    alternating gradients; the aggregate harness compresses the n workers'
    gradients once (hard-threshold) and aggregates their messages."""
    import torch
    import paper_2108_00951_gb300 as efs
    from paper_2108_00951_gb300 import workloads

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    efs.load_library()
    w = workloads.BY_NAME[args.workload]
    d = w.d
    lam = (workloads.density_lambda(w, workloads_gradient(w, 0, 0, dev), w.density)
           if w.density is not None else w.lambdas[args.lam_index])
    ks = w.topk_values()
    k = ks[min(args.lam_index, len(ks) - 1)]
    e = torch.zeros(d, device=dev)
    cnt = torch.zeros(1, dtype=torch.int32, device=dev)
    ev = lambda: torch.cuda.Event(enable_timing=True)  # noqa: E731
    t0, t1 = ev(), ev()
    if args.harness == "aggregate":
        idx_s = torch.empty(d, dtype=torch.int32, device=dev)
        val_s = torch.empty(d, dtype=torch.float32, device=dev)
        idx, val, tiles, counts = [], [], [], []
        # each worker's message after `warmup` EF iterations (the density
        # grows from the first iteration's to the loop's steady state)
        for i in range(w.n):
            e.zero_()
            tl = torch.empty(efs.tiles_for(d), dtype=torch.int32, device=dev)
            for t in range(max(1, args.warmup)):
                efs.ef_hard_threshold(workloads_gradient(w, i, t % 2, dev), e, w.gamma, lam,
                                      idx_s, val_s, cnt, tiles_out=tl)
            c = int(cnt.item())
            idx.append(idx_s[:max(c, 1)].clone())
            val.append(val_s[:max(c, 1)].clone())
            tiles.append(tl)
            counts.append(c)
        del idx_s, val_s
        cnt_n = torch.tensor(counts, dtype=torch.int32, device=dev)
        dense = torch.empty(d, device=dev)
        for s in range(3 + args.steps):
            if s == 3:
                t0.record()
            efs.sparse_aggregate(idx, val, cnt_n, d, dense, tiles=tiles)
        t1.record()
        torch.cuda.synchronize()
        per = t0.elapsed_time(t1) * 1e3 / max(args.steps, 1)
        byts = 8 * sum(counts) + 4 * d
    else:
        dtype = torch.bfloat16 if args.harness == "ht_bf16" else torch.float32
        grads = [workloads.gradient(w, 0, t, device=dev, dtype=dtype) for t in range(2)]
        cap = k if args.harness == "topk" else d
        if args.harness == "topk_layerwise":
            frac = w.topk_fracs[min(args.lam_index, len(w.topk_fracs) - 1)] if w.topk_fracs \
                else k / d
            seg_end, seg_k = workloads.segment_ends(w), workloads.layerwise_k(w, frac)
            cap = sum(seg_k)
        idx = torch.empty(cap, dtype=torch.int32, device=dev)
        val = torch.empty(cap, dtype=torch.float32, device=dev)
        for s in range(args.warmup + args.steps):
            if s == args.warmup:
                t0.record()
            g = grads[s % 2]
            if args.harness in ("ht", "ht_bf16"):
                efs.ef_hard_threshold(g, e, w.gamma, lam, idx, val, cnt)
            elif args.harness == "topk":
                efs.ef_topk(g, e, w.gamma, k, idx, val, cnt)
            else:
                efs.ef_topk_layerwise(g, e, w.gamma, seg_end, seg_k, idx, val, cnt)
        t1.record()
        torch.cuda.synchronize()
        per = t0.elapsed_time(t1) * 1e3 / max(args.steps, 1)
        gb = 2 if args.harness == "ht_bf16" else 4
        byts = (gb + 8) * d + 8 * int(cnt.item())
    if efs.ef_check_status() != efs.EF_OK:
        raise RuntimeError("device error in the harness")
    return {"harness": args.harness, "workload": w.name, "d": d, "steps": args.steps,
            "warmup": args.warmup, "us_per_call": round(per, 2),
            "last_call_algorithmic_bytes": int(byts),
            "note": "one worker's calls back to back: a harness for profiler captures, "
                    "not a bench value"}


def run_e2e(args, efs, torch, dev, dist, grads, d, n, gamma, lam, stream):
    """The hard-threshold iteration through the public API with host data:
    per step, H2D of the n gradients from pinned memory, n compress calls,
    the aggregate, and D2H of the dense result. Pipelined as a user would:
    the uploads run on their own stream into two alternating sets of device
    buffers (worker i's compress waits only for its own upload), and the
    dense result's download runs on a third stream, overlapping the next
    step's uploads. Events order every reuse of a buffer."""
    host_g = [g.cpu().pin_memory() for g in grads]
    host_out = [torch.empty(d, dtype=torch.float32).pin_memory() for _ in range(2)]
    dev_g = [[torch.empty(d, device=dev) for _ in range(n)] for _ in range(2)]
    e = [torch.zeros(d, device=dev) for _ in range(n)]
    idx = [torch.empty(d, dtype=torch.int32, device=dev) for _ in range(n)]
    val = [torch.empty(d, dtype=torch.float32, device=dev) for _ in range(n)]
    tiles = [torch.empty(efs.tiles_for(d), dtype=torch.int32, device=dev) for _ in range(n)]
    cnt = torch.zeros(args.steps + args.warmup, n, dtype=torch.int32, device=dev)
    dense = [torch.empty(d, device=dev) for _ in range(2)]
    up, down = torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)
    ev = lambda: torch.cuda.Event()  # noqa: E731
    uploaded = [[ev() for _ in range(n)] for _ in range(2)]   # dev_g[b][i] filled
    consumed = [[ev() for _ in range(n)] for _ in range(2)]   # dev_g[b][i] read
    reduced = [ev() for _ in range(2)]                         # dense[b] written
    fetched = [ev() for _ in range(2)]                         # dense[b] read back
    for b in range(2):  # every buffer starts free
        for i in range(n):
            consumed[b][i].record(stream)
        fetched[b].record(stream)

    def step(s):
        b = s % 2
        with torch.cuda.stream(up):
            for i in range(n):
                up.wait_event(consumed[b][i])
                dev_g[b][i].copy_(host_g[i], non_blocking=True)
                uploaded[b][i].record(up)
        for i in range(n):
            stream.wait_event(uploaded[b][i])
            efs.ef_hard_threshold(dev_g[b][i], e[i], gamma, lam, idx[i], val[i],
                                  cnt[s, i:i + 1], stream=stream, tiles_out=tiles[i])
            consumed[b][i].record(stream)
        stream.wait_event(fetched[b])
        efs.sparse_aggregate(idx, val, cnt[s], d, dense[b], stream=stream, tiles=tiles)
        reduced[b].record(stream)
        with torch.cuda.stream(down):
            down.wait_event(reduced[b])
            host_out[b].copy_(dense[b], non_blocking=True)
            fetched[b].record(down)

    for s in range(args.warmup):
        step(s)
    torch.cuda.synchronize()
    barrier(dist, dev)
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    up.wait_event(t0)  # the first upload starts after t0
    for s in range(args.warmup, args.warmup + args.steps):
        step(s)
    stream.wait_event(fetched[(args.warmup + args.steps - 1) % 2])  # the last read-back
    t1.record(stream)
    torch.cuda.synchronize()
    barrier(dist, dev)
    secs = t0.elapsed_time(t1) / 1e3
    byts = float(12 * d * n * args.steps + 8 * cnt[args.warmup:].double().sum().item())
    secs, byts = reduce_timing(dist, secs, byts, dev)
    return {"value": round(byts / secs / 1e9, 2), "unit": "GB/s",
            "h2d_bytes_per_step": 4 * d * n, "d2h_bytes_per_step": 4 * d,
            "ms_per_step": round(secs / args.steps * 1e3, 4),
            "pipeline": "uploads, compute and download on three streams, double-buffered"}


# ------------------------------------------------------------ CPU oracle legs
def cpu_model() -> str:
    """The host CPU's model name (lscpu, else /proc/cpuinfo)."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.strip().startswith("Model name:"):
                return line.split(":", 1)[1].strip()
    except Exception:
        pass
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                if line.lower().startswith(("model name", "cpu model")):
                    return line.split(":", 1)[1].strip()
    except Exception:
        pass
    import platform
    return platform.processor() or platform.machine()


def cpu_baseline(args, grads, d, gamma, lam, k):
    """The oracle as it stands, single-threaded on this host: hard-threshold
    calls on the first workers' full-size gradients for about
    args.cpu_seconds, in the same unit as the headline."""
    import numpy as np
    import oracle
    e = np.zeros(d, np.float32)
    calls, byts, t_start = 0, 0.0, time.perf_counter()
    while True:
        idx, _, e = oracle.ef_hard_threshold(grads[calls % len(grads)], e, gamma, lam)
        calls += 1
        byts += ht_bytes(d, idx.size)
        el = time.perf_counter() - t_start
        if el >= args.cpu_seconds:
            break
    return {"value": round(byts / el / 1e9, 4), "unit": "GB/s", "cores": 1, "kind": "oracle",
            "sample": "%d single-threaded oracle hard-threshold calls at full d=%d (%.1f s)"
                      % (calls, d, el),
            "host_cores_available": os.cpu_count(), "cpu_model": cpu_model()}


def run_reference(args):
    """The reference arm: the CPU oracle (there is no reference code for this
    paper) on this host, timed over the same workload, metric and unit; each
    step is one full-size hard-threshold call of one simulated worker."""
    import numpy as np
    import torch
    import oracle
    from paper_2108_00951_gb300 import workloads

    rank, world, _ = dist_env()
    if rank != 0:
        return None
    w = workloads.BY_NAME[args.workload]
    grads = [workloads.gradient(w, i, 0).numpy() for i in range(2)]
    lam = (workloads.density_lambda(w, torch.from_numpy(grads[0]), w.density)
           if w.density is not None else w.lambdas[0])
    e = np.zeros(w.d, np.float32)
    for s in range(args.warmup):
        _, _, e = oracle.ef_hard_threshold(grads[s % 2], e, w.gamma, lam)
    byts, t0 = 0.0, time.perf_counter()
    for s in range(args.steps):
        idx, _, e = oracle.ef_hard_threshold(grads[s % 2], e, w.gamma, lam)
        byts += ht_bytes(w.d, idx.size)
    el = time.perf_counter() - t0
    value = byts / el / 1e9
    return {
        "impl": "reference",
        "metric": METRIC,
        "value": round(value, 4),
        "unit": "GB/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(el / args.steps * 1e3, 3),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "f32",
        "data": "synthetic (seeded %s-shaped gradients)" % w.name,
        "config": {"workload": "%s: d=%d, one simulated worker's hard-threshold call per step"
                               % (w.name, w.d), "global_batch": 1, "seq_len": None,
                   "parallelism": "single CPU thread"},
        "cpu_baseline": {"value": round(value, 4), "unit": "GB/s", "cores": 1, "kind": "oracle",
                         "sample": "%d full-size oracle hard-threshold calls" % args.steps,
                         "cpu_model": cpu_model()},
        "e2e": {"value": round(value, 4), "unit": "GB/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }


def main(argv=None):
    args = parse_args(argv)
    if args.impl == "reference":
        out = run_reference(args)
    elif args.harness:
        out = run_harness(args)
    else:
        out = run_ours(args)
    if out is not None:
        print(json.dumps(out), flush=True)
    try:
        import torch.distributed as dist
        if dist.is_initialized():
            dist.destroy_process_group()
    except Exception:
        pass
    return 0


if __name__ == "__main__":
    sys.exit(main())
