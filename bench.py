#!/usr/bin/env python
"""Throughput of the adapter fine-tuning step (forward, loss, early-stopped backward, Adam)
on the BERT-large-shaped workload, versus the unfreezing depth d (k = L - d).

One "step" is ra_forward + ra_backward_truncated(k) + ra_adapter_update over one batch of
32 x 256 synthetic tokens (24 layers, H 1024, 16 heads, FFN 4096, adapters m 64), replayed
from a CUDA graph; inputs are resident in HBM when the timed region starts.  The headline
is samples/s at d = 12 (a frozen prefix of 12 blocks plus a 12-block backward); the sweep
over d = 1, 6, 12, 24 is in "sweep", and the BERT-base-shaped sweep (d = 1, 3, 6, 12) in
"base".  A step streams several GB, far above the 129 MB L2, so no flush is needed
between steps.

  python bench.py [--gpus N --steps K --warmup W]      # the CUDA path (one JSON line)
  python bench.py --impl reference ...                 # the fp64 oracle on the host cores

Under torchrun (N > 1) every rank runs an independent replica (the step does not shard:
"replicas only"); value = all ranks' samples / the slowest rank's time.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "fine-tune samples/sec vs unfrozen depth k"
UNIT = "samples/s"
DEFAULT_CONFIG = "large"
# workloads (--config): depth sweep and headline depth of each
SWEEPS = {"base": ([1, 3, 6, 12], 6), "large": ([1, 6, 12, 24], 12), "llama": ([4], 4),
          "tiny": ([1, 2], 1)}
HEADLINE_D = 12
SWEEP = [1, 6, 12, 24]
# sequences per oracle step in the bounded CPU sample of each workload
CPU_SAMPLE_BATCH = {"base": 2, "large": 1, "llama": 1, "tiny": 4}


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", default=DEFAULT_CONFIG)
    ap.add_argument("--no-extra", action="store_true", help="skip the BERT-base sweep")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--schedule", action="store_true",
                    help="run the 600-step top-down unfreezing schedule on the BERT-base workload")
    ap.add_argument("--cpu-worker", default=None, help=argparse.SUPPRESS)
    return ap.parse_args()


# ---------------------------------------------------------------------------------------
# oracle legs (host cores)
# ---------------------------------------------------------------------------------------

def oracle_sample_rate(cfg_name, depth, batch, min_seconds, steps=None):
    """fp64 oracle steps (forward, loss, early-stopped backward, Adam) on `batch` sequences
    of the workload; returns (samples/s, steps run, seconds)."""
    import dataclasses
    import synth
    from oracle import ringada_oracle as O
    cfg = dataclasses.replace(synth.CONFIGS[cfg_name], batch=batch)
    w = synth.make_workload(cfg, 0)
    layers, head = O.to_f64_params(w["layers"], w["head"])
    opt = O.Adam(lr=1e-4)
    n, t0 = 0, time.perf_counter()
    while True:
        r = O.step(cfg, layers, head, w["x"], w["labels"], depth)
        O.apply_update(cfg, layers, head, r, opt)
        n += 1
        el = time.perf_counter() - t0
        if (steps is not None and n >= steps) or (steps is None and el >= min_seconds):
            break
    return batch * n / el, n, el


def cpu_worker(spec):
    cfg_name, depth, batch, secs = spec.split(",")
    rate, n, el = oracle_sample_rate(cfg_name, int(depth), int(batch), float(secs))
    print(json.dumps(dict(rate=rate, steps=n, seconds=el)))


def run_cpu_baseline(cfg_name, depth, batch, seconds):
    cores = os.cpu_count() or 1
    env = dict(os.environ, OMP_NUM_THREADS=str(cores), OPENBLAS_NUM_THREADS=str(cores),
               MKL_NUM_THREADS=str(cores), CUDA_VISIBLE_DEVICES="")
    spec = "%s,%d,%d,%g" % (cfg_name, depth, batch, seconds)
    r = subprocess.run([sys.executable, os.path.abspath(__file__), "--cpu-worker", spec],
                       capture_output=True, text=True, env=env, timeout=900)
    if r.returncode != 0:
        return {"value": None, "unit": UNIT, "cores": cores, "kind": "oracle",
                "sample": "failed: " + r.stderr.strip()[-300:]}
    res = json.loads(r.stdout.strip().splitlines()[-1])
    return {"value": res["rate"], "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": "%d oracle steps (fp64 numpy, BLAS on %d threads) of %s at d=%d on %d of "
                      "the batch's sequences, %.1f s" % (res["steps"], cores, cfg_name, depth, batch,
                                                        res["seconds"])}


def workload_config(name, depth, world=1):
    """The `config` object of the JSON line: the same for the CUDA arm and the reference arm."""
    import synth
    cfg = synth.CONFIGS[name]
    return {"workload": "%s-shaped adapter step (%d layers, H %d, %d heads, FFN %d, adapters "
                        "m %d, batch %d x %d), d=%d" % (name, cfg.n_layers, cfg.hidden, cfg.n_heads,
                                                         cfg.ffn, cfg.adapter_dim, cfg.batch,
                                                         cfg.seq, depth),
            "global_batch": cfg.batch * world, "seq_len": cfg.seq, "depth": depth,
            "parallelism": "replicas" if world > 1 else "single",
            "l2": "inputs larger than L2 (several GB streamed per step)"}


def reference_main(args):
    _, rank, _ = rank_env()
    if rank != 0:
        return 0
    global SWEEP, HEADLINE_D
    SWEEP, HEADLINE_D = SWEEPS[args.config]
    import synth
    cfg = synth.CONFIGS[args.config]
    cores = os.cpu_count() or 1
    # warm-up and timed oracle steps, each a bounded sample (one sequence of the batch)
    oracle_sample_rate(args.config, HEADLINE_D, 1, 0, steps=max(1, min(args.warmup, 2)))
    rate, n, el = oracle_sample_rate(args.config, HEADLINE_D, 1, 0, steps=args.steps)
    line = {
        "impl": "reference", "metric": METRIC, "value": rate, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000 * el / n,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic",
        "config": workload_config(args.config, HEADLINE_D, args.gpus),
        "cpu_baseline": {"value": rate, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": "%d fp64 oracle steps, each on 1 of the %d sequences of %d "
                                   "tokens (samples/s = sequences per second)" % (n, cfg.batch, cfg.seq)},
        "e2e": {"value": rate, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))
    return 0


# ---------------------------------------------------------------------------------------
# GPU leg
# ---------------------------------------------------------------------------------------

CLOCK_FIELDS = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
                "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
                "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")


def start_clock_sampler(index):
    """nvidia-smi sampling every 50 ms for the whole GPU-timed part of the run; the samples
    carry timestamps so each timed region gets its own record (clock_record)."""
    path = tempfile.mktemp(prefix="clocks_", suffix=".csv")
    try:
        f = open(path, "w")
        p = subprocess.Popen(["nvidia-smi", "-i", str(index), "--query-gpu=" + CLOCK_FIELDS,
                              "--format=csv,noheader,nounits", "-lms", "50"], stdout=f,
                             stderr=subprocess.DEVNULL)
        return p, f, path
    except Exception:
        return None, None, path


def stop_clock_sampler(h):
    """Stops the sampler; returns the samples as (unix time, sm MHz, max MHz, reasons)."""
    import datetime
    p, f, path = h
    if p is None:
        return None
    p.terminate()
    p.wait(timeout=10)
    f.close()
    names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
    out = []
    for line in open(path):
        parts = [x.strip() for x in line.split(",")]
        if len(parts) < 10:
            continue
        try:
            ts = datetime.datetime.strptime(parts[0], "%Y/%m/%d %H:%M:%S.%f").timestamp()
            sm, smax = float(parts[2]), float(parts[3])
        except ValueError:
            continue
        out.append((ts, sm, smax, {nm for nm, v in zip(names, parts[6:10]) if v.lower() == "active"}))
    os.unlink(path)
    return out


def clock_record(samples, t0=None, t1=None):
    """Median SM clock, max clock and active throttle reasons of the samples in [t0, t1]
    (all samples without a window; the nearest sample when a region is shorter than the
    sampling period)."""
    if samples is None:
        return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
    sel = [s for s in samples if (t0 is None or s[0] >= t0) and (t1 is None or s[0] <= t1)]
    if not sel and samples and t0 is not None:
        mid = 0.5 * (t0 + t1)
        sel = [min(samples, key=lambda s: abs(s[0] - mid))]
    if not sel:
        return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
    reasons = set()
    for s in sel:
        reasons |= s[3]
    return {"sm_mhz": statistics.median(s[1] for s in sel), "sm_max_mhz": max(s[2] for s in sel),
            "reasons": sorted(reasons), "samples": len(sel)}


def measured_peaks():
    try:
        return json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json"))), "measured"
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, "fallback"


def gemm_traffic():
    """DRAM bytes per launch of the tensor-core GEMM from the committed ncu summary, if the
    kernel source has not changed since the capture (else null)."""
    import hashlib
    path = os.path.join(ROOT, "profiles", "gemm_traffic.txt")
    src = os.path.join(ROOT, "paper_2502_19864_gb300", "csrc", "k_gemm_tc.cu")
    try:
        kv = dict(l.split("=", 1) for l in open(path).read().split() if "=" in l)
        h = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
        if kv.get("source_sha") != h:
            return None, "kernel changed since the capture"
        return float(kv["bytes_per_flop"]), kv.get("case", "")
    except Exception:
        return None, "no capture"


class Runner:
    """A model context plus CUDA graphs of one step per depth."""

    def __init__(self, cfg, max_depth, device, prefix_buffers=0):
        import torch
        import synth
        from paper_2502_19864_gb300 import ringada as R
        self.torch, self.R, self.cfg = torch, R, cfg
        w = synth.make_workload(cfg, 0)
        arch = R.RA_ENCODER_POSTLN if cfg.arch == "encoder" else R.RA_DECODER_PRENORM
        self.model = R.Model(R.make_cfg(arch, cfg.n_layers, cfg.hidden, cfg.n_heads, cfg.ffn,
                                        cfg.n_out, cfg.batch, cfg.seq,
                                        R.RA_BF16 if cfg.dtype == "bf16" else R.RA_F32,
                                        int(cfg.head_trainable), max_depth, cfg.norm_eps,
                                        cfg.rope_theta,
                                        R.RA_ADAPTERS_POST_FFN if cfg.adapters == "paper"
                                        else R.RA_ADAPTERS_HOULSBY, prefix_buffers),
                             cfg.adapter_dim, device=device)
        self.model.set_weights(w["layers"], w["head"])
        dt = torch.bfloat16 if cfg.dtype == "bf16" else torch.float32
        self.x = torch.tensor(w["x"], dtype=torch.float32).to(dt).to(device)
        self.labels = torch.tensor(w["labels"], dtype=torch.int32).to(device)
        self.loss = torch.zeros(1, dtype=torch.float32, device=device)
        self.x_host = torch.tensor(w["x"], dtype=torch.float32).to(dt).pin_memory()
        self.labels_host = torch.tensor(w["labels"], dtype=torch.int32).pin_memory()
        self.loss_host = torch.zeros(1, dtype=torch.float32).pin_memory()
        self.graphs = {}       # plain graphs of one step per depth (what is timed)
        self.ograph = {}       # per depth: two graphs of the overlapped step (prefix buffers)
        self.pgraphs = {}      # the same step with a CUDA event around every kernel
        self.launches = {}
        self.saved = {}

    def step(self, d, stream=None):
        R, c = self.R, self.model.ctx
        R.ra_set_unfrozen_depth(c, d)
        R.ra_forward(c, self.x.data_ptr(), self.labels.data_ptr(), self.cfg.batch, self.cfg.seq,
                     self.loss.data_ptr(), None, stream)
        R.ra_backward_truncated(c, self.cfg.n_layers - d, stream)
        R.ra_adapter_update(c, stream=stream)

    def capture(self, d, profile=False):
        torch, R = self.torch, self.R
        n0 = R.ra_kernel_launches()
        self.step(d)                      # eager warm-up (also counts the launches of a step)
        torch.cuda.synchronize()
        self.launches[d] = R.ra_kernel_launches() - n0
        self.saved[d] = self.model.stats()["saved_bytes_in_use"]
        g = torch.cuda.CUDAGraph()
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        R.ra_profile_enable(self.model.ctx, profile)
        with torch.cuda.graph(g, stream=s, capture_error_mode="relaxed"):
            self.step(d, torch.cuda.current_stream())
        R.ra_profile_enable(self.model.ctx, False)
        torch.cuda.synchronize()
        (self.pgraphs if profile else self.graphs)[d] = g
        return g

    def capture_overlap(self, d):
        """Two graphs of the step with the next batch's frozen prefix overlapped: graph b runs
        the suffix (blocks k..L-1, head), backward and update of the batch whose prefix is
        in buffer b on the capture stream, and the prefix of the next batch into buffer 1 - b
        on a second stream (forked and joined inside the graph).  Replaying 0, 1, 0, ...
        processes one batch per replay."""
        torch, R, c, cfg = self.torch, self.R, self.model.ctx, self.cfg
        R.ra_set_unfrozen_depth(c, d)
        side = torch.cuda.Stream()
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            R.ra_forward_prefix(c, self.x.data_ptr(), cfg.batch, cfg.seq, 0, stream=s.cuda_stream)
        torch.cuda.synchronize()
        graphs = []
        for b in (0, 1):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=s, capture_error_mode="relaxed"):
                cur = torch.cuda.current_stream()
                side.wait_stream(cur)
                R.ra_forward_prefix(c, self.x.data_ptr(), cfg.batch, cfg.seq, 1 - b,
                                    stream=side.cuda_stream)
                R.ra_forward_suffix(c, b, self.labels.data_ptr(), self.loss.data_ptr(), None,
                                    stream=cur.cuda_stream)
                R.ra_backward_truncated(c, cfg.n_layers - d, stream=cur.cuda_stream)
                R.ra_adapter_update(c, stream=cur.cuda_stream)
                cur.wait_stream(side)
            graphs.append(g)
        torch.cuda.synchronize()
        # buffer 0 holds a prefix for the first replay of graph 0 (graph 1 refills it)
        with torch.cuda.stream(s):
            R.ra_forward_prefix(c, self.x.data_ptr(), cfg.batch, cfg.seq, 0, stream=s.cuda_stream)
        torch.cuda.synchronize()
        self.ograph[d] = graphs

    def time_overlap(self, d, steps, warmup):
        torch = self.torch
        g = self.ograph[d]
        for i in range(2 * ((warmup + 1) // 2)):
            g[i % 2].replay()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for i in range(steps):
            g[i % 2].replay()
        b.record()
        torch.cuda.synchronize()
        return a.elapsed_time(b) / steps

    def kernel_times(self, d, reps):
        """Per-kernel device times of the step at depth d: the profiled graph (an event
        before and after every kernel) replayed `reps` times; per category, the mean over the
        replays of (time, flops, bytes, calls) of one step.  The events sit between kernels
        and take away the launch overlap, so the step is timed on the plain graph instead."""
        torch, R = self.torch, self.R
        g = self.pgraphs[d]
        acc = {}
        for _ in range(reps):
            g.replay()
            torch.cuda.synchronize()
            for k, v in R.ra_profile_read(self.model.ctx).items():
                a = acc.setdefault(k, {"ms": 0.0, "flops": v["flops"], "bytes": v["bytes"],
                                       "calls": v["calls"]})
                a["ms"] += v["ms"] / reps
        return acc

    def time_steps(self, d, steps, warmup):
        torch = self.torch
        g = self.graphs[d]
        for _ in range(warmup):
            g.replay()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(steps):
            g.replay()
        b.record()
        torch.cuda.synchronize()
        return a.elapsed_time(b) / steps

    def gemm_replay(self, d, reps):
        """The GEMM launches of one step at depth d, recorded from an eager step and replayed
        back to back in a CUDA graph (the launch overlap they have inside the step, which
        the profiled pass's event pairs take away).  Each replay (about 6 ms of GEMMs) is
        timed on its own after a 30 ms pause, as the burst peak is measured: run back to
        back for a third of a second they reach the power cap, which the step, where the
        GEMMs alternate with memory-bound kernels, does not.  Returns (launches, flops, the
        median ms per replay)."""
        torch, R, c = self.torch, self.R, self.model.ctx
        R.ra_profile_gemm_log(c, True)
        self.step(d)
        torch.cuda.synchronize()
        R.ra_profile_gemm_log(c, False)
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s, capture_error_mode="relaxed"):
            n, fl = R.ra_profile_gemm_replay(c, stream=torch.cuda.current_stream().cuda_stream)
        for _ in range(3):
            g.replay()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        times = []
        for _ in range(reps):
            time.sleep(0.03)
            a.record()
            g.replay()
            b.record()
            torch.cuda.synchronize()
            times.append(a.elapsed_time(b))
        return n, fl, statistics.median(times)

    def time_e2e_overlap(self, d, steps):
        """Host-buffer path of the overlapped schedule: per step the pinned H2D copy of the
        batch whose prefix the step starts, the two-graph step, D2H of the loss."""
        torch = self.torch
        g = self.ograph[d]
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        t0 = time.perf_counter()
        a.record()
        for i in range(steps):
            self.x.copy_(self.x_host, non_blocking=True)
            self.labels.copy_(self.labels_host, non_blocking=True)
            g[i % 2].replay()
            self.loss_host.copy_(self.loss, non_blocking=True)
        b.record()
        torch.cuda.synchronize()
        wall = time.perf_counter() - t0
        ms = max(a.elapsed_time(b), 1000 * wall) / steps
        h2d = self.x.numel() * self.x.element_size() + self.labels.numel() * 4
        return ms, h2d, 4

    def time_e2e(self, d, steps):
        """Host-buffer path: pinned H2D copy of the batch, the step, D2H of the loss."""
        torch = self.torch
        g = self.graphs[d]
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        t0 = time.perf_counter()
        a.record()
        for _ in range(steps):
            self.x.copy_(self.x_host, non_blocking=True)
            self.labels.copy_(self.labels_host, non_blocking=True)
            g.replay()
            self.loss_host.copy_(self.loss, non_blocking=True)
        b.record()
        torch.cuda.synchronize()
        wall = time.perf_counter() - t0
        ms = max(a.elapsed_time(b), 1000 * wall) / steps
        h2d = self.x.numel() * self.x.element_size() + self.labels.numel() * 4
        return ms, h2d, 4


def rank_env():
    """(world size, rank, local rank) from the torchrun environment; (1, 0, 0) without it."""
    return (int(os.environ.get("WORLD_SIZE", "1")), int(os.environ.get("RANK", "0")),
            int(os.environ.get("LOCAL_RANK", "0")))


def max_over_ranks(dist, values, device):
    """Element-wise maximum over the ranks of per-rank floats (the slowest rank's times);
    the values themselves when there is no process group."""
    if dist is None:
        return [float(v) for v in values]
    import torch
    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return t.tolist()


def job_value(world, batch, ms):
    """Whole-job samples/s: the samples of every replica over the slowest replica's step."""
    return world * batch / (ms / 1000.0)


def gemm_rate(prof, peaks):
    """GEMM throughput of one step from the profiled pass, against the measured peaks."""
    g = prof.get("gemm")
    if not g or g["ms"] <= 0:
        return None
    tf = g["flops"] / (g["ms"] / 1000.0) / 1e12
    return {"tflops": tf, "frac_burst": tf / peaks["bf16_tflops"],
            "frac_sustained": tf / peaks["bf16_tflops_sustained"], "calls": g["calls"],
            "flops": g["flops"], "ms": g["ms"]}


def gpu_main(args):
    import torch
    import synth
    world, rank, local = rank_env()
    dist = None
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    else:
        torch.cuda.set_device(0)
    device = "cuda:%d" % torch.cuda.current_device()

    import __graft_entry__
    __graft_entry__.build()
    from paper_2502_19864_gb300 import ringada as R

    cfg = synth.CONFIGS[args.config]
    global SWEEP, HEADLINE_D
    SWEEP, HEADLINE_D = SWEEPS[args.config]
    peaks, peak_kind = measured_peaks()
    steps, warmup = args.steps, max(3, args.warmup)

    # CPU baseline first (its own process, before the GPU work starts)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = run_cpu_baseline(args.config, HEADLINE_D,
                               min(cfg.batch, CPU_SAMPLE_BATCH.get(args.config, 1)), 12.0)

    run = Runner(cfg, max(SWEEP), device, prefix_buffers=int(cfg.arch == "encoder"))
    sweep = {}
    for d in SWEEP:
        run.capture(d)
    run.capture(HEADLINE_D, profile=True)
    # the clock sampler runs through every timed region; each region keeps its window
    clk = start_clock_sampler(torch.cuda.current_device())
    windows = {}
    # sweep points (not the headline)
    for d in SWEEP:
        if d != HEADLINE_D:
            t0 = time.time()
            sweep[d] = run.time_steps(d, steps, warmup)
            windows["d=%d" % d] = (t0, time.time())
    # the headline depth as one sequential graph per step
    t0 = time.time()
    seq_ms = run.time_steps(HEADLINE_D, steps, warmup)
    windows["sequential"] = (t0, time.time())
    sweep[HEADLINE_D] = seq_ms
    # headline: the method's schedule.  Encoders run the next batch's frozen prefix on a
    # second stream while this batch's suffix, backward and update run (Section III-A: the
    # forward below the unfreezing depth does not depend on them); one batch per step, the
    # same kernels, results bitwise those of the sequential step.  Decoders: the plain graph.
    overlapped = cfg.arch == "encoder"
    if overlapped:
        run.capture_overlap(HEADLINE_D)
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    t0 = time.time()
    ms = run.time_overlap(HEADLINE_D, steps, warmup) if overlapped else run.time_steps(HEADLINE_D, steps, warmup)
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    windows["headline"] = (t0, time.time())
    t0 = time.time()
    e2e_ms, h2d, d2h = run.time_e2e_overlap(HEADLINE_D, steps) if overlapped else run.time_e2e(HEADLINE_D, steps)
    windows["e2e"] = (t0, time.time())
    # per-kernel device times: a further timed region, the same step with an event around
    # every kernel (replays of the profiled graph)
    t0 = time.time()
    prof = run.kernel_times(HEADLINE_D, min(steps, 50))
    windows["kernel_times"] = (t0, time.time())
    launches_headline = run.launches[HEADLINE_D]
    saved_by_d = dict(run.saved)
    # the next batch's frozen prefix on a second stream, overlapping this batch's suffix,
    # backward and update (same work per step; timed the same way)
    overlap = None
    if cfg.arch == "encoder":
        overlap = {}
        t0 = time.time()
        for d in SWEEP:
            if d == HEADLINE_D:
                o_ms = ms  # the headline (timed above)
            else:
                run.capture_overlap(d)
                o_ms = run.time_overlap(d, steps, warmup)
            overlap["d=%d" % d] = {"ms_per_step": o_ms, "samples_per_s": job_value(world, cfg.batch, o_ms),
                                   "sequential_ms_per_step": sweep[d],
                                   "speedup": sweep[d] / o_ms}
        windows["overlap"] = (t0, time.time())
    # the step's GEMM launches back to back (a further timed region)
    t0 = time.time()
    g_n, g_fl, g_ms = run.gemm_replay(HEADLINE_D, max(5, min(steps, 20)))
    windows["gemm_replay"] = (t0, time.time())
    R.ra_set_unfrozen_depth(run.model.ctx, HEADLINE_D)

    # the slowest rank's times (headline, end to end and every sweep point)
    sweep_d = sorted(sweep)
    red = max_over_ranks(dist, [ms, e2e_ms] + [sweep[d] for d in sweep_d], device)
    ms, e2e_ms = red[0], red[1]
    sweep = dict(zip(sweep_d, red[2:]))
    seq_ms = sweep[HEADLINE_D]

    B = cfg.batch
    value = job_value(world, B, ms)
    gr = gemm_rate(prof, peaks)
    traffic_per_flop, traffic_note = gemm_traffic()
    g = prof["gemm"]
    launches_per_gemm = max(1, g["calls"])
    replay_tf = g_fl / (g_ms / 1000.0) / 1e12 if g_ms > 0 else None
    roof = {
        "kernel": "frozen-weight and dX GEMMs (tcgen05, bf16 in, fp32 accumulate), all launches of one step",
        "bound": "tensor", "unit": "TFLOP/s",
        "achieved": replay_tf,
        "peak": peaks["bf16_tflops"],
        "peak_kind": "%s dense bf16 burst (cuBLAS GEMM timed alone; the SM clock stays at its maximum "
                     "through this step)" % peak_kind,
        "frac": replay_tf / peaks["bf16_tflops"] if replay_tf else None,
        "frac_of_sustained": replay_tf / peaks["bf16_tflops_sustained"] if replay_tf else None,
        "peak_sustained": peaks["bf16_tflops_sustained"],
        "launches": g_n,
        "flops_per_launch": g_fl / max(1, g_n),
        "avg_launch_us": 1000.0 * g_ms / max(1, g_n),
        "traffic": (traffic_per_flop * g["flops"] / launches_per_gemm) if traffic_per_flop else None,
        "traffic_note": traffic_note,
        "timing": "the step's %d GEMM launches (same shapes, operands, epilogues and buffers) replayed "
                  "back to back in a CUDA graph; each replay timed alone with CUDA events after a 30 ms "
                  "pause, as the burst peak is (back to back for longer they reach the power cap, which "
                  "the step does not); median of the replays; avg launch duration = replay time / "
                  "launches" % g_n,
        "event_pair": {"achieved": gr["tflops"] if gr else None,
                       "frac": gr["frac_burst"] if gr else None,
                       "note": "each GEMM launch between its own pair of CUDA events inside the profiled "
                               "step graph: adds the launch gap and prologue that programmatic "
                               "dependent launch hides in the step (lower bound)"},
    }
    if cfg.dtype != "bf16":
        # fp32 models run the SIMT GEMM (FFMA): against the FFMA peak of 152 SMs x 128 lanes x
        # 2 flops x 2.07 GHz, not the tensor-core peak
        ffma_peak = 152 * 128 * 2 * 2.07e9 / 1e12
        roof.update({"kernel": "frozen-weight and dX GEMMs (SIMT fp32, FFMA), all launches of one step",
                     "bound": "alu", "peak": ffma_peak,
                     "peak_kind": "FFMA issue rate: 152 SMs x 128 lanes x 2 flops x 2070 MHz",
                     "frac": replay_tf / ffma_peak if replay_tf else None,
                     "frac_of_sustained": None, "peak_sustained": None, "traffic": None,
                     "traffic_note": "the DRAM capture covers the tensor-core GEMM"})
        roof["event_pair"]["frac"] = (gr["tflops"] / ffma_peak) if gr and gr["tflops"] else None
    phases = {k: {"ms": v["ms"], "calls": v["calls"],
                  "tflops": (v["flops"] / v["ms"] / 1e9) if v["ms"] > 0 and v["flops"] else None,
                  "gbs": (v["bytes"] / v["ms"] / 1e6) if v["ms"] > 0 and v["bytes"] else None}
              for k, v in prof.items()}
    phases_sum = sum(v["ms"] for v in prof.values())

    extra = None
    if rank == 0 and not args.no_extra and args.config == "large":
        del run
        torch.cuda.empty_cache()
        extra = base_sweep(torch, R, synth, device, peaks, steps, warmup, windows)
    samples = stop_clock_sampler(clk)
    clocks = clock_record(samples, *windows["headline"])
    clocks["whole_run"] = clock_record(samples, min(w[0] for w in windows.values()),
                                       max(w[1] for w in windows.values()))
    clocks["by_region"] = {k: clock_record(samples, *w) for k, w in windows.items()
                           if k != "headline"}

    if rank != 0:
        if dist:
            dist.destroy_process_group()
        return 0
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": steps,
        "warmup": warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": cfg.dtype, "data": "synthetic",
        "config": dict(workload_config(args.config, HEADLINE_D, world), cuda_graph=True),
        "sweep": {"d=%d" % d: {"samples_per_s": job_value(world, B, sweep[d]),
                               "ms_per_step": sweep[d], "k": cfg.n_layers - d,
                               "saved_activation_bytes": saved_by_d[d]}
                  for d in sorted(sweep)},
        "monotone_in_k": all(sweep[a] > sweep[b] for a, b in zip(sorted(sweep)[1:], sorted(sweep))),
        "saved_bytes_at_headline": saved_by_d[HEADLINE_D],
        "roofline": roof,
        "phases_ms": phases,
        "phases_note": "per-kernel times from the profiled replay of the sequential step (an "
                       "event pair around every kernel removes the launch overlap); their sum is "
                       "%.3f ms, %.2fx the plain sequential step" % (phases_sum, phases_sum / seq_ms if seq_ms else 0.0),
        "schedule": ("the next batch's frozen prefix (layers below k) on a second stream while this "
                     "batch's suffix, backward and update run (Section III-A); one batch per step"
                     if overlapped else "one graph per step"),
        "sequential": {"samples_per_s": job_value(world, B, seq_ms), "ms_per_step": seq_ms,
                       "note": "the same step with every kernel on one stream"},
        "clocks": clocks,
        "e2e": {"value": job_value(world, B, e2e_ms), "unit": UNIT,
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": e2e_ms},
        "gpu_launches": launches_headline * steps,
        "gpu_launches_per_step": launches_headline,
        "cpu_baseline": cpu,
        "prefix_overlap": overlap,
        "base": extra,
    }
    print(json.dumps(line))
    if dist:
        dist.destroy_process_group()
    return 0


def base_sweep(torch, R, synth, device, peaks, steps, warmup, windows):
    """The BERT-base-shaped step over d = 1, 3, 6, 12: samples/s and, at d = 6, the GEMMs'
    throughput from a profiled replay."""
    cfg = synth.CONFIGS["base"]
    ds, hd = SWEEPS["base"]
    run = Runner(cfg, max(ds), device, prefix_buffers=1)
    out = {}
    for d in ds:
        run.capture(d)
        run.capture_overlap(d)
    run.capture(hd, profile=True)
    t0 = time.time()
    for d in ds:
        ms = run.time_steps(d, steps, warmup)
        o_ms = run.time_overlap(d, steps, warmup)
        out["d=%d" % d] = {"samples_per_s": cfg.batch / (ms / 1000.0), "ms_per_step": ms,
                           "saved_activation_bytes": run.saved[d],
                           "prefix_overlap": {"samples_per_s": cfg.batch / (o_ms / 1000.0),
                                              "ms_per_step": o_ms, "speedup": ms / o_ms}}
    prof = run.kernel_times(hd, min(steps, 50))
    g_n, g_fl, g_ms = run.gemm_replay(hd, max(5, min(steps, 20)))
    windows["base"] = (t0, time.time())
    out["gemm_at_d=%d" % hd] = gemm_rate(prof, peaks)
    rtf = g_fl / (g_ms / 1000.0) / 1e12
    out["gemm_replay_at_d=%d" % hd] = {"tflops": rtf, "frac_burst": rtf / peaks["bf16_tflops"],
                                       "launches": g_n, "ms": g_ms}
    out["phases_ms_at_d=%d" % hd] = {k: round(v["ms"], 4) for k, v in prof.items()}
    return out


def schedule_main(args):
    """The schedule workload: 600 steps of BERT-base with d(s) = min(1 + s // 50, 12), Adam
    lr 1e-4, one fresh synthetic batch per step (host pinned buffer -> device each step).
    Reports per-depth step time and phase breakdown, saved-activation bytes per depth, and
    the loss trajectory (the first five losses are checked against the oracle in the tests)."""
    import torch
    import synth
    import __graft_entry__
    __graft_entry__.build()
    from paper_2502_19864_gb300 import ringada as R
    torch.cuda.set_device(0)
    cfg = synth.CONFIGS["base"]
    run = Runner(cfg, 12, "cuda:0")
    n_steps, interval = 600, 50
    batches = [synth.make_batch(cfg, 1000 + i) for i in range(4)]
    xs = [torch.tensor(x, dtype=torch.float32).to(torch.bfloat16).pin_memory() for x, _ in batches]
    ys = [torch.tensor(y, dtype=torch.int32).pin_memory() for _, y in batches]
    per_d = {}
    losses = []
    for d in range(1, 13):
        run.capture(d)
    torch.cuda.synchronize()
    t_all = time.perf_counter()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n_steps)]
    loss_host = torch.zeros(n_steps, dtype=torch.float32).pin_memory()
    for s in range(n_steps):
        d = R.schedule_depth(s, interval=interval, d0=1, d_max=12)
        run.x.copy_(xs[s % 4], non_blocking=True)
        run.labels.copy_(ys[s % 4], non_blocking=True)
        ev[s][0].record()
        run.graphs[d].replay()
        ev[s][1].record()
        loss_host[s:s + 1].copy_(run.loss, non_blocking=True)
    torch.cuda.synchronize()
    wall = time.perf_counter() - t_all
    for s in range(n_steps):
        d = R.schedule_depth(s, interval=interval, d0=1, d_max=12)
        per_d.setdefault(d, []).append(ev[s][0].elapsed_time(ev[s][1]))
    losses = loss_host.tolist()
    # per-phase breakdown and saved bytes per depth (one profiled replay each)
    phases, saved = {}, {}
    for d in range(1, 13):
        run.capture(d, profile=True)
        prof = run.kernel_times(d, 5)
        phases["d=%d" % d] = {k: round(v["ms"], 4) for k, v in prof.items()}
        saved["d=%d" % d] = run.saved[d]
    out = {
        "workload": "schedule: bert-base 600 steps, d = min(1 + s // 50, 12), Adam lr 1e-4",
        "steps": n_steps, "wall_s": wall,
        "ms_per_step_by_depth": {"d=%d" % d: statistics.median(v) for d, v in sorted(per_d.items())},
        "samples_per_s_overall": n_steps * cfg.batch / (sum(sum(v) for v in per_d.values()) / 1000.0),
        "phases_ms_by_depth": phases,
        "saved_activation_bytes_by_depth": saved,
        "loss_first5": losses[:5], "loss_every50": losses[::50], "loss_last": losses[-1],
    }
    print(json.dumps(out))
    return 0


def main():
    args = parse()
    if args.schedule:
        return schedule_main(args)
    if args.cpu_worker:
        cpu_worker(args.cpu_worker)
        return 0
    if args.impl == "reference":
        return reference_main(args)
    return gpu_main(args)


if __name__ == "__main__":
    sys.exit(main())
