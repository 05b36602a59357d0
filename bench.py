#!/usr/bin/env python
"""Benchmark of the RDN layer hot path on GB300.

A step is one pass of the whole training-side hot path over one batch of
the fwd+bwd workload (RDN, B=8, H=16, T=4096, d_k=d_v=128, bf16 inputs, fp32
states, chunk 64, clip 1): rdn_fwd (saving the chunk-start states) followed
by rdn_bwd.  `value` is tokens/s (a token = one (b, t) position with all 16
heads) over all ranks.  The decode workload (N=256 sequences, H=16, D=128,
fp32 states in place, 1000 steps) is timed in the same run and reported as
HBM GB/s under "decode".

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

One JSON line is printed by rank 0.  With --gpus N > 1 (one process per GPU
under torchrun) every rank runs an independent replica on its own batch
(the layer has no parameters and no exchange step): "scaling" is "weak".
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

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "RDN fwd+bwd tokens/sec (H=16,d=128,T=4096 bf16); % bf16 tensor peak; decode GB/s"
WORKLOAD = "rdn_fwd_bwd_bf16_B8H16T4096D128"
DECODE_WORKLOAD = "rdn_decode_N256H16D128"
C = 64

# Algorithmic work per token-head at d_k = d_v = d, chunk C (triangular
# products counted at half, each unit-lower inverse at (2/3) C^3 per chunk):
#   forward F = 12 d^2 + 2 C d + 5 C d + (4/3) C^2, split into
#     the state-carrying scan   12 d^2 + 5 C d   (products with S, R and the
#                                                 C x C x d_v chunk products)
#     the per-chunk prep        2 C d + (4/3) C^2 (Gram matrices, inverses)
#   backward = 2 x forward (two products per forward product), same split:
#     the reverse scan carrying dS, dR            12 d^2 + 5 C d
#     the products over the value dimension        12 d^2 + 5 C d
#     (dK, dQ state terms; C x C gradients)
#     the backward of the prep                     2 (2 C d + (4/3) C^2)
#   (the tensor-core bwd_post does the last two; the SIMT path splits them
#   into bwd_scan and bwd_finish).  Recomputation of forward pieces is not
#   algorithmic work (counted 0).
#   The same work with every C x C x d product counted as a dense tile (the
#   triangular ones at full size): forward + 7 C d per token-head.
def flops_per_token_head(d=128, c=C):
    scan = 12 * d * d + 5 * c * d
    prep = 2 * c * d + (4.0 / 3.0) * c * c
    return dict(fwd=scan + prep, fwd_scan=scan, fwd_prep=prep, bwd_scan=2 * scan,
                bwd_chain=scan, bwd_post=scan + 2 * prep, bwd_finish=2 * prep, recompute=0.0,
                step=3 * (scan + prep), step_dense_tiles=3 * (scan + prep + 7 * c * d))


# kernel name (as recorded by the library) -> algorithmic flop per token-head
KERNEL_WORK = {"chunk_scan": "fwd_scan", "fwd_tc_scan": "fwd_scan", "chunk_prep": "fwd_prep",
               "bwd_scan": "bwd_scan", "bwd_chain": "bwd_chain", "bwd_post": "bwd_post",
               "bwd_finish": "bwd_finish", "bwd_recompute": "recompute"}

# decode: read + write S and R fp32, plus q, k, v, o bf16 and three fp32 gates
def decode_bytes_per_head(d=128):
    return 4 * d * d * 4 + 4 * d * 2 + 3 * 4


def _peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return dict(hbm=float(p["hbm_gbs"]), bf16=float(p["bf16_tflops"]),
                    bf16_sust=float(p.get("bf16_tflops_sustained", p["bf16_tflops"])),
                    source="measured")
    except Exception:
        return dict(hbm=6800.0, bf16=1900.0, bf16_sust=1700.0, source="fallback")


# ------------------------------------------------------------------ clocks
class ClockSampler:
    """nvidia-smi sampling of SM clock and throttle reasons during a region:
    samples every 50 ms with their timestamps; the summary keeps those that
    fall inside the region marked by begin() / end() (host wall clock)."""

    Q = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    PERIOD_MS = 50

    def __init__(self, gpu_index, enabled=True):
        self.gpu = gpu_index
        self.enabled = enabled
        self.proc = None
        self.path = None
        self.t0 = self.t1 = None

    def begin(self):
        self.t0 = time.time()

    def end(self):
        self.t1 = time.time()

    def __enter__(self):
        if not self.enabled:
            return self
        fd, self.path = tempfile.mkstemp(prefix="rdn_clocks_", suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", str(self.PERIOD_MS)],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
        return False

    def summary(self):
        if not self.enabled:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["not sampled (--profile)"]}
        if self.proc is None or not self.path:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        with open(self.path) as f:
            lines = f.readlines()
        os.unlink(self.path)
        rows, where = clock_rows_in_region(lines, self.t0, self.t1)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        reasons = set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            for nm, val in zip(names, r[5:9]):
                if val.lower() in ("active", "1"):
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": sorted(reasons),
                "samples": len(rows), "sampled": where,
                "region_ms": (None if self.t0 is None or self.t1 is None
                              else round(1e3 * (self.t1 - self.t0), 1)),
                "power_w_max": max((float(r[3]) for r in rows
                                    if r[3].replace(".", "").isdigit()), default=None)}


def clock_rows_in_region(lines, t0, t1):
    """The nvidia-smi CSV rows (timestamp first) whose time falls in [t0, t1]
    (host epoch seconds); if none does (a region shorter than the sampling
    period), the first row after t0.  Returns (rows, "in region" | "first
    after start" | "all")."""
    import datetime
    rows = []
    for ln in lines:
        parts = [p.strip() for p in ln.split(",")]
        if len(parts) < 9:
            continue
        try:
            ts = datetime.datetime.strptime(parts[0], "%Y/%m/%d %H:%M:%S.%f").timestamp()
        except ValueError:
            ts = None
        rows.append((ts, parts))
    if t0 is None or t1 is None or any(ts is None for ts, _ in rows):
        return [r for _, r in rows], "all"
    inside = [r for ts, r in rows if t0 <= ts <= t1]
    if inside:
        return inside, "in region"
    after = [r for ts, r in rows if ts > t0]
    return after[:1], "first after start"


# ------------------------------------------------------------- distributed
def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def init_dist(ws):
    if ws <= 1:
        return None
    import torch.distributed as dist
    if not dist.is_initialized():
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        dist.init_process_group("gloo")
    return dist


def barrier(dist):
    if dist is not None:
        dist.barrier()


def max_over_ranks(dist, x):
    """Largest value of x over all ranks (timing exchange only)."""
    if dist is None:
        return float(x)
    import torch
    t = torch.tensor([float(x)], dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(dist, x):
    if dist is None:
        return float(x)
    import torch
    t = torch.tensor([float(x)], dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


def aggregate(dist, local_ms, local_units):
    """Whole-job throughput: units of all ranks / slowest rank's time."""
    t = max_over_ranks(dist, local_ms)
    u = sum_over_ranks(dist, local_units)
    return t, u / (t / 1e3)


# -------------------------------------------------------------- CPU oracle
def time_oracle_sample(target_s=15.0, max_heads=None):
    """fp64 oracle fwd+bwd on a bounded sample of the workload (whole
    sequences of T=4096 for a subset of heads), on all host cores."""
    import numpy as np
    import oracle
    from rdn_synthetic import WORKLOADS, make_workload_inputs

    oracle.build()
    w = WORKLOADS[WORKLOAD]
    threads = oracle.max_threads()

    def heads_as_batch(t, nh):
        """[B,T,H,...] -> the first nh (b,h) sequences as [nh,T,1,...]."""
        t = t.double().numpy()
        t = np.moveaxis(t, 2, 1)                      # [B,H,T,...]
        t = t.reshape(-1, *t.shape[2:])[:nh]          # [B*H,T,...] -> [nh,T,...]
        return np.ascontiguousarray(np.expand_dims(t, 2))

    def run(nh):
        B = max(1, (nh + w.H - 1) // w.H)
        x = make_workload_inputs(w, B=B, seed=1)
        q, k, v, g, be, gm, dO = (heads_as_batch(x[n], nh)
                                  for n in ("q", "k", "v", "g", "beta", "gamma", "dO"))
        t0 = time.perf_counter()
        oracle.rdn_fwd(q, k, v, g, be, gm, w.clip)
        oracle.rdn_bwd(q, k, v, g, be, gm, w.clip, None, None, dO)
        return time.perf_counter() - t0

    probe_heads = min(threads, 16)
    dt = run(probe_heads)
    nh = probe_heads
    if dt < target_s:
        nh = int(probe_heads * max(1.0, target_s / max(dt, 1e-3)))
        nh = max(probe_heads, (nh // threads) * threads)
        if max_heads:
            nh = min(nh, max_heads)
        dt = run(nh)
    tokens = nh * w.T / w.H
    # one head on one thread: the oracle's single-core rate
    oracle.set_threads(1)
    try:
        dt1 = run(1)
    finally:
        oracle.set_threads(threads)
    single = (w.T / w.H) / dt1
    return dict(value=tokens / dt, unit="tokens/s", cores=min(threads, nh), kind="oracle",
                single_thread_value=single, single_thread_sample=f"1 (b,h) head, T={w.T}, "
                f"{dt1:.1f} s on 1 thread",
                sample=f"fp64 oracle fwd+bwd on {nh} of the workload's (b,h) heads, "
                       f"full T={w.T} each ({nh * w.T} token-heads = {tokens:.0f} tokens), "
                       f"{dt:.1f} s on {min(threads, nh)} OpenMP threads")


def cpu_model():
    """The host CPU's model name, as the OS reports it."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for ln in out.splitlines():
            if ln.startswith("Model name:"):
                return ln.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        with open("/proc/cpuinfo") as f:
            for ln in f:
                if ln.lower().startswith("model name"):
                    return ln.split(":", 1)[1].strip()
    except OSError:
        pass
    import platform
    return platform.processor() or platform.machine()


def time_oracle_configs(target_s=2.0):
    """The oracle on the other workloads, on the host's cores and on one
    thread: the forward workloads (one whole-T head per thread, and one head
    on one thread; rate = heads x T / H / time) and the decode step (a sample
    of the N sequences, all H heads, for one step, scaled to all of them)."""
    import oracle
    from rdn_synthetic import WORKLOADS, make_decode_inputs, make_workload_inputs

    oracle.build()
    threads = oracle.max_threads()
    out = {}

    def heads_as_batch(t, nh):
        t = np.moveaxis(t, 2, 1)
        t = t.reshape(-1, *t.shape[2:])[:nh]
        return np.ascontiguousarray(np.expand_dims(t, 2))

    def fwd_rate(w, nh):
        x = make_workload_inputs(w, seed=3)
        a = {n: (None if t is None else t.double().numpy()) for n, t in x.items()}
        nh = min(nh, w.B * w.H)
        q, k, v, g, be, gm = (heads_as_batch(a[n], nh) for n in ("q", "k", "v", "g", "beta",
                                                                 "gamma"))
        st = lambda t: None if t is None else np.ascontiguousarray(
            t.reshape(-1, 1, *t.shape[2:])[:nh])
        variant = oracle.RLA if w.op == "rla_fwd" else oracle.RDN
        t0 = time.perf_counter()
        oracle.fwd(variant, q, k, v, g, be, gm, w.clip, st(a["S0"]), st(a["R0"]))
        dt = time.perf_counter() - t0
        return nh, dt, nh * w.T / w.H / dt  # tokens/s (a token = all H heads)

    for name in ("rla_fwd_f32_B1H2T256D64", "rdn_fwd_bf16_B8H16T2048D128",
                 "rdn_fwd_bf16_B2H16T16384D128_state"):
        w = WORKLOADS[name]
        nh, dt, val = fwd_rate(w, threads)  # one whole-T head per thread
        oracle.set_threads(1)
        try:
            nh1, dt1, val1 = fwd_rate(w, 1)
        finally:
            oracle.set_threads(threads)
        out[name] = {"value": val, "unit": "tokens/s", "cores": min(threads, nh),
                     "single_thread_value": val1,
                     "sample": f"fp64 oracle forward of {nh} of the {w.B * w.H} (b,h) heads, "
                               f"T={w.T} each, {dt:.2f} s; one head on one thread "
                               f"{dt1:.2f} s (rate = heads x T / H / time)"}
    wd = WORKLOADS["rdn_decode_N256H16D128"]

    def dec_rate(n_seq):
        y = make_decode_inputs(n_seq, wd.H, wd.D, steps=1, seed=4)
        a = {k_: t.double().numpy() for k_, t in y.items()}
        t0 = time.perf_counter()
        oracle.decode_step(oracle.RDN, a["q"][0], a["k"][0], a["v"][0], a["g"][0],
                           a["beta"][0], a["gamma"][0], wd.clip, a["S"], a["R"])
        return time.perf_counter() - t0

    nseq = 8
    dt = dec_rate(nseq)
    nseq = max(1, min(wd.B, int(nseq * target_s / max(dt, 1e-4))))
    dt = dec_rate(nseq)
    oracle.set_threads(1)
    try:
        dt1 = dec_rate(1)
    finally:
        oracle.set_threads(threads)
    scale = wd.B / nseq
    out[wd.name] = {"value": 1.0 / (dt * scale), "unit": "steps/s (all 256 x 16 heads)",
                    "cores": min(threads, nseq * wd.H),
                    "single_thread_value": 1.0 / (dt1 * wd.B),
                    "sample": f"one fp64 oracle decode step of {nseq} of the {wd.B} sequences "
                              f"(x {wd.H} heads), {dt:.3f} s, scaled by {scale:.0f} to all "
                              f"{wd.B}; one sequence on one thread {dt1:.3f} s, scaled by "
                              f"{wd.B}"}
    return out


# ------------------------------------------------------------ reference arm
def run_reference(args):
    ws, rank, _ = dist_env()
    if rank != 0:
        return 0
    import numpy as np
    import oracle
    from rdn_synthetic import WORKLOADS, make_workload_inputs

    oracle.build()
    w = WORKLOADS[WORKLOAD]
    threads = oracle.max_threads()
    # each step: all 16 heads of one sequence (T = 4096 tokens)
    x = make_workload_inputs(w, B=1, seed=2)
    a = {n: (None if t is None else t.double().numpy()) for n, t in x.items()}

    def step():
        oracle.rdn_fwd(a["q"], a["k"], a["v"], a["g"], a["beta"], a["gamma"], w.clip)
        oracle.rdn_bwd(a["q"], a["k"], a["v"], a["g"], a["beta"], a["gamma"], w.clip, None,
                       None, a["dO"])

    for _ in range(args.warmup):
        step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step()
    dt = time.perf_counter() - t0
    tokens = w.T * args.steps
    val = tokens / dt
    line = {"impl": "reference", "metric": METRIC, "value": val, "unit": "tokens/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": dt * 1e3 / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": _config(w),
            "cpu_baseline": {"value": val, "unit": "tokens/s", "cores": min(threads, w.H),
                             "kind": "oracle",
                             "sample": f"each step: fp64 oracle fwd+bwd of one sequence "
                                       f"(B=1 of the workload's B=8), all H={w.H} heads, "
                                       f"T={w.T}"},
            "e2e": {"value": val, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def _workload(args):
    """The fwd+bwd workload, optionally shrunk (--B/--T) for profiler captures."""
    import dataclasses
    from rdn_synthetic import WORKLOADS
    w = WORKLOADS[WORKLOAD]
    if args.B or args.T:
        B, T = args.B or w.B, args.T or w.T
        w = dataclasses.replace(w, B=B, T=T, name=f"rdn_fwd_bwd_bf16_B{B}H{w.H}T{T}D{w.D}")
    return w


def _config(w):
    return {"workload": w.name, "B": w.B, "T": w.T, "H": w.H, "d_k": w.D, "d_v": w.D,
            "chunk": w.chunk, "clip": w.clip, "states": "fp32", "parallelism": "replicas",
            "l2": f"no flush: inputs larger than L2 (q,k,v,dO = "
                  f"{4 * w.B * w.T * w.H * w.D * 2 / 1e6:.0f} MB bf16 per step)"}


def _traffic(kernel):
    """DRAM bytes per launch from the committed ncu summary, if it was taken
    on the current kernel source (else None)."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            tab = json.load(f)
        ent = tab.get(kernel)
        if not ent:
            return None
        import hashlib
        srcs = ent["source"] if isinstance(ent["source"], list) else [ent["source"]]
        hs = hashlib.sha256()
        for sname in srcs:
            hs.update(open(os.path.join(ROOT, sname), "rb").read())
        h = hs.hexdigest()[:16]
        if h != ent["source_sha256_16"]:
            return None
        return float(ent["bytes_per_launch_full_workload"])
    except Exception:
        return None


# ------------------------------------------------------------------ our arm
def run_ours(args):
    import torch

    ws, rank, local = dist_env()
    dist = init_dist(ws)
    torch.cuda.set_device(local)
    import paper_2509_25223_gb300 as rdn
    from rdn_synthetic import WORKLOADS, make_decode_inputs, make_workload_inputs, packed_lengths

    rdn.library()  # fails loudly when the CUDA library is missing
    w = _workload(args)
    peaks = _peaks()
    dev = torch.device("cuda", local)
    x = make_workload_inputs(w, device=dev, device_rng=True, seed=rank)
    names = ("q", "k", "v", "g", "beta", "gamma")
    B, T, H, D = w.B, w.T, w.H, w.D
    NC = (T + C - 1) // C
    o = torch.empty(B, T, H, D, dtype=torch.bfloat16, device=dev)
    wsf = torch.empty(rdn.workspace_bytes("rdn_fwd", B, T, H, D, save_for_bwd=True),
                      dtype=torch.uint8, device=dev)
    wsb = torch.empty(rdn.workspace_bytes("rdn_bwd", B, T, H, D), dtype=torch.uint8, device=dev)
    grads = dict(dq=torch.empty_like(x["q"]), dk=torch.empty_like(x["k"]),
                 dv=torch.empty_like(x["v"]),
                 dg=torch.empty(B, T, H, device=dev), dbeta=torch.empty(B, T, H, device=dev),
                 dgamma=torch.empty(B, T, H, device=dev),
                 dS0=torch.empty(B, H, D, D, device=dev), dR0=torch.empty(B, H, D, D, device=dev))

    def step(inp):
        _, _, _, Sc, Rc = rdn.rdn_fwd(*(inp[n] for n in names), clip=w.clip,
                                      return_chunk_states=True, out=o, workspace=wsf,
                                      save_for_bwd=True)
        rdn.rdn_bwd(*(inp[n] for n in names), inp["dO"], clip=w.clip, S_chunks=Sc,
                    R_chunks=Rc, workspace=wsb, out=grads, fwd_workspace=wsf, fwd_saved=True)

    for _ in range(args.warmup):
        step(x)
    torch.cuda.synchronize()
    barrier(dist)
    stream = torch.cuda.current_stream()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local, enabled=not args.profile) as clk:
        with rdn.LaunchTimer() as lt:
            torch.cuda.synchronize()
            clk.begin()
            e0.record(stream)
            for _ in range(args.steps):
                step(x)
            e1.record(stream)
            torch.cuda.synchronize()
            clk.end()
    barrier(dist)
    local_ms = e0.elapsed_time(e1)
    tokens_per_step = B * T
    tmax, value = aggregate(dist, local_ms, tokens_per_step * args.steps)
    ms_per_step = tmax / args.steps
    fl = flops_per_token_head(D)
    token_heads = B * T * H

    kern = lt.summary()
    dom = max(kern.items(), key=lambda kv: kv[1][1])
    dom_name, (dom_n, dom_total, dom_mean) = dom
    dom_flop = fl[KERNEL_WORK[dom_name]] * token_heads
    achieved = dom_flop / (dom_mean * 1e-3) / 1e12
    peak = peaks["bf16_sust"]
    roof = {"kernel": dom_name, "bound": "tensor", "achieved": achieved, "peak": peak,
            "unit": "TFLOP/s", "frac": achieved / peak, "traffic": _traffic(dom_name),
            "peak_kind": f"bf16 dense, {peaks['source']} sustained (kernel timed inside a long step)",
            "algorithmic_flop_per_launch": dom_flop, "mean_launch_ms": dom_mean}
    step_tflops = fl["step"] * token_heads / (ms_per_step * 1e-3) / 1e12
    step_tflops_dense = fl["step_dense_tiles"] * token_heads / (ms_per_step * 1e-3) / 1e12

    # ---- end to end through the public API: pinned host in, host out.  Each
    # step copies all its inputs in from pinned host memory and reads its
    # result, the layer output o, back to the host (the gradients stay on the
    # device, where a training step's optimizer uses them); the copies run on
    # their own streams, so that step i + 1's inputs arrive and step i's output
    # leaves while a step computes (two device buffer sets, ordered by events).
    e2e_val = h2d = d2h = e2e_steps = None
    if not args.profile:  # (profiler captures time the step alone)
        host = {n: x[n].cpu().pin_memory() for n in names + ("dO",)}
        dev_in = [{n: torch.empty_like(x[n]) for n in host} for _ in range(2)]
        outs = [(torch.empty_like(o), {n: torch.empty_like(t) for n, t in grads.items()})
                for _ in range(2)]
        host_out = {"o": torch.empty(o.shape, dtype=o.dtype, pin_memory=True)}
        h2d = sum(t.numel() * t.element_size() for t in host.values())
        d2h = sum(t.numel() * t.element_size() for t in host_out.values())
        s_in, s_out = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
        ev = lambda: torch.cuda.Event()
        in_ready, in_free = [ev(), ev()], [ev(), ev()]
        out_ready, out_free = [ev(), ev()], [ev(), ev()]

        def e2e_step(i):
            bsel = i % 2
            with torch.cuda.stream(s_in):
                if i >= 2:
                    s_in.wait_event(in_free[bsel])
                for n, t in host.items():
                    dev_in[bsel][n].copy_(t, non_blocking=True)
                in_ready[bsel].record(s_in)
            oo, gg = outs[bsel]
            stream.wait_event(in_ready[bsel])
            if i >= 2:
                stream.wait_event(out_free[bsel])
            _, _, _, Sc, Rc = rdn.rdn_fwd(*(dev_in[bsel][n] for n in names), clip=w.clip,
                                          return_chunk_states=True, out=oo, workspace=wsf,
                                          save_for_bwd=True)
            rdn.rdn_bwd(*(dev_in[bsel][n] for n in names), dev_in[bsel]["dO"], clip=w.clip,
                        S_chunks=Sc, R_chunks=Rc, workspace=wsb, out=gg, fwd_workspace=wsf,
                        fwd_saved=True)
            in_free[bsel].record(stream)
            out_ready[bsel].record(stream)
            with torch.cuda.stream(s_out):
                s_out.wait_event(out_ready[bsel])
                for n, t in host_out.items():
                    t.copy_(oo if n == "o" else gg[n], non_blocking=True)
                out_free[bsel].record(s_out)

        # (steady state of the two-deep pipeline: the first input copy and the last
        # output read are not overlapped with compute, so they are spread over
        # at least 30 steps, as over the many steps of a training run)
        e2e_steps = max(30, min(args.steps, 60))
        for i in range(2):
            e2e_step(i)
        torch.cuda.synchronize()
        barrier(dist)
        e0.record(s_in)
        for i in range(e2e_steps):
            e2e_step(i)
        e1.record(s_out)
        torch.cuda.synchronize()
        barrier(dist)
        _, e2e_val = aggregate(dist, e0.elapsed_time(e1), tokens_per_step * e2e_steps)

    # ---- decode: N=256, H=16, D=128, 1000 steps in place
    dec = None
    if not args.no_decode:
        wd = WORKLOADS[DECODE_WORKLOAD]
        steps_d = args.decode_steps
        y = make_decode_inputs(wd.B, wd.H, wd.D, steps=steps_d + 10, device=dev, device_rng=True,
                               seed=100 + rank)
        S, R = y["S"], y["R"]
        od = torch.empty(wd.B, wd.H, wd.D, dtype=torch.bfloat16, device=dev)

        def dstep(i):
            rdn.rdn_decode_step(y["q"][i], y["k"][i], y["v"][i], y["g"][i], y["beta"][i],
                                y["gamma"][i], S, R, clip=wd.clip, out=od)

        for i in range(10):
            dstep(i)
        torch.cuda.synchronize()
        barrier(dist)
        with rdn.LaunchTimer(capacity=steps_d + 8) as ltd:
            e0.record(stream)
            for i in range(steps_d):
                dstep(10 + i)
            e1.record(stream)
            torch.cuda.synchronize()
        barrier(dist)
        tdec = max_over_ranks(dist, e0.elapsed_time(e1))
        heads = wd.B * wd.H
        nbytes = decode_bytes_per_head(wd.D) * heads
        gbs = sum_over_ranks(dist, nbytes * steps_d) / (tdec * 1e-3) / 1e9
        kd = ltd.summary().get("decode", (0, 0.0, 0.0))
        kern_gbs = nbytes / (kd[2] * 1e-3) / 1e9 if kd[2] > 0 else None
        dec = {"workload": wd.name, "value": gbs, "unit": "GB/s", "steps": steps_d,
               "us_per_step": tdec * 1e3 / steps_d, "bytes_per_step": nbytes,
               "frac_of_hbm_peak": gbs / peaks["hbm"], "hbm_peak_gbs": peaks["hbm"],
               "kernel_mean_us": kd[2] * 1e3, "kernel_gbs": kern_gbs,
               "state_bytes": 2 * S.numel() * 4,
               "l2": "no flush: 1.07 GB of state per step, larger than L2"}
        del y, S, R

    # ---- RLA fwd+bwd on the same workload (rla_fwd -> rla_bwd, chunk states
    # and records reused as in the RDN step)
    rla = None
    if not args.no_rla:
        wsr = torch.empty(rdn.workspace_bytes("rla_fwd", B, T, H, D, save_for_bwd=True),
                          dtype=torch.uint8, device=dev)

        def rstep(inp):
            _, _, _, Sc_, Rc_ = rdn.rla_fwd(*(inp[n] for n in names), clip=w.clip,
                                            return_chunk_states=True, out=o, workspace=wsr,
                                            save_for_bwd=True)
            rdn.rla_bwd(*(inp[n] for n in names), inp["dO"], clip=w.clip, S_chunks=Sc_,
                        R_chunks=Rc_, workspace=wsb, out=grads, fwd_workspace=wsr,
                        fwd_saved=True)

        rsteps = max(1, args.rla_steps)
        rstep(x)
        torch.cuda.synchronize()
        barrier(dist)
        with rdn.LaunchTimer() as ltr:
            e0.record(stream)
            for _ in range(rsteps):
                rstep(x)
            e1.record(stream)
            torch.cuda.synchronize()
        barrier(dist)
        tr, rval = aggregate(dist, e0.elapsed_time(e1), tokens_per_step * rsteps)
        rla = {"workload": w.name.replace("rdn_", "rla_"), "value": rval, "unit": "tokens/s",
               "steps": rsteps, "ms_per_step": tr / rsteps,
               "path": "tensor-core kernels as the RDN step (hi + lo copies of S where "
                       "RLA's uncontracted state needs them; identity T matrices)",
               "kernels": {k: {"launches": n, "mean_ms": m}
                           for k, (n, t, m) in ltr.summary().items()}}
        del wsr

    # ---- forward-only workloads (RDN forward, B=8 T=2048, and the long
    # context B=2 T=16384 with initial states and final states returned):
    # tokens/s and the forward's algorithmic flop rate against the tensor peak
    fwd = None
    if not args.no_forward:
        fwd = {}
        for wname in ("rdn_fwd_bf16_B8H16T2048D128", "rdn_fwd_bf16_B2H16T16384D128_state"):
            wf = WORKLOADS[wname]
            xf = make_workload_inputs(wf, device=dev, device_rng=True, seed=rank)
            of = torch.empty(wf.B, wf.T, wf.H, wf.D, dtype=torch.bfloat16, device=dev)
            wsff = torch.empty(rdn.workspace_bytes("rdn_fwd", wf.B, wf.T, wf.H, wf.D),
                               dtype=torch.uint8, device=dev)
            ret = wf.nonzero_state

            def fwd_step():
                rdn.rdn_fwd(*(xf[n] for n in names), clip=wf.clip, S0=xf["S0"], R0=xf["R0"],
                            return_final_state=ret, out=of, workspace=wsff)

            for _ in range(3):
                fwd_step()
            torch.cuda.synchronize()
            barrier(dist)
            fsteps = max(3, args.steps)
            e0.record(stream)
            for _ in range(fsteps):
                fwd_step()
            e1.record(stream)
            torch.cuda.synchronize()
            barrier(dist)
            tfw, fvals = aggregate(dist, e0.elapsed_time(e1), wf.B * wf.T * fsteps)
            ms_f = tfw / fsteps
            tfl = fl["fwd"] * wf.B * wf.T * wf.H / (ms_f * 1e-3) / 1e12
            fwd[wname] = {"value": fvals, "unit": "tokens/s", "ms_per_step": ms_f,
                          "steps": fsteps, "tflops": tfl, "frac_of_bf16_peak": tfl / peak,
                          "states": "S0, R0 in, S_T, R_T out" if ret else "zero, not returned"}
            del xf, of, wsff

    # ---- the paper's variants (variant_flags, fp32 chunk kernels) on the
    # bench workload: RDN fwd+bwd with each flag, as the RDN step above
    var = None
    if not args.no_variants:
        var = {"workload": w.name, "steps": 1, "flags": {},
               "path": "tensor-core kernels for every flag (runtime modes of the generic "
                       "kernel instances)"}
        wsbv_ = torch.empty(rdn.workspace_bytes("rdn_bwd", B, T, H, D,
                                                variant_flags=rdn.TANH_RESIDUAL),
                            dtype=torch.uint8, device=dev)
        # (the tanh residual saves a 16-bit derivative per element, not a mask bit)
        wsfv_ = torch.empty(rdn.workspace_bytes("rdn_fwd", B, T, H, D, save_for_bwd=True,
                                                variant_flags=rdn.TANH_RESIDUAL),
                            dtype=torch.uint8, device=dev)
        for fname, fl in (("decayed_residual", rdn.DECAYED_RESIDUAL),
                          ("plain_combine", rdn.PLAIN_COMBINE),
                          ("tanh_residual", rdn.TANH_RESIDUAL),
                          ("stateless_aux", rdn.STATELESS_AUX)):
            def fstep(inp):  # (the RDN step's options: chunk states, saved intermediates)
                _, _, _, Sc_, Rc_ = rdn.rdn_fwd(*(inp[n] for n in names), clip=w.clip,
                                                return_chunk_states=True, out=o, workspace=wsfv_,
                                                save_for_bwd=True, variant_flags=fl)
                rdn.rdn_bwd(*(inp[n] for n in names), inp["dO"], clip=w.clip, S_chunks=Sc_,
                            R_chunks=Rc_, workspace=wsbv_, out=grads, fwd_workspace=wsfv_,
                            fwd_saved=True, variant_flags=fl)
            fstep(x)
            torch.cuda.synchronize()
            barrier(dist)
            e0.record(stream)
            fstep(x)
            e1.record(stream)
            torch.cuda.synchronize()
            barrier(dist)
            tf, fval = aggregate(dist, e0.elapsed_time(e1), tokens_per_step)
            var["flags"][fname] = {"value": fval, "unit": "tokens/s", "ms_per_step": tf}
        del wsbv_, wsfv_

    # ---- packed variable-length sequences: the same B*T tokens per head as
    # one packed row of seeded log-uniform lengths in [64, 8192] (the last one
    # cut to fill the row), RDN fwd+bwd exactly as the step above
    vl = None
    if not args.no_varlen:
        lens = packed_lengths(B * T)
        cu = torch.tensor(np.concatenate([[0], np.cumsum(lens)]), dtype=torch.int32, device=dev)
        N = len(lens)
        xv = {n: x[n].view(1, B * T, *x[n].shape[2:]) for n in names + ("dO",)}
        ov = o.view(1, B * T, H, D)
        wsfv = torch.empty(rdn.workspace_bytes("rdn_fwd", 1, B * T, H, D, save_for_bwd=True,
                                               cu_seqlens=cu), dtype=torch.uint8, device=dev)
        wsbv = torch.empty(rdn.workspace_bytes("rdn_bwd", 1, B * T, H, D, cu_seqlens=cu),
                           dtype=torch.uint8, device=dev)
        gv = {n: (t.view(1, B * T, *t.shape[2:]) if n not in ("dS0", "dR0") else
                  torch.empty(N, H, D, D, device=dev)) for n, t in grads.items()}

        def vstep(inp):
            _, _, _, Sc_, Rc_ = rdn.rdn_fwd(*(inp[n] for n in names), clip=w.clip,
                                            return_chunk_states=True, out=ov, workspace=wsfv,
                                            save_for_bwd=True, cu_seqlens=cu)
            rdn.rdn_bwd(*(inp[n] for n in names), inp["dO"], clip=w.clip, S_chunks=Sc_,
                        R_chunks=Rc_, workspace=wsbv, out=gv, fwd_workspace=wsfv,
                        fwd_saved=True, cu_seqlens=cu)

        vsteps = max(1, args.steps)
        for _ in range(3):
            vstep(xv)
        torch.cuda.synchronize()
        barrier(dist)
        with rdn.LaunchTimer() as ltv:
            e0.record(stream)
            for _ in range(vsteps):
                vstep(xv)
            e1.record(stream)
            torch.cuda.synchronize()
        barrier(dist)
        tv, vval = aggregate(dist, e0.elapsed_time(e1), tokens_per_step * vsteps)
        vl = {"workload": f"rdn_fwd_bwd_packed_bf16_N{N}_T{B * T}H{H}D{D}", "value": vval,
              "unit": "tokens/s", "steps": vsteps, "ms_per_step": tv / vsteps,
              "num_seqs": N, "lengths": {"min": int(min(lens)), "max": int(max(lens)),
                                         "mean": float(np.mean(lens))},
              "chunks_per_head": int(sum((L + C - 1) // C for L in lens)),
              "vs_fixed_length": vval / value,
              "kernels": {k: {"launches": n, "mean_ms": m}
                          for k, (n, t, m) in ltv.summary().items()}}
        del wsfv, wsbv, gv

    # ---- q, k prologue (SiLU + L2 norm) and its backward on the bench
    # workload's q, k: algorithmic bytes = each element read and written once
    # (the backward also reads dy), against the measured HBM peak
    pro = None
    if not args.no_prologue:
        dq_, dk_ = torch.empty_like(x["q"]), torch.empty_like(x["k"])
        yq_, yk_ = torch.empty_like(x["q"]), torch.empty_like(x["k"])

        # each direction timed in its own loop (as a layer's forward and its
        # backward run apart in a training step)
        pro_fwd = lambda: rdn.qk_prologue(x["q"], x["k"], out=(yq_, yk_))
        pro_bwd = lambda: rdn.qk_prologue_bwd(x["q"], x["k"], x["dO"], x["dO"], out=(dq_, dk_))
        psteps = 20
        kp = {}
        for fn_ in (pro_fwd, pro_bwd):
            for _ in range(3):
                fn_()
            torch.cuda.synchronize()
            with rdn.LaunchTimer(capacity=psteps + 8) as ltp:
                for _ in range(psteps):
                    fn_()
                torch.cuda.synchronize()
            kp.update(ltp.summary())
        elem = x["q"].numel() * x["q"].element_size()  # bytes of one tensor
        fwd_bytes, bwd_bytes = 4 * elem, 6 * elem
        mf, mb = kp["qk_prologue"][2], kp["qk_prologue_bwd"][2]
        pro = {"workload": "qk_prologue_bf16_B8T4096H16D128 (q and k)",
               "fwd_ms": mf, "fwd_gbs": fwd_bytes / (mf * 1e-3) / 1e9,
               "bwd_ms": mb, "bwd_gbs": bwd_bytes / (mb * 1e-3) / 1e9,
               "fwd_frac_of_hbm_peak": fwd_bytes / (mf * 1e-3) / 1e9 / peaks["hbm"],
               "bwd_frac_of_hbm_peak": bwd_bytes / (mb * 1e-3) / 1e9 / peaks["hbm"],
               "bytes": {"fwd": fwd_bytes, "bwd": bwd_bytes}, "launches": psteps,
               "l2": "no flush: 268 MB of q, k per pass, larger than L2"}
        del dq_, dk_, yq_, yk_

        # the same map inside the library (RDN_FLAG_QK_NORM): the RDN step
        # above with q, k taken as raw projections -- the forward's per-chunk
        # pass normalises the rows it loads; the backward leaves dq, dk in
        # fp32 and one streaming pass applies the map's Jacobian
        wsfq = torch.empty(rdn.workspace_bytes("rdn_fwd", B, T, H, D, save_for_bwd=True,
                                               qk_norm=True), dtype=torch.uint8, device=dev)

        def qstep(inp):
            _, _, _, Sc_, Rc_ = rdn.rdn_fwd(*(inp[n] for n in names), clip=w.clip,
                                            return_chunk_states=True, out=o, workspace=wsfq,
                                            save_for_bwd=True, qk_norm=True)
            rdn.rdn_bwd(*(inp[n] for n in names), inp["dO"], clip=w.clip, S_chunks=Sc_,
                        R_chunks=Rc_, workspace=wsb, out=grads, fwd_workspace=wsfq,
                        fwd_saved=True, qk_norm=True)

        qsteps = max(3, args.steps)
        for _ in range(3):
            qstep(x)
        torch.cuda.synchronize()
        barrier(dist)
        with rdn.LaunchTimer() as ltq:
            e0.record(stream)
            for _ in range(qsteps):
                qstep(x)
            e1.record(stream)
            torch.cuda.synchronize()
        barrier(dist)
        tq, qval = aggregate(dist, e0.elapsed_time(e1), tokens_per_step * qsteps)
        pro["fused_step"] = {
            "workload": w.name + " with RDN_FLAG_QK_NORM", "value": qval, "unit": "tokens/s",
            "steps": qsteps, "ms_per_step": tq / qsteps,
            "overhead_ms_vs_step": tq / qsteps - ms_per_step,
            "separate_passes_ms": mf + mb,
            "kernels": {k: {"launches": n, "mean_ms": m} for k, (n, t, m) in ltq.summary().items()}}
        del wsfq

    cpu = None
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        cpu = time_oracle_sample(target_s=args.cpu_seconds)
        cpu["cpu_model"] = cpu_model()
        cpu["configs"] = time_oracle_configs()

    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": ws,
                "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_per_step,
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
                "dtype": "bf16", "data": "synthetic", "config": _config(w),
                "roofline": roof, "step_tflops": step_tflops,
                "step_frac_of_bf16_peak": step_tflops / peak,
                "step_tflops_dense_tiles": step_tflops_dense,
                "step_frac_of_bf16_peak_dense_tiles": step_tflops_dense / peak,
                "cpu_baseline": cpu,
                "e2e": {"value": e2e_val, "unit": "tokens/s", "h2d_bytes_per_step": h2d,
                        "d2h_bytes_per_step": d2h, "steps": e2e_steps,
                        "copies": "all inputs in from pinned host memory and the output o "
                                  "back, every step, on their own streams, overlapped with "
                                  "the compute of the neighbouring steps (two device buffer "
                                  "sets); the gradients stay on the device; the timed "
                                  "region includes the unoverlapped first input copy and "
                                  "last output read"},
                "gpu_launches": lt.launches,
                "kernels": {k: {"launches": n, "total_ms": t, "mean_ms": m,
                                "share": t / sum(v[1] for v in kern.values())}
                            for k, (n, t, m) in kern.items()},
                "clocks": clk.summary(), "decode": dec, "rla": rla, "prologue": pro,
                "varlen": vl, "variants": var, "forward": fwd}
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()
    return 0


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    # (default: 60 timed steps for this arm, ~0.2 s, so that the 50 ms clock
    # samples fall inside the timed region; 10 oracle steps for the reference)
    ap.add_argument("--steps", type=int, default=None)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--decode-steps", type=int, default=1000)
    ap.add_argument("--no-decode", action="store_true")
    ap.add_argument("--rla-steps", type=int, default=3)
    ap.add_argument("--no-rla", action="store_true")
    ap.add_argument("--no-prologue", action="store_true")
    ap.add_argument("--no-varlen", action="store_true")
    ap.add_argument("--no-variants", action="store_true")
    ap.add_argument("--no-forward", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--profile", action="store_true",
                    help="for profiler captures: the timed step only -- no clock sampler, "
                         "end-to-end leg, CPU baseline or other workloads")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--B", type=int, default=0, help="override B (profiling captures only)")
    ap.add_argument("--T", type=int, default=0, help="override T (profiling captures only)")
    args = ap.parse_args(argv)
    if args.steps is None:
        args.steps = 60 if args.impl == "ours" else 10
    if args.profile:
        args.no_decode = args.no_rla = args.no_prologue = args.no_varlen = True
        args.no_variants = args.no_forward = args.no_cpu_baseline = True
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
