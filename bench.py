#!/usr/bin/env python
"""Throughput of the cache-aware routing + expert-residency step on GB300.

Metric: stream-token-layer route+cache decisions per second.  One step is
one full pass of the path (router heads, Top-K, refinement, access,
retention, accounting) over the whole workload: every stream, token and
layer, from a cold cache state.  Inputs are synthetic (seeded AR(1) hidden
states and N(0, 1/d) router weights) with the shapes of the named backbone
and already resident in HBM when the timed region starts; the hidden states
(12.9 GB for the Qwen3-30B shape) are far larger than L2, so no flush is
needed between steps.

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]
Multi-GPU (torchrun): streams are independent, every rank runs its own
streams (weak scaling), no data-path collective; timing is the max over ranks.
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
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import crc_synth as S  # noqa: E402

METRIC = "stream-token-layer route+cache decisions/sec"
UNIT = "decisions/s"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default=S.QWEN3_30B.name, choices=sorted(S.WORKLOADS))
    ap.add_argument("--chunk", type=int, default=0, help="tokens per workspace chunk (0 = auto)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--capacity", type=int, default=0,
                    help="cache slots C per (stream, layer) (0 = the workload's; the sweep takes 16/32/64/96)")
    ap.add_argument("--proactive", type=int, default=None,
                    help="proactive-load bound R (default: the workload's; the large shape takes 2 or 8)")
    ap.add_argument("--tokens", type=int, default=0,
                    help="override T (a smaller case, e.g. for an ncu capture)")
    ap.add_argument("--only", choices=["fused", "pair", "router", "scan", "loss", "transfer"],
                    default="fused",
                    help="fused: crc_route_and_cache as one fused kernel (default); pair: "
                         "crc_route_scores then crc_cache_scan; router / scan: one part alone; "
                         "loss: the soft Top-B coverage losses and their gradient "
                         "(crc_cache_loss) on the router's probabilities; transfer: one "
                         "stream's expert copies (crc_transfer_plan / crc_transfer_replay)")
    ap.add_argument("--top-b", type=int, default=0,
                    help="with --only loss: B of the soft Top-B loss (0 = the paper's: 20 for "
                         "N = 128, 8 for N = 32)")
    ap.add_argument("--tau", type=float, default=0.0,
                    help="with --only loss: temperature (0 = the paper's: 0.03 for N = 128, "
                         "0.05 for N = 32)")
    ap.add_argument("--policy", choices=["method", "lru", "lfu", "lrfu", "spatio_lru"],
                    default="method",
                    help="with --only scan: time a comparison policy's scan "
                         "(crc_cache_scan_policy, LRFU lambda 0.5) instead of the method's")
    return ap.parse_args()


# --------------------------------------------------------------------------- #
def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return d, "measured"
    except (OSError, ValueError):
        return dict(FALLBACK_PEAKS), "fallback"


def rank_seed(rank: int) -> int:
    """Seed of a rank's synthetic hidden states: under torchrun every rank runs
    its own B streams (weak scaling), so no two ranks replay the same data."""
    return 1000 * rank


def max_over_ranks(x: float, world: int, device=None) -> float:
    """The slowest rank's time: the job ends when the last rank does
    (all_reduce MAX on the rank's device; one process: x itself)."""
    if world <= 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(units_per_rank: int, world: int, ms_per_step: float) -> float:
    """Whole-job throughput: the units every rank processed over the slowest
    rank's time per step."""
    return units_per_rank * world / (ms_per_step / 1000.0)


def algorithmic(w, units: int, heads: int):
    """Algorithmic flops and HBM bytes of the fused step for `units` decisions:
    2*d*H*N flops per unit; bf16 hidden state read once (2d bytes), the
    weights once per pass, trace-free accounting."""
    flops = 2.0 * w.d * heads * w.N * units
    bytes_ = 2.0 * w.d * units + 2.0 * w.L * heads * w.N * w.d
    return flops, bytes_


def workload_config(w, chunk=None):
    cfg = {"workload": f"{w.name}: L={w.L} N={w.N} K={w.K} d={w.d} C={w.C} R={w.R} "
                       f"B={w.B} T={w.T}",
           "L": w.L, "N": w.N, "K": w.K, "d": w.d, "C": w.C, "R": w.R,
           "streams": w.B, "tokens": w.T, "expert_bytes": w.expert_bytes,
           "rho_t": w.rho_t, "rho_l": w.rho_l,
           "l2": "inputs larger than L2 (hidden states %.1f GB per step), no flush"
                 % (2.0 * w.units * w.d / 1e9)}
    if chunk:
        cfg["chunk_tokens"] = chunk
    return cfg


class ClockSampler:
    """nvidia-smi samples (every 20 ms) of SM clock, power and throttle reasons
    during the timed region: the context waits for the first sample before the
    region starts, and the summary keeps the samples time-stamped inside it."""
    Q = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    NAMES = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]

    def __init__(self, gpu_id: str):
        self.gpu_id = gpu_id
        self.proc = None
        self.lines = []
        self.t0 = self.t1 = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", self.gpu_id, f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "20"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
            deadline = time.time() + 5.0
            while not self.lines and time.time() < deadline and self.proc.poll() is None:
                time.sleep(0.01)
        except OSError:
            self.proc = None
        self.t0 = time.time()
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *a):
        self.t1 = time.time()
        time.sleep(0.05)
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.t.join(timeout=2)

    @staticmethod
    def _stamp(text: str):
        import datetime
        try:
            return datetime.datetime.strptime(text.strip(), "%Y/%m/%d %H:%M:%S.%f").timestamp()
        except ValueError:
            return None

    def summary(self):
        sm, mx, pw, reasons = [], [], [], set()
        for ln in self.lines:
            parts = [x.strip() for x in ln.split(",")]
            if len(parts) < 9:
                continue
            ts = self._stamp(parts[0])
            if ts is None or self.t0 is None or not (self.t0 - 0.03 <= ts <= self.t1 + 0.03):
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
                pw.append(float(parts[3]))
            except ValueError:
                continue
            for n, v in zip(self.NAMES, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0,
                    "window_s": None if self.t0 is None else round(self.t1 - self.t0, 3)}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx),
                "sm_min_mhz": min(sm), "power_w": statistics.median(pw),
                "reasons": sorted(reasons), "samples": len(sm),
                "window_s": round(self.t1 - self.t0, 3)}


def gpu_id_for_smi(torch, dev: int) -> str:
    try:
        u = str(torch.cuda.get_device_properties(dev).uuid)
        return u if u.startswith("GPU-") else "GPU-" + u
    except Exception:
        vis = os.environ.get("CUDA_VISIBLE_DEVICES")
        if vis:
            return vis.split(",")[dev]
        return str(dev)


# The sources each profiled kernel is built from: a committed traffic figure
# stands only while none of them has changed.
KERNEL_SOURCES = {
    "fused": ["fused.cu", "fused.cuh", "fused_launch.cuh", "fused_n16.cu", "fused_n32.cu",
              "fused_n64.cu", "fused_n128.cu", "router_gemm.cuh", "cache_scan.cuh",
              "crc_device.cuh"],
    "router": ["router.cu", "router_gemm.cuh", "crc_device.cuh"],
    "scan": ["scan.cu", "scan_traced.cu", "scan_launch.cuh", "cache_scan.cuh", "crc_device.cuh"],
    "policy": ["policy.cu", "policy_launch.cuh", "policy_lru.cu", "policy_lfu.cu",
               "policy_lrfu.cu", "policy_spatio.cu", "policy_scan.cuh", "cache_scan.cuh",
               "crc_device.cuh"],
    "loss": ["loss.cu", "cache_scan.cuh", "crc_device.cuh"],
}


def kernel_family(kernel: str) -> str:
    for fam in ("policy", "fused", "router", "loss"):
        if fam in kernel:
            return fam
    return "scan"


def source_hash(kernel: str) -> str:
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2609_04895_gb300", "csrc")
    for f in sorted(KERNEL_SOURCES[kernel_family(kernel)]):
        with open(os.path.join(csrc, f), "rb") as fh:
            h.update(f.encode() + fh.read())
    return h.hexdigest()[:16]


def committed_traffic(kernel: str, workload: str):
    """DRAM bytes per unit from a committed ncu capture, if taken on the current sources."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            d = json.load(f)
    except (OSError, ValueError):
        return None, None
    e = d.get(kernel, {}).get(workload)
    if not e or e.get("src_sha") != source_hash(kernel):
        return None, None
    return e.get("dram_bytes_per_unit"), e.get("source")


# --------------------------------------------------------------------------- #
def cpu_oracle_sample(w, seconds: float):
    """Times the CPU oracle (as it stands) on a bounded sample of workload w:
    the first streams and tokens, all layers, fp64 router heads + scan."""
    import numpy as np

    import oracle
    oracle.build()
    threads = oracle.default_threads()
    Wb = S.weights(w, seed=0)

    def run(nb, nt):
        h = S.hidden(w.with_(B=nb), seed=0, T=nt)
        t0 = time.perf_counter()
        res = oracle.run(h, Wb, w.N, w.K, w.C, w.R, margins=False, nthreads=threads)
        dt = time.perf_counter() - t0
        return dt, res

    pilot_t = min(8, w.T)
    dt, _ = run(1, pilot_t)
    rate = (pilot_t * w.L) / max(dt, 1e-6)
    want_units = rate * seconds
    nt = int(min(w.T, max(pilot_t, want_units // w.L)))
    nb = int(min(w.B, max(1, want_units // (w.L * nt))))
    dt, res = run(nb, nt)
    units = nb * nt * w.L
    del res, np
    return {"value": units / dt, "unit": UNIT, "cores": threads, "kind": "oracle",
            "sample": f"{nb} stream(s) x {nt} tokens x {w.L} layers = {units} decisions "
                      f"(fp64 router heads + literal scan), {dt:.1f} s wall"}, units, dt


def policy_report(P, stats, p, m):
    """Hit, AdjHit, Load/token (Sec. 4.1) and the overlap model's exposed
    loading cost per decode token at no and at full prefetch overlap, in
    expert transfers (multiply by the seconds per expert transfer)."""
    return {"hit": m["hit"], "adj_hit": m["adj_hit"],
            "load_MB_per_token": m["load_per_token_bytes"] / 1e6,
            "t_load_transfers_per_token": {"eta0": P.load_time(stats, p, 1.0, 0.0),
                                           "eta1": P.load_time(stats, p, 1.0, 1.0)}}


def workload_of(args):
    w = S.WORKLOADS[args.workload]
    if args.tokens:
        w = w.with_(T=args.tokens)
    if args.capacity:
        w = w.with_(C=args.capacity)
    if args.proactive is not None:
        w = w.with_(R=args.proactive)
    return w


LOSS_METRIC = "stream-token-layer coverage-loss units/sec (forward + gradient)"
LOSS_UNIT = "units/s"


def loss_settings(args, w):
    """(B, tau) of the soft Top-B loss: the paper's main settings by backbone."""
    top_b = args.top_b or (20 if w.N >= 128 else 8)
    tau = args.tau or (0.03 if w.N >= 128 else 0.05)
    return min(top_b, w.N), tau


def loss_workload_config(w, top_b, tau):
    cfg = workload_config(w)
    cfg.update({"top_b": top_b, "tau": tau, "w_T": 1.0, "w_ST": 1.0,
                "inputs": "router probabilities [B][T][L][3][N] fp32 from the router GEMM on "
                          "the synthetic hidden states (untimed)",
                "l2": "inputs larger than L2 (probabilities %.1f GB per step), no flush"
                      % (12.0 * w.N * w.units / 1e9)})
    return cfg


def loss_oracle_sample(w, top_b, tau, seconds):
    """Times oracle.cache_loss (as it stands, one thread) on the first streams
    of the workload (whole sequences): synthetic distributions of its shape."""
    import oracle
    oracle.build()
    pilot = S.distributions(1, min(64, w.T), w.L, w.N, seed=0)
    t0 = time.perf_counter()
    oracle.cache_loss(pilot, top_b, tau)
    rate = pilot.shape[1] * w.L / max(time.perf_counter() - t0, 1e-6)     # units/s
    nb = int(max(1, min(w.B, rate * seconds // (w.T * w.L))))
    nt = w.T if nb > 1 or rate * seconds >= w.T * w.L else int(max(8, rate * seconds // w.L))
    pb = S.distributions(nb, nt, w.L, w.N, seed=0)
    t0 = time.perf_counter()
    oracle.cache_loss(pb, top_b, tau)
    dt = time.perf_counter() - t0
    units = nb * nt * w.L
    return {"value": units / dt, "unit": LOSS_UNIT, "cores": 1, "kind": "oracle",
            "sample": f"{nb} stream(s) x {nt} tokens x {w.L} layers = {units} units (fp64 "
                      f"losses and logit gradient), {dt:.1f} s wall"}, units, dt


def run_reference_loss(args, w):
    import oracle
    oracle.build()
    top_b, tau = loss_settings(args, w)
    budget = max(1.0, min(6.0, 150.0 / max(1, args.steps + args.warmup)))
    _, units, dt = loss_oracle_sample(w, top_b, tau, budget)
    nb = max(1, units // (w.T * w.L))
    nt = units // (nb * w.L)
    pb = S.distributions(nb, nt, w.L, w.N, seed=0)
    for _ in range(args.warmup):
        oracle.cache_loss(pb, top_b, tau)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        oracle.cache_loss(pb, top_b, tau)
    dt = time.perf_counter() - t0
    value = units * args.steps / dt
    line = {
        "metric": LOSS_METRIC, "value": value, "unit": LOSS_UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000 * dt / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic",
        "config": dict(loss_workload_config(w, top_b, tau),
                       inputs="seeded synthetic distributions of the same shape (host)"),
        "impl": "reference",
        "cpu_baseline": {"value": value, "unit": LOSS_UNIT, "cores": 1, "kind": "oracle",
                         "sample": f"{nb} stream(s) x {nt} tokens x {w.L} layers = {units} "
                                   f"units per step"},
        "e2e": {"value": value, "unit": LOSS_UNIT, "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def run_loss(args, P, C, w, p, dev, stream, rank, world):
    """Times crc_cache_loss over the whole workload: per step, both coverage
    losses at every (stream, token, layer), their means and the gradient with
    respect to the three heads' logits.  The probabilities come from the
    router GEMM on the synthetic hidden states (untimed)."""
    import torch
    import torch.distributed as dist
    top_b, tau = loss_settings(args, w)
    Wd = P.synth_weights(w.L, w.N, w.d, seed=0, device=dev)
    hd, _ = P.synth_hidden(w.B, w.T, w.L, w.d, seed=rank_seed(rank), rho_t=w.rho_t,
                           rho_l=w.rho_l, device=dev)
    probs = P.route_scores(p, hd, Wd, heads=3)
    del hd, Wd
    loss = torch.empty((w.B, w.T, w.L, 2), dtype=torch.float32, device=dev)
    means = torch.empty(2, dtype=torch.float64, device=dev)
    grad = torch.empty_like(probs)
    ws_bytes = C.crc_loss_workspace_bytes(p, w.T)
    ws = torch.empty(max(ws_bytes, 256), dtype=torch.uint8, device=dev)

    def step(src=probs):
        C.crc_cache_loss(p, src.data_ptr(), w.T, 3, top_b, tau, 1.0, 1.0, loss.data_ptr(),
                         means.data_ptr(), grad.data_ptr(), ws.data_ptr(), ws.numel(), stream)

    for _ in range(max(3, args.warmup)):
        step()
    torch.cuda.synchronize()
    assert C.crc_device_error() == 0
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(gpu_id_for_smi(torch, dev.index or 0)) as clk:
        C.crc_profile_begin()
        n0 = C.crc_launch_count()
        e0.record(stream)
        for _ in range(args.steps):
            step()
        e1.record(stream)
        torch.cuda.synchronize()
        launches = C.crc_launch_count() - n0
        kt = C.crc_profile_end()
    ms = max_over_ranks(e0.elapsed_time(e1), world, dev)
    if world > 1:
        dist.barrier()
    ms_per_step = ms / args.steps
    value = job_rate(w.units, world, ms_per_step)
    L_T, L_ST = (float(x) for x in means.cpu())

    # roofline of the loss kernel: probabilities read once, gradient and losses written once
    pk, pk_src = peaks()
    per_unit = 24.0 * w.N + 8.0
    avg_ms = kt["loss"]["ms"] / max(1, kt["loss"]["launches"])
    achieved = per_unit * w.units / (avg_ms / 1000.0) / 1e9
    if w.N in (16, 32) and top_b <= 16:         # short rows: 16 elements per lane
        kp = 2 if top_b <= 2 else 4 if top_b <= 4 else 8 if top_b <= 8 else 16
        kname = f"cache_loss_rows_kernel<{w.N // 16},{kp}>"
    else:
        V = 1 if w.N <= 32 else 2 if w.N <= 64 else 4 if w.N <= 128 else 8
        kname = f"cache_loss_kernel<{V}>"
    tr, _ = committed_traffic(kname, w.name)
    roof = {"bound": "hbm", "achieved": achieved, "peak": pk["hbm_gbs"], "unit": "GB/s",
            "frac": achieved / pk["hbm_gbs"], "traffic": None if tr is None else tr * w.units,
            "kernel": kname, "peak_source": f"{pk_src} (copy)", "avg_launch_ms": avg_ms,
            "launches": kt["loss"]["launches"],
            "share_of_step": kt["loss"]["ms"] / ms if ms else None,
            "bytes_per_unit": per_unit}
    kernels = {k: {"launches": v["launches"], "ms_per_step": v["ms"] / args.steps}
               for k, v in kt.items() if v["launches"]}

    e2e = None
    if not args.no_e2e:
        # the public call from pinned (huge-page) host probabilities; the means come back
        host, host_mem = pinned_host(P, probs.shape, torch.float32)
        host.copy_(probs)
        out = torch.empty(2, dtype=torch.float64, pin_memory=True)
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        f0.record(stream)
        for _ in range(args.steps):
            probs.copy_(host, non_blocking=True)
            step()
            out.copy_(means, non_blocking=True)
        f1.record(stream)
        torch.cuda.synchronize()
        ems = max_over_ranks(f0.elapsed_time(f1), world, dev)
        e2e = {"value": job_rate(w.units, world, ems / args.steps), "unit": LOSS_UNIT,
               "h2d_bytes_per_step": int(probs.numel() * 4), "d2h_bytes_per_step": 16,
               "ms_per_step": ems / args.steps, "host_memory": host_mem}
        del host

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:
        cpu, _, _ = loss_oracle_sample(w, top_b, tau, args.cpu_seconds)
    if rank == 0:
        line = {
            "metric": LOSS_METRIC, "value": value, "unit": LOSS_UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": max(3, args.warmup), "ms_per_step": ms_per_step,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic", "config": dict(loss_workload_config(w, top_b, tau), path="loss"),
            "roofline": roof, "kernels": kernels, "cpu_baseline": cpu, "e2e": e2e,
            "gpu_launches": int(launches), "clocks": clk.summary(),
            "losses": {"L_T": L_T, "L_ST": L_ST},
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()
    return 0


TRANSFER_METRIC = "expert bytes moved per second (host pool -> HBM cache slots)"


def run_transfer(args, P, C, w, p, dev, stream, rank, world):
    """Replays the expert copies of stream 0: the router and the scan run once
    with cache traces (untimed), crc_transfer_plan turns the stream's cache
    sets into copies, and each timed step enqueues all of them
    (crc_transfer_replay, one cudaMemcpyAsync of expert_bytes per copy) from a
    pinned host pool to a device cache of L x C slots.  The pool holds 64
    expert images, copy (l, e) reading image (l N + e) mod 64: the bytes and
    sizes are the real ones, the images repeat."""
    import numpy as np
    import torch
    T = args.tokens or 256
    w = w.with_(T=T)
    Wd = P.synth_weights(w.L, w.N, w.d, seed=0, device=dev)
    hd, _ = P.synth_hidden(w.B, w.T, w.L, w.d, seed=rank_seed(rank), rho_t=w.rho_t,
                           rho_l=w.rho_l, device=dev)
    st = P.State(p, device=dev)
    tr = P.Trace.alloc(p, w.T, device=dev, caches=True)
    P.route_and_cache(p, hd, Wd, st, tr)
    stats = st.read(want_chain_counters=True)
    assert stats["error"] == 0, stats
    del hd, Wd
    mid = tr.cache_mid[0].cpu().numpy()
    aft = tr.cache_after[0].cpu().numpy()
    t0 = time.perf_counter()
    plan, _ = P.transfer_plan(p, mid, aft)
    plan_ms = 1000 * (time.perf_counter() - t0)
    eb = int(p.expert_bytes)
    counters = stats["chain_counters"].reshape(w.B, w.L, 3)[0]
    assert len(plan) == int(counters[:, 1].sum() + counters[:, 2].sum())
    pool_n = 64
    pool = torch.empty(pool_n * eb, dtype=torch.uint8, pin_memory=True)
    pool.fill_(7)
    slots = torch.empty((w.L, w.C, eb), dtype=torch.uint8, device=dev)
    # the host link's copy rate: one pinned copy of the whole pool, best of 3
    big = slots.view(-1)[:pool.numel()]
    best = None
    for _ in range(3):
        a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a0.record(stream)
        big.copy_(pool, non_blocking=True)
        a1.record(stream)
        torch.cuda.synchronize()
        ms = a0.elapsed_time(a1)
        best = ms if best is None else min(best, ms)
    peak_gbs = pool.numel() / (best / 1000.0) / 1e9

    def step():
        C.crc_transfer_replay(p, plan.ctypes.data, len(plan), pool.data_ptr(), pool_n,
                              slots.data_ptr(), stream)

    for _ in range(max(3, args.warmup)):
        step()
    torch.cuda.synchronize()
    steps = args.steps
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(gpu_id_for_smi(torch, dev.index or 0)) as clk:
        e0.record(stream)
        for _ in range(steps):
            step()
        e1.record(stream)
        torch.cuda.synchronize()
    ms = e0.elapsed_time(e1)
    ms_per_step = ms / steps
    moved = len(plan) * eb
    value = moved / (ms_per_step / 1000.0)
    m = P.metrics({k: stats[k] for k in stats}, p)
    tok_ms = ms_per_step / T
    if rank == 0:
        line = {
            "metric": TRANSFER_METRIC, "value": value, "unit": "B/s", "n_gpus": world,
            "steps": steps, "warmup": max(3, args.warmup), "ms_per_step": ms_per_step,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "u8",
            "data": "synthetic",
            "config": dict(workload_config(w), path="transfer", stream=0,
                           copies_per_step=int(len(plan)), bytes_per_step=int(moved),
                           proactive_copies=int((plan["proactive"] == 1).sum()),
                           pool_images=pool_n, plan_ms=plan_ms),
            "roofline": {"bound": "c2c", "achieved": value / 1e9, "peak": peak_gbs,
                         "unit": "GB/s", "frac": value / 1e9 / peak_gbs, "traffic": None,
                         "kernel": "cudaMemcpyAsync host -> device (one per planned copy)",
                         "peak_source": "one pinned host -> device copy of the whole pool, "
                                        "measured in this run"},
            "transfer_ms_per_token": tok_ms,
            "load_model": {"hit": m["hit"], "adj_hit": m["adj_hit"],
                           "load_MB_per_token": m["load_per_token_bytes"] / 1e6},
            "cpu_baseline": None, "e2e": None, "gpu_launches": 0,
            "clocks": clk.summary(),
        }
        print(json.dumps(line), flush=True)
    return 0


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    w = workload_of(args)
    if args.only == "loss":
        return run_reference_loss(args, w)
    import oracle
    oracle.build()
    threads = oracle.default_threads()
    Wb = S.weights(w, seed=0)
    # one stream per host core (the oracle's scan runs a thread per stream,
    # its router heads a thread per core), as many tokens as make one step a
    # few seconds of oracle time
    ns = max(1, min(w.B, threads))
    h1 = S.hidden(w, seed=0, streams=range(ns), T=min(4, w.T))
    t0 = time.perf_counter()
    oracle.run(h1, Wb, w.N, w.K, w.C, w.R, margins=False, nthreads=threads)
    rate = ns * h1.shape[1] * w.L / max(time.perf_counter() - t0, 1e-6)
    budget = max(1.0, min(6.0, 150.0 / max(1, args.steps + args.warmup)))
    nt = int(min(w.T, max(4, rate * budget // (ns * w.L))))
    h = S.hidden(w, seed=0, streams=range(ns), T=nt)
    for _ in range(args.warmup):
        oracle.run(h, Wb, w.N, w.K, w.C, w.R, margins=False, nthreads=threads)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        oracle.run(h, Wb, w.N, w.K, w.C, w.R, margins=False, nthreads=threads)
    dt = time.perf_counter() - t0
    units = ns * nt * w.L
    value = units * args.steps / dt
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000 * dt / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": workload_config(w), "impl": "reference",
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle",
                         "sample": f"{ns} stream(s) x {nt} tokens x {w.L} layers = {units} "
                                   f"decisions per step of the workload named in config "
                                   f"(fp64 router heads + literal scan)"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# --------------------------------------------------------------------------- #
def main():
    args = parse_args()
    if args.impl == "reference":
        return run_reference(args)

    import torch
    import torch.distributed as dist

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl")

    from paper_2609_04895_gb300 import build as B_
    B_.build()
    import paper_2609_04895_gb300 as P
    C = P.crc

    w = workload_of(args)
    p = P.problem_of(w)
    heads = 3 if w.R > 0 else 2
    dev = torch.device("cuda", local)
    stream = torch.cuda.current_stream()
    if args.only == "loss":
        return run_loss(args, P, C, w, p, dev, stream, rank, world)
    if args.only == "transfer":
        return run_transfer(args, P, C, w, p, dev, stream, rank, world)
    if 2 * w.B * w.T * w.L * w.d > STREAM_BYTES:
        return run_streamed(args, P, C, w, p, heads, dev, stream, rank, world)

    # inputs, resident in HBM before timing (untimed generation)
    Wd = P.synth_weights(w.L, w.N, w.d, seed=0, device=dev)
    hd, _ = P.synth_hidden(w.B, w.T, w.L, w.d, seed=rank_seed(rank), rho_t=w.rho_t,
                           rho_l=w.rho_l, device=dev)
    chunk = args.chunk or w.T
    ws_bytes = (C.crc_fused_workspace_bytes(p) if args.only == "fused" and not args.chunk
                else C.crc_workspace_bytes(p, chunk))
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=dev)
    st = P.State(p, device=dev)
    torch.cuda.synchronize()

    if args.only != "fused":
        scores = P.route_scores(p, hd, Wd, heads=heads)
        args.no_e2e = args.no_e2e or args.only != "pair"

    def step():
        if args.only == "router":
            C.crc_route_scores(p, hd.data_ptr(), Wd.data_ptr(), w.T, heads, scores.data_ptr(),
                               stream)
            return
        st.init()
        if args.only == "scan":
            if args.policy != "method":
                C.crc_cache_scan_policy(p, scores.data_ptr(), w.T, st.ptr, st.nbytes, None,
                                        C.POLICIES[args.policy], 1, stream)
            else:
                C.crc_cache_scan(p, scores.data_ptr(), w.T, st.ptr, st.nbytes, None, stream)
            return
        if args.only == "pair":
            C.crc_route_scores(p, hd.data_ptr(), Wd.data_ptr(), w.T, heads, scores.data_ptr(),
                               stream)
            C.crc_cache_scan(p, scores.data_ptr(), w.T, st.ptr, st.nbytes, None, stream)
            return
        C.crc_route_and_cache(p, hd.data_ptr(), Wd.data_ptr(), w.T, st.ptr, st.nbytes, None,
                              ws.data_ptr(), ws.numel(), stream)

    for _ in range(max(3, args.warmup)):
        step()
    stats = st.read()
    assert stats["error"] == 0 and stats["tokens"] == (0 if args.only == "router" else w.T), stats
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()

    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(gpu_id_for_smi(torch, local)) as clk:
        C.crc_profile_begin()
        n0 = C.crc_launch_count()
        e0.record(stream)
        for _ in range(args.steps):
            step()
        e1.record(stream)
        torch.cuda.synchronize()
        launches = C.crc_launch_count() - n0
        kt = C.crc_profile_end()
    ms = max_over_ranks(e0.elapsed_time(e1), world, dev)
    if world > 1:
        dist.barrier()
    ms_per_step = ms / args.steps
    units_all = w.units * world
    value = job_rate(w.units, world, ms_per_step)

    # a comparison policy's scan reads p^R only (Spatio-only: and p^S)
    scan_heads = heads if args.policy == "method" else (2 if args.policy == "spatio_lru" else 1)
    clocks = clk.summary()
    roof, path_roof, kernels = rooflines(kt, w, heads, args.steps, ms, ms_per_step, scan_heads,
                                         clocks)
    if args.policy != "method" and roof.get("kernel") == "cache_scan_kernel":
        roof["kernel"] = f"cache_scan_policy_kernel ({args.policy})"

    # end to end through the C ABI from pinned host memory
    e2e = None
    if not args.no_e2e:
        held = [hd]                 # the device copy is dropped before the host round trip
        del hd
        e2e = end_to_end(args, P, C, w, p, held, Wd, st, ws, stream, dev, world, units_all)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:
        cpu, _, _ = cpu_oracle_sample(w, args.cpu_seconds)

    if rank == 0:
        m = P.metrics(stats, p)
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": max(3, args.warmup), "ms_per_step": ms_per_step,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic",
            "config": dict(workload_config(w, None if args.only == "fused" and not args.chunk
                                           else chunk), path=args.only, policy=args.policy,
                           workspace_bytes=int(ws_bytes)),
            "roofline": roof, "path_roofline": path_roof, "kernels": kernels,
            "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": int(launches),
            "clocks": clocks,
            "policy": policy_report(P, stats, p, m),
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()
    return 0


def tensor_peak(pk, clocks):
    """The bf16 peak that matches the timed region's clock regime: the measured
    sustained figure (a GEMM held at the power cap) when the power cap held the
    SM clock for most of the region (median below 95 % of the maximum), else
    the burst figure."""
    capped = (bool(clocks) and "sw_power_cap" in (clocks.get("reasons") or [])
              and clocks.get("sm_mhz") is not None
              and clocks["sm_mhz"] < 0.95 * (clocks.get("sm_max_mhz") or clocks["sm_mhz"]))
    if capped:
        return pk["bf16_tflops_sustained"], "sustained: sw_power_cap active in the timed region"
    return pk["bf16_tflops"], "burst"


def rooflines(kt, w, heads, steps, ms, ms_per_step, scan_heads=None, clocks=None):
    """Roofline of the dominant kernel (timed live over the timed region) and of
    the whole path (max of flops at the bf16 peak and bytes at HBM bandwidth)."""
    pk, pk_src = peaks()
    tpk, tpk_kind = tensor_peak(pk, clocks)
    dom = max(("fused", "router", "scan"), key=lambda k: kt[k]["ms"])
    avg_ms = kt[dom]["ms"] / max(1, kt[dom]["launches"])
    t_s = kt[dom]["ms"] / 1000.0
    if dom == "scan":
        flops = 0.0
        bytes_ = 4.0 * (scan_heads or heads) * w.N * w.units * steps   # probabilities read once
        kname = "cache_scan_kernel"
    elif dom == "router":
        flops = 2.0 * w.d * heads * w.N * w.units * steps
        bytes_ = (2.0 * w.d + 4.0 * heads * w.N) * w.units * steps   # + scores written
        kname = f"router_heads_kernel<{w.N},{heads}>"
    else:
        flops, bytes_ = algorithmic(w, w.units, heads)
        flops, bytes_ = flops * steps, bytes_ * steps
        kname = f"fused_route_cache_kernel<{w.N},{heads}>"
    t_flop = flops / (tpk * 1e12)
    t_byte = bytes_ / (pk["hbm_gbs"] * 1e9)
    if t_flop >= t_byte:
        roof = {"bound": "tensor", "achieved": flops / t_s / 1e12, "peak": tpk,
                "unit": "TFLOP/s", "frac": t_flop / t_s,
                "frac_of_burst": flops / (pk["bf16_tflops"] * 1e12) / t_s,
                "frac_of_sustained": flops / (pk["bf16_tflops_sustained"] * 1e12) / t_s}
    else:
        roof = {"bound": "hbm", "achieved": bytes_ / t_s / 1e9, "peak": pk["hbm_gbs"],
                "unit": "GB/s", "frac": t_byte / t_s}
    per_unit, src = committed_traffic(kname, w.name)
    units_per_launch = w.units * steps / max(1, kt[dom]["launches"])
    roof["traffic"] = None if per_unit is None else per_unit * units_per_launch
    roof.update({"kernel": kname, "peak_source": f"{pk_src} ({tpk_kind if roof['bound'] == 'tensor' else 'copy'})",
                 "avg_launch_ms": avg_ms, "launches": kt[dom]["launches"],
                 "share_of_step": kt[dom]["ms"] / ms if ms else None})
    # whole-path roofline: the slower of the flops at the bf16 peak and the bytes at HBM bandwidth
    fl, by = algorithmic(w, w.units, heads)
    t_roof = max(fl / (tpk * 1e12), by / (pk["hbm_gbs"] * 1e9))
    path_roof = {"t_roof_ms": 1000 * t_roof, "frac": 1000 * t_roof / ms_per_step,
                 "bound": "tensor" if fl / (tpk * 1e12) >= by / (pk["hbm_gbs"] * 1e9)
                 else "hbm", "tensor_peak": tpk_kind}
    kernels = {k: {"launches": v["launches"], "ms_per_step": v["ms"] / steps}
               for k, v in kt.items() if v["launches"]}
    return roof, path_roof, kernels


E2E_CHUNK = 128          # tokens per host-to-device copy of the end-to-end step
STREAM_BYTES = 128 << 30     # hidden states above this are generated per chunk
STREAM_CHUNK = 128           # tokens per chunk of a streamed workload


def run_streamed(args, P, C, w, p, heads, dev, stream, rank, world):
    """Workloads whose hidden states do not fit in HBM (the 1.6 TB large shape).
    A step walks the T tokens in 128-token chunks: the device generator writes
    a chunk (untimed; the AR(1) field continues through its carry), and the
    fused route-and-cache call on it is timed with CUDA events on the stream.
    The step time is the sum of its timed calls."""
    import torch
    import torch.distributed as dist
    CH = min(STREAM_CHUNK, w.T)
    n_chunks = (w.T + CH - 1) // CH
    Wd = P.synth_weights(w.L, w.N, w.d, seed=0, device=dev)
    hflat = torch.empty(w.B * CH * w.L * w.d, dtype=torch.bfloat16, device=dev)
    carry = torch.zeros((w.B, w.L, w.d), dtype=torch.float32, device=dev)
    ws_bytes = C.crc_fused_workspace_bytes(p)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=dev)
    st = P.State(p, device=dev)
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(n_chunks)]

    def step(timed):
        st.init()
        carry.zero_()
        for c in range(n_chunks):
            t0 = c * CH
            n = min(CH, w.T - t0)
            h = hflat[: w.B * n * w.L * w.d].view(w.B, n, w.L, w.d)
            P.synth_hidden(w.B, n, w.L, w.d, seed=rank_seed(rank), rho_t=w.rho_t, rho_l=w.rho_l,
                           t0=t0, carry=carry, out=h, device=dev)
            if timed:
                evs[c][0].record(stream)
            C.crc_route_and_cache(p, h.data_ptr(), Wd.data_ptr(), n, st.ptr, st.nbytes, None,
                                  ws.data_ptr(), ws.numel(), stream)
            if timed:
                evs[c][1].record(stream)
        if not timed:
            return 0.0
        torch.cuda.synchronize()
        return sum(a.elapsed_time(b) for a, b in evs)

    for _ in range(max(3, args.warmup)):
        step(False)
    stats = st.read()
    assert stats["error"] == 0 and stats["tokens"] == w.T, stats
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(gpu_id_for_smi(torch, int(os.environ.get("LOCAL_RANK", "0")))) as clk:
        C.crc_profile_begin()
        ms = 0.0
        for _ in range(args.steps):
            ms += step(True)
        kt = C.crc_profile_end()
    stats = st.read()
    ms = max_over_ranks(ms, world, dev)
    ms_per_step = ms / args.steps
    units_all = w.units * world
    value = job_rate(w.units, world, ms_per_step)
    clocks = clk.summary()
    roof, path_roof, kernels = rooflines(kt, w, heads, args.steps, ms, ms_per_step, None, clocks)
    kernels.pop("synth", None)
    kernels.pop("state", None)
    launches = sum(kt[k]["launches"] for k in ("fused", "router", "scan"))
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:
        cpu, _, _ = cpu_oracle_sample(w, args.cpu_seconds)
    if rank == 0:
        m = P.metrics(stats, p)
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": max(3, args.warmup), "ms_per_step": ms_per_step,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic",
            "config": dict(workload_config(w, CH), path="fused, streamed",
                           workspace_bytes=int(ws_bytes),
                           timing="sum of per-call CUDA events; chunk generation untimed"),
            "roofline": roof, "path_roofline": path_roof, "kernels": kernels,
            "cpu_baseline": cpu,
            "e2e": None, "e2e_note": "hidden states exceed host and device memory; "
                                     "generated on the device per chunk",
            "gpu_launches": int(launches), "clocks": clocks,
            "policy": policy_report(P, stats, p, m),
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()
    return 0


def end_to_end(args, P, C, w, p, held, Wd, st, ws, stream, dev, world, units_all):
    """The same metric through the C ABI's host-input call: every step copies
    its hidden states from pinned host memory (crc_host_alloc's huge pages; in
    128-token chunks, each copy overlapping the step on the previous chunk) and
    reads its counters back, inside the timed region."""
    import torch
    import torch.distributed as dist
    hd = held.pop()
    h_host, host_mem = pinned_host(P, hd.shape, hd.dtype)
    h_host.copy_(hd)
    del hd
    torch.cuda.empty_cache()
    chunk = min(E2E_CHUNK, w.T)
    staging = torch.empty(C.crc_host_staging_bytes(p, chunk), dtype=torch.uint8, device=dev)
    torch.cuda.synchronize()

    def e2e_step():
        st.init()
        C.crc_route_and_cache_host(p, h_host.data_ptr(), Wd.data_ptr(), w.T, chunk, st.ptr,
                                   st.nbytes, staging.data_ptr(), staging.numel(),
                                   ws.data_ptr(), ws.numel(), stream)
        return st.read()      # synchronises; reads the step's counters back

    for _ in range(2):
        e2e_step()
    if world > 1:
        dist.barrier()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        r = e2e_step()
    dt = max_over_ranks(time.perf_counter() - t0, world, dev)
    assert r["error"] == 0
    h2d = int(h_host.numel() * h_host.element_size())
    return {"value": units_all * args.steps / dt, "unit": UNIT,
            "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": int(256 + p.B * p.L * 64),
            "ms_per_step": 1000 * dt / args.steps,
            "call": f"crc_route_and_cache_host, {chunk}-token chunks", "host_memory": host_mem,
            "host_link_gbs": host_link_gbs(h_host, staging, stream),
            "h2d_gbs": h2d / (dt / args.steps) / 1e9}


def pinned_host(P, shape, dtype):
    """Pinned host memory for an end-to-end input: crc_host_alloc's huge pages,
    else (registration refused on this host) cudaHostAlloc's, named in the line."""
    import torch
    try:
        return P.pinned_empty(shape, dtype), "crc_host_alloc (huge pages)"
    except P.CrcError as e:
        return torch.empty(shape, dtype=dtype, pin_memory=True), f"cudaHostAlloc ({e})"


def host_link_gbs(h_host, dev_buf, stream) -> float:
    """This run's host-to-device copy rate: one plain pinned copy of up to
    4 GiB (best of 3, CUDA events), the ceiling for the end-to-end step."""
    import torch
    n = min(h_host.numel() * h_host.element_size(), dev_buf.numel(), 4 << 30)
    src = h_host.view(-1).view(torch.uint8)[:n]
    dst = dev_buf[:n]
    best = float("inf")
    for _ in range(3):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        dst.copy_(src, non_blocking=True)
        e1.record(stream)
        torch.cuda.synchronize()
        best = min(best, e0.elapsed_time(e1) / 1e3)
    return n / best / 1e9


if __name__ == "__main__":
    sys.exit(main())
