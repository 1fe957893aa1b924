#!/usr/bin/env python
"""Benchmark of the ResBM boundary bottleneck on GB300: one step = encode fwd -> decode fwd ->
decode bwd -> encode bwd (with the weight-gradient reductions) over one batch of T tokens.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--config large_bf16] [--impl resbm|reference]

Prints ONE JSON line (rank 0). value = boundary tokens per second over all ranks, timed over K
resbm_boundary_step calls (inputs resident in HBM); `e2e` = the same with pinned host buffers and
the host<->device copies inside the timed region; `roofline` = the dominant op's algorithmic HBM
bytes / its CUDA-event time against the measured copy bandwidth; `cpu_baseline` = the fp64
oracle on the host cores, on a bounded token sample. With N > 1 (torchrun) every rank runs an
independent replica of the workload on its own GPU (the boundary op has no exchange step when
run as one pipeline boundary per GPU); the slowest rank's time counts.
"""
import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2604_11947_gb300 import synth  # noqa: E402

OPS = ("enc_fwd", "dec_fwd", "dec_bwd", "enc_bwd")
METRIC = "boundary tokens/sec and achieved HBM GB/s (fwd+bwd) vs GB300 peak at 1 GPU"


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=200)
    p.add_argument("--warmup", type=int, default=10)
    p.add_argument("--config", default="large_bf16", choices=sorted(synth.CONFIGS))
    p.add_argument("--tokens", type=int, default=None,
                   help="override T (smaller cases for profiler captures; not a bench line)")
    p.add_argument("--impl", default="resbm", choices=("resbm", "reference"))
    p.add_argument("--generic", action="store_true", help="force the CUDA-core kernels")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-cpu", action="store_true", help="skip the oracle CPU baseline")
    return p.parse_args()


# ---- algorithmic bytes (per op) -------------------------------------------------------------
def op_bytes(cfg):
    """HBM bytes each op must move at minimum: activations once, weights once, P in fp32."""
    T, d, r, m = cfg.T, cfg.d, cfg.r, cfg.m
    e = 2 if cfg.dtype == "bf16" else 4
    return {
        # F read, X[:, :r] read, B write, P write; We1, We2 read
        "enc_fwd": T * (e * d + 2 * e * r + 4 * m) + e * (d * m + m * r),
        # B read, Y write; Wd1, Wd2 read
        "dec_fwd": T * (e * r + e * d) + e * (r * m + m * d),
        # dY read, B read, dB write; weights read; dWd1, dWd2 written (fp32)
        "dec_bwd": T * (e * d + 2 * e * r) + e * (r * m + m * d) + 4 * (r * m + m * d),
        # F read, dF write, dB read, P read, dX[:, :r] read + write; weights; dWe1, dWe2
        "enc_bwd": T * (2 * e * d + 3 * e * r + 4 * m) + e * (d * m + m * r) + 4 * (d * m + m * r),
    }


def op_flops(cfg):
    T, d, r, m = cfg.T, cfg.d, cfg.r, cfg.m
    return {"enc_fwd": 2 * T * (d * m + m * r), "dec_fwd": 2 * T * (r * m + m * d),
            "dec_bwd": 2 * T * (r * m + 2 * m * d + m * r) + 2 * T * r * m,
            "enc_bwd": 2 * T * (r * m + 2 * d * m + m * r)}


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            j = json.load(f)
        return {"hbm_gbs": j["hbm_gbs"], "bf16_tflops": j["bf16_tflops"], "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "source": "fallback"}


def kernel_sources_sha():
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2604_11947_gb300", "csrc")
    for f in sorted(os.listdir(csrc)):
        with open(os.path.join(csrc, f), "rb") as fh:
            h.update(f.encode() + fh.read())
    return h.hexdigest()[:16]


def traffic_for(op, cfg):
    """DRAM bytes per launch from the committed ncu summary, if taken on the current kernels."""
    path = os.path.join(ROOT, "profiles", "dram_traffic.json")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        j = json.load(f)
    if j.get("kernel_sources_sha") != kernel_sources_sha():
        return None
    ent = j.get("ops", {}).get(cfg.name, {}).get(op)
    return None if ent is None else ent.get("dram_bytes_per_launch")


# ---- clocks during the timed region ---------------------------------------------------------
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    NAMES = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")

    def __init__(self, device_uuid=None):
        self.uuid = device_uuid
        self.lines = []
        self.proc = None

    def start(self):
        cmd = ["nvidia-smi", "--query-gpu=" + self.FIELDS, "--format=csv,noheader,nounits",
               "-lms", "50"]
        if self.uuid:
            cmd += ["-i", self.uuid]
        try:
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL,
                                         text=True)
        except OSError:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"],
                    "samples": 0}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=5)
        sm, smax, power, reasons = [], [], [], set()
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
                power.append(float(parts[3]))
            except ValueError:
                continue
            for name, val in zip(self.NAMES, parts[5:9]):
                if val.lower() == "active":
                    reasons.add(name)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "power_w_max": max(power) if power else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ---- the CPU baseline (fp64 oracle) ---------------------------------------------------------
_sample_cache = {}


def oracle_sample_run(cfg, n):
    """The oracle's full boundary step on the first n tokens of the workload; returns seconds
    (input generation excluded)."""
    import oracle
    key = (cfg.name, n)
    if key not in _sample_cache:
        _sample_cache.clear()
        h = {k: synth.tensor(cfg, k, nrows=n) for k in ("X", "F", "dY")}
        for k in ("We1", "We2", "Wd1", "Wd2"):
            h[k] = synth.tensor(cfg, k)
        _sample_cache[key] = h
    h = _sample_cache[key]
    t0 = time.perf_counter()
    oracle.boundary_step(h["X"], h["F"], h["dY"], h["We1"], h["We2"], h["Wd1"], h["Wd2"],
                         act=cfg.act, merge=cfg.merge)
    return time.perf_counter() - t0


def oracle_rate(cfg, budget_s):
    """Calibrate on a small sample, then time a sample sized to about budget_s seconds."""
    n0 = min(cfg.T, 64)
    t0 = oracle_sample_run(cfg, n0)
    n = int(min(cfg.T, max(n0, budget_s / max(t0, 1e-6) * n0)))
    t = oracle_sample_run(cfg, n) if n != n0 else t0
    return n, t


def cpu_baseline(cfg, budget_s=15.0, one_core_budget_s=5.0):
    """The oracle on all host cores (OpenMP) and on one core, each on a bounded token sample."""
    import oracle
    cores = oracle.max_threads()
    n, t = oracle_rate(cfg, budget_s)
    oracle.set_threads(1)
    try:
        n1, t1 = oracle_rate(cfg, one_core_budget_s)
    finally:
        oracle.set_threads(cores)
    return {"value": n / t, "unit": "tokens/s", "cores": cores, "kind": "oracle",
            "sample": "fp64 oracle boundary step (encode fwd, decode fwd, decode bwd, encode bwd, "
                      "weight gradients over the sample) on tokens 0..%d of the %s workload, "
                      "%.2f s on %d threads" % (n - 1, cfg.name, t, cores),
            "one_core": {"value": n1 / t1, "unit": "tokens/s", "cores": 1,
                         "sample": "tokens 0..%d, %.2f s" % (n1 - 1, t1)}}


def describe(cfg, extra=None):
    c = {"workload": "%s: T=%d tokens, d=%d, r=%d (%dx compression), m=%d, %s I/O, act=%s, "
                     "merge=%d" % (cfg.name, cfg.T, cfg.d, cfg.r, cfg.d // cfg.r, cfg.m, cfg.dtype,
                                   cfg.act, cfg.merge),
         "T": cfg.T, "d": cfg.d, "r": cfg.r, "m": cfg.m, "act": cfg.act, "merge": cfg.merge,
         "inputs": "seeded synthetic: X, F ~ N(0,1) x per-token log-normal(0,0.5); dY ~ N(0,1); "
                   "weights N(0, 1/fan_in)"}
    if extra:
        c.update(extra)
    return c


def run_reference(args, cfg, rank):
    """The reference arm: the fp64 oracle as it stands, on the host cores."""
    if rank != 0:
        return
    import oracle
    total_budget = 120.0
    per_step = max(0.05, total_budget / max(1, args.steps + args.warmup))
    n0 = min(cfg.T, 16)
    t0 = oracle_sample_run(cfg, n0)
    n = int(min(cfg.T, max(n0, per_step / max(t0, 1e-6) * n0)))
    for _ in range(args.warmup):
        oracle_sample_run(cfg, n)
    times = [oracle_sample_run(cfg, n) for _ in range(args.steps)]
    total = sum(times)
    value = n * args.steps / total
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * total / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": describe(cfg, {"sample_tokens_per_step": n}),
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": oracle.max_threads(),
                             "kind": "oracle",
                             "sample": "tokens 0..%d of the %s workload per step" % (n - 1, cfg.name)},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ---- multi-rank host logic (one independent replica per GPU) --------------------------------
def max_over_ranks(ms, dist, device):
    """The slowest rank's time: every rank gets the maximum of all ranks' `ms`."""
    if not dist:
        return ms
    import torch
    t = torch.tensor([float(ms)], device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(tokens_per_rank, world, steps, ms_total):
    """Whole-job tokens/s: the tokens all ranks processed over the slowest rank's time."""
    return tokens_per_rank * world * steps / (ms_total / 1e3)


# ---- the GPU arm ----------------------------------------------------------------------------
def main():
    args = parse()
    cfg = synth.CONFIGS[args.config]
    if args.tokens:
        cfg = cfg.with_(name="%s_T%d" % (cfg.name, args.tokens), T=args.tokens)
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        run_reference(args, cfg, rank)
        return

    import torch
    from paper_2604_11947_gb300 import build, resbm

    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA GPU (there is no CPU fallback)")
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    build.build()
    lib = resbm.load()

    flags = resbm.RESBM_FLAG_GENERIC if args.generic else 0
    desc = resbm.desc_from_config(cfg, flags)
    io = torch.bfloat16 if cfg.dtype == "bf16" else torch.float32
    dev = {k: torch.from_numpy(synth.tensor(cfg, k)).to("cuda").to(io)
           for k in ("X", "F", "dY", "We1", "We2", "Wd1", "Wd2")}
    out = resbm.step_outputs(desc)
    ws = resbm.workspace(desc, resbm.RESBM_OP_BOUNDARY_STEP)
    wsz = ws.numel()
    stream = torch.cuda.current_stream()

    def step(ev=None):
        if ev is not None:
            ev[0].record(stream)
        resbm.resbm_encode_fwd(desc, dev["X"], dev["F"], dev["We1"], dev["We2"], out["B"], out["P"], ws)
        if ev is not None:
            ev[1].record(stream)
        resbm.resbm_decode_fwd(desc, out["B"], dev["Wd1"], dev["Wd2"], out["Y"], ws)
        if ev is not None:
            ev[2].record(stream)
        resbm.resbm_decode_bwd(desc, dev["dY"], out["B"], dev["Wd1"], dev["Wd2"], out["dB"],
                               out["dWd1"], out["dWd2"], ws)
        if ev is not None:
            ev[3].record(stream)
        resbm.resbm_encode_bwd(desc, out["dB"], dev["F"], out["P"], dev["We1"], dev["We2"],
                               out["dF"], out["dX"], out["dWe1"], out["dWe2"], ws)
        if ev is not None:
            ev[4].record(stream)

    def fused_step():
        resbm.resbm_boundary_step(desc, ws, X=dev["X"], F=dev["F"], dY=dev["dY"], We1=dev["We1"],
                                  We2=dev["We2"], Wd1=dev["Wd1"], Wd2=dev["Wd2"], **out)

    for _ in range(max(args.warmup, 0)):
        fused_step()
    for _ in range(max(args.warmup, 0)):
        step()
    torch.cuda.synchronize()

    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(5)] for _ in range(args.steps)]
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    props = torch.cuda.get_device_properties(local)
    uuid = getattr(props, "uuid", None)
    uuid = None if uuid is None else (str(uuid) if str(uuid).startswith("GPU-") else "GPU-" + str(uuid))
    clocks = ClockSampler(uuid)
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    clocks.start()
    time.sleep(0.15)
    # timed region: K boundary steps through the library's step call, no events in between
    # (an event between two kernels ends their programmatic-dependent-launch overlap)
    launches0 = resbm.resbm_kernel_launches()
    start.record(stream)
    for i in range(args.steps):
        fused_step()
    end.record(stream)
    torch.cuda.synchronize()
    launches = resbm.resbm_kernel_launches() - launches0
    # second timed pass, same K steps as four op calls with events between them: the per-op
    # times of the roofline (these steps are a few percent slower than the ones above)
    for i in range(args.steps):
        step(evs[i])
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    clk = clocks.stop()
    ms_total = max_over_ranks(start.elapsed_time(end), dist, "cuda")
    ms_step = ms_total / max(args.steps, 1)
    value = job_throughput(cfg.T, world, args.steps, ms_total)

    op_ms = {op: statistics.mean(evs[i][j].elapsed_time(evs[i][j + 1]) for i in range(args.steps))
             for j, op in enumerate(OPS)}
    bytes_ = op_bytes(cfg)
    flops = op_flops(cfg)
    peaks = measured_peaks()
    dom = max(OPS, key=lambda o: op_ms[o])
    achieved = bytes_[dom] / (op_ms[dom] / 1e3) / 1e9
    step_bytes = sum(bytes_.values())
    roofline = {"bound": "hbm", "kernel": dom, "achieved": achieved, "peak": peaks["hbm_gbs"],
                "unit": "GB/s", "frac": achieved / peaks["hbm_gbs"],
                "traffic": traffic_for(dom, cfg),
                "peak_source": peaks["source"] + " copy bandwidth (MEASURED_PEAKS.json hbm_gbs)",
                "algorithmic_bytes_per_launch": bytes_[dom],
                "timing": "per-op CUDA events on the launching stream in a second timed pass "
                          "of the same K steps (op calls with events between them)",
                "per_op": {o: {"ms": op_ms[o], "alg_bytes": bytes_[o],
                               "GBps": bytes_[o] / (op_ms[o] / 1e3) / 1e9,
                               "frac": bytes_[o] / (op_ms[o] / 1e3) / 1e9 / peaks["hbm_gbs"],
                               "TFLOPs": flops[o] / (op_ms[o] / 1e3) / 1e12} for o in OPS},
                "step_GBps": step_bytes / (ms_step / 1e3) / 1e9}

    e2e = None
    if not args.no_e2e:
        e2e = run_e2e(args, cfg, desc, dev, out, ws, resbm, torch, dist, world)

    line = {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": cfg.dtype,
            "data": "synthetic",
            "config": describe(cfg, {"parallelism": "replicas x%d (one boundary per GPU)" % world,
                                     "l2": "inputs X, F, dY of %d MiB each exceed the 129 MB L2; "
                                           "no flush" % (cfg.T * cfg.d * (2 if cfg.dtype == "bf16" else 4) >> 20),
                                     "path": "generic CUDA-core" if args.generic else "default"}),
            "hbm_GBps_step": roofline["step_GBps"],
            "roofline": roofline, "e2e": e2e, "gpu_launches": launches,
            "clocks": clk}
    if rank == 0 and world == 1 and not args.no_cpu:
        line["cpu_baseline"] = cpu_baseline(cfg)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()


def run_e2e(args, cfg, desc, dev, out, ws, resbm, torch, dist, world):
    """The same step through the C ABI with HOST buffers (resbm_boundary_step_host): inputs in
    pinned host memory, results back into pinned host memory, every copy inside the call and
    inside the timed region. Two calls are kept in flight (two streams, two device workspaces,
    two sets of host results), so one step's results travel back while the next step's inputs
    travel in, as a training loop fed from the host would run them."""
    ins = ("X", "F", "dY", "We1", "We2", "Wd1", "Wd2")
    res = ("B", "Y", "dB", "dF", "dWe1", "dWe2", "dWd1", "dWd2")
    host_in = {k: dev[k].cpu().pin_memory() for k in ins}
    host_out = [{k: torch.empty(out[k].shape, dtype=out[k].dtype).pin_memory() for k in res}
                for _ in range(2)]
    wss = [resbm.workspace(desc, resbm.RESBM_OP_BOUNDARY_STEP_HOST) for _ in range(2)]
    streams = [torch.cuda.Stream() for _ in range(2)]
    es = host_in["F"].element_size()
    # what the call copies: X[:, :r] only (the identity path), F, dY and the weights in; the
    # results out
    h2d = cfg.T * cfg.r * es + sum(host_in[k].numel() * es for k in ins if k != "X")
    d2h = sum(t.numel() * t.element_size() for t in host_out[0].values())
    # up to 100 steps (≈0.65 s): the host link sometimes stalls for ~100 ms (seen as 30-55 ms
    # gaps between consecutive steps whose steady pace is 6.4 ms); a short window would charge
    # one such stall to a handful of steps
    n = max(2, min(args.steps, 100))

    def step(i):
        b = i % 2
        resbm.resbm_boundary_step_host(desc, wss[b], stream=streams[b], **host_in, **host_out[b])

    for i in range(2):
        step(i)
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    t0 = time.perf_counter()
    for i in range(n):
        step(i)
    torch.cuda.synchronize()
    ms = max_over_ranks((time.perf_counter() - t0) * 1e3, dist, "cuda")
    return {"value": job_throughput(cfg.T, world, n, ms), "unit": "tokens/s",
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "steps": n,
            "ms_per_step": ms / n,
            "api": "resbm_boundary_step_host (host buffers; copies inside the call)",
            "pipelined": "two calls in flight on two streams with two device workspaces; "
                         "host wall clock from the first copy to the last result on the host"}


if __name__ == "__main__":
    main()
