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
    p.add_argument("--no-extra", action="store_true",
                   help="skip the other workloads (T=16384 d=2048 r=16 and the d=8192 r-sweep)")
    p.add_argument("--rmsnorm-only", action="store_true",
                   help="run only the decoder forward + RMSNorm comparison (for profiler captures; "
                        "--steps / --warmup apply); prints its JSON object, not a bench line")
    p.add_argument("--hbm-forms-only", action="store_true",
                   help="only the HBM rate of each access form (resbm_measure_hbm_form), 1 GiB buffers")
    p.add_argument("--ffn-only", action="store_true",
                   help="run only the FFN down-projection + encoder comparison (for profiler captures; "
                        "--steps / --warmup apply); prints its JSON object, not a bench line")
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


NOMINAL_HBM_GBS = 8000.0    # the GB300's nominal HBM3e bandwidth (the 70 % target is stated on it)
TARGET_FRAC = 0.70


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            j = json.load(f)
        return {"hbm_gbs": j["hbm_gbs"], "bf16_tflops": j["bf16_tflops"],
                "bf16_tflops_sustained": j.get("bf16_tflops_sustained", j["bf16_tflops"]),
                "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
            "source": "fallback"}


# The files that define the fused boundary kernels the bench workload runs (their device code;
# their launch rules in tc.cu have not changed since these files were split out): the committed
# DRAM traffic is valid while these hash the same.
BENCH_KERNEL_FILES = ("common.cuh", "tc_common.cuh", "tc_wgrad.cuh", "tc_enc_fwd.cuh", "tc_dec_fwd.cuh",
                      "tc_dec_bwd.cuh", "tc_enc_bwd.cuh")


def kernel_sources_sha():
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2604_11947_gb300", "csrc")
    for f in BENCH_KERNEL_FILES:
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
def device_inputs(cfg, torch, reuse=None):
    """The workload's seeded inputs in HBM. `reuse`: tensors of another workload with the same
    (T, d) whose X, F, dY are the same draws (the tensors depend only on their shapes)."""
    io = torch.bfloat16 if cfg.dtype == "bf16" else torch.float32
    dev = {}
    for k in ("X", "F", "dY", "We1", "We2", "Wd1", "Wd2"):
        if reuse is not None and k in ("X", "F", "dY") and reuse[k].shape == synth.shapes(cfg)[k]:
            dev[k] = reuse[k]
        else:
            dev[k] = torch.from_numpy(synth.tensor(cfg, k)).to("cuda").to(io)
    return dev


class Workload:
    """One workload's device tensors and its two ways of running a step: the library's step call
    (timed for `value`) and the four op calls with events between them (per-op times)."""

    def __init__(self, cfg, flags, dev, resbm, torch):
        self.cfg, self.dev, self.resbm, self.torch = cfg, dev, resbm, torch
        self.desc = resbm.desc_from_config(cfg, flags)
        self.out = resbm.step_outputs(self.desc)
        self.ws = resbm.workspace(self.desc, resbm.RESBM_OP_BOUNDARY_STEP)
        self.stream = torch.cuda.current_stream()

    def fused_step(self):
        d, o = self.dev, self.out
        self.resbm.resbm_boundary_step(self.desc, self.ws, X=d["X"], F=d["F"], dY=d["dY"], We1=d["We1"],
                                       We2=d["We2"], Wd1=d["Wd1"], Wd2=d["Wd2"], **o)

    def op_step(self, ev=None):
        r, d, o, desc, ws = self.resbm, self.dev, self.out, self.desc, self.ws
        if ev is not None:
            ev[0].record(self.stream)
        r.resbm_encode_fwd(desc, d["X"], d["F"], d["We1"], d["We2"], o["B"], o["P"], ws)
        if ev is not None:
            ev[1].record(self.stream)
        r.resbm_decode_fwd(desc, o["B"], d["Wd1"], d["Wd2"], o["Y"], ws)
        if ev is not None:
            ev[2].record(self.stream)
        r.resbm_decode_bwd(desc, d["dY"], o["B"], d["Wd1"], d["Wd2"], o["dB"], o["dWd1"], o["dWd2"], ws)
        if ev is not None:
            ev[3].record(self.stream)
        r.resbm_encode_bwd(desc, o["dB"], d["F"], o["P"], d["We1"], d["We2"], o["dF"], o["dX"],
                           o["dWe1"], o["dWe2"], ws)
        if ev is not None:
            ev[4].record(self.stream)

    def warm(self, n):
        for _ in range(max(n, 0)):
            self.fused_step()
        for _ in range(max(n, 0)):
            self.op_step()
        self.torch.cuda.synchronize()

    def time_steps(self, steps):
        """ms of `steps` step calls between two events, no event in between (an event between
        two kernels ends their programmatic-dependent-launch overlap), and the launches they
        made."""
        torch = self.torch
        start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        l0 = self.resbm.resbm_kernel_launches()
        start.record(self.stream)
        for _ in range(steps):
            self.fused_step()
        end.record(self.stream)
        torch.cuda.synchronize()
        return start.elapsed_time(end), self.resbm.resbm_kernel_launches() - l0

    def time_ops(self, steps):
        """Mean ms of each op over `steps` op-wise steps (CUDA events on the launching stream)."""
        torch = self.torch
        evs = [[torch.cuda.Event(enable_timing=True) for _ in range(5)] for _ in range(steps)]
        for i in range(steps):
            self.op_step(evs[i])
        torch.cuda.synchronize()
        return {op: statistics.mean(evs[i][j].elapsed_time(evs[i][j + 1]) for i in range(steps))
                for j, op in enumerate(OPS)}


def per_op_table(cfg, op_ms, peaks):
    """Each op's time, algorithmic GB/s and FLOP rate, and its fractions of the measured copy
    bandwidth, of the nominal 8 TB/s and of the sustained bf16 tensor rate."""
    bytes_, flops = op_bytes(cfg), op_flops(cfg)
    t = {}
    for o in OPS:
        gbs = bytes_[o] / (op_ms[o] / 1e3) / 1e9
        tfs = flops[o] / (op_ms[o] / 1e3) / 1e12
        t[o] = {"ms": op_ms[o], "alg_bytes": bytes_[o], "GBps": gbs, "frac": gbs / peaks["hbm_gbs"],
                "frac_of_8TBps": gbs / NOMINAL_HBM_GBS, "TFLOPs": tfs,
                "frac_of_bf16_sustained": tfs / peaks["bf16_tflops_sustained"]}
    return t


def extra_workload(name, cfg, flags, resbm, torch, steps, warmup, peaks, reuse=None):
    """The step on another workload (fewer steps): tokens/s, GB/s and per-op fractions."""
    dev = device_inputs(cfg, torch, reuse)
    w = Workload(cfg, flags, dev, resbm, torch)
    w.warm(warmup)
    ms, launches = w.time_steps(steps)
    op_ms = w.time_ops(steps)
    ms_step = ms / steps
    step_bytes = sum(op_bytes(cfg).values())
    step_flops = sum(op_flops(cfg).values())
    per_op = per_op_table(cfg, op_ms, peaks)
    res = {"workload": describe(cfg)["workload"], "steps": steps, "warmup": warmup,
           "value": cfg.T / (ms_step / 1e3), "unit": "tokens/s", "ms_per_step": ms_step,
           "step_GBps": step_bytes / (ms_step / 1e3) / 1e9,
           "step_frac": step_bytes / (ms_step / 1e3) / 1e9 / peaks["hbm_gbs"],
           "step_TFLOPs": step_flops / (ms_step / 1e3) / 1e12,
           "gpu_launches_per_step": launches / steps,
           "min_op_frac": min(v["frac"] for v in per_op.values()),
           "per_op": per_op}
    if cfg.r >= 256:   # compute-bound point: the tensor rate is its roofline
        res["bound"] = "tensor"
        res["step_frac_of_bf16_sustained"] = res["step_TFLOPs"] / peaks["bf16_tflops_sustained"]
    else:
        res["bound"] = "hbm"
    del w
    return res, dev


def ffn_encode_workload(resbm, torch, steps=20, warmup=3):
    """The encoder fused into the FFN down-projection against the unfused chain, at the fifth
    workload's boundary (T = 16384, FFN width 5632, d = 2048, r = m = 16): fused (F never stored),
    fused with F stored (for the backward), and the down-projection by torch.matmul (cuBLAS) with F
    stored then resbm_encode_fwd reading it back."""
    T, f, d, r, m = 16384, 5632, 2048, 16, 16
    cfg = synth.BoundaryConfig("ffn_encode", T=T, d=d, r=r, m=m)
    g = torch.Generator(device="cuda")
    g.manual_seed(0)
    H = (torch.randn(T, f, device="cuda", generator=g) * 0.5).to(torch.bfloat16)
    W2 = (torch.randn(f, d, device="cuda", generator=g) / f ** 0.5).to(torch.bfloat16)
    X = torch.randn(T, d, device="cuda", generator=g).to(torch.bfloat16)
    We1 = (torch.randn(d, m, device="cuda", generator=g) / d ** 0.5).to(torch.bfloat16)
    We2 = (torch.randn(m, r, device="cuda", generator=g) / m ** 0.5).to(torch.bfloat16)
    desc = resbm.desc_from_config(cfg)
    ws = resbm.ffn_down_encode_workspace(desc, f)
    ws_enc = resbm.workspace(desc, resbm.RESBM_OP_ENCODE_FWD)
    B = torch.empty(T, r, dtype=torch.bfloat16, device="cuda")
    P = torch.empty(T, m, dtype=torch.float32, device="cuda")
    F = torch.empty(T, d, dtype=torch.bfloat16, device="cuda")
    runs = {"fused": lambda: resbm.resbm_ffn_down_encode_fwd(desc, H, W2, X, We1, We2, B, P, None, ws),
            "fused_storing_F": lambda: resbm.resbm_ffn_down_encode_fwd(desc, H, W2, X, We1, We2, B, P, F, ws),
            "unfused_cublas_then_encode": lambda: (torch.matmul(H, W2, out=F),
                                                   resbm.resbm_encode_fwd(desc, X, F, We1, We2, B, P, ws_enc))}
    res = {"workload": "FFN down-projection (T=%d, FFN width %d, d=%d) with the ResBM encoder (r=m=%d) "
                       "after it, bf16" % (T, f, d, r), "steps": steps, "flops": 2 * T * f * d + 2 * T * d * m}
    for name, fn in runs.items():
        for _ in range(warmup):
            fn()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(steps):
            fn()
        b.record()
        torch.cuda.synchronize()
        ms = a.elapsed_time(b) / steps
        res[name] = {"ms": ms, "TFLOPs": res["flops"] / (ms / 1e3) / 1e12}
    res["F_bytes_not_stored"] = 2 * T * d * 2   # written and read back by the unfused chain
    return res


def rmsnorm_alg_bytes(T, d, r, m):
    """Algorithmic HBM bytes (bf16) of the decoder forward + RMSNorm forms at T tokens: the fused
    pair reads B twice, the weights twice and gamma, writes Y and N, and writes then reads each
    row's 2 d / 256 fp32 partial sums (d / 256 column chunks of two halves, m <= 32); the unfused
    chain reads B and the weights once, writes Y, reads it back and writes N."""
    nch = d // 256
    w = 2 * (r * m + m * d)
    return {"fused": T * (2 * 2 * r + 2 * 2 * d + 2 * 4 * 2 * nch) + 2 * w + 2 * d,
            "unfused_decode_then_torch_rms_norm": T * (2 * r + 3 * 2 * d) + w + 2 * d,
            "decode_fwd_alone": T * (2 * r + 2 * d) + w}


def decode_rmsnorm_workload(resbm, torch, peaks, steps=50, warmup=5):
    """The decoder forward with the next block's pre-attention RMSNorm fused in, at the headline
    shape (T = 65536, d = 4096, r = m = 32, bf16): resbm_decode_fwd_rmsnorm (Y and N, Y never read
    back) against resbm_decode_fwd followed by torch's rms_norm over the stored Y, and the decoder
    forward alone. Algorithmic bytes: the fused pair reads B twice and the row sums of squares
    once, writes them, Y and N; the unfused chain reads B, writes Y, reads Y, writes N."""
    cfg = synth.CONFIGS["large_bf16"]
    T, d, r, m = cfg.T, cfg.d, cfg.r, cfg.m
    desc = resbm.desc_from_config(cfg)
    g = torch.Generator(device="cuda")
    g.manual_seed(0)
    B = torch.randn(T, r, device="cuda", generator=g).to(torch.bfloat16)
    Wd1 = (torch.randn(r, m, device="cuda", generator=g) / r ** 0.5).to(torch.bfloat16)
    Wd2 = (torch.randn(m, d, device="cuda", generator=g) / m ** 0.5).to(torch.bfloat16)
    gamma = (1 + 0.1 * torch.randn(d, device="cuda", generator=g)).to(torch.bfloat16)
    Y = torch.empty(T, d, dtype=torch.bfloat16, device="cuda")
    N = torch.empty(T, d, dtype=torch.bfloat16, device="cuda")
    ws = resbm.workspace(desc, resbm.RESBM_OP_DECODE_FWD_RMSNORM)
    ws_dec = resbm.workspace(desc, resbm.RESBM_OP_DECODE_FWD)
    eps = 1e-5
    runs = {"fused": lambda: resbm.resbm_decode_fwd_rmsnorm(desc, B, Wd1, Wd2, gamma, eps, Y, N, ws),
            "unfused_decode_then_torch_rms_norm": lambda: (
                resbm.resbm_decode_fwd(desc, B, Wd1, Wd2, Y, ws_dec),
                torch.nn.functional.rms_norm(Y, (d,), gamma, eps)),
            "decode_fwd_alone": lambda: resbm.resbm_decode_fwd(desc, B, Wd1, Wd2, Y, ws_dec)}
    alg = rmsnorm_alg_bytes(T, d, r, m)
    res = {"workload": "decoder forward + the next block's RMSNorm (T=%d, d=%d, r=m=%d, bf16)" % (T, d, r),
           "steps": steps, "inputs_exceed_l2": True}
    for name, fn in runs.items():
        for _ in range(warmup):
            fn()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(steps):
            fn()
        b.record()
        torch.cuda.synchronize()
        ms = a.elapsed_time(b) / steps
        gbs = alg[name] / (ms / 1e3) / 1e9
        res[name] = {"ms": ms, "alg_bytes": alg[name], "GBps": gbs, "frac": gbs / peaks["hbm_gbs"]}
    res["bytes_saved_by_fusion"] = alg["unfused_decode_then_torch_rms_norm"] - alg["fused"]
    # the backward: resbm_rmsnorm_bwd (dY + the norm's input gradient, dgamma) against torch's
    # rms_norm backward (autograd of a recomputed forward) followed by the residual add
    dN = torch.randn(T, d, device="cuda", generator=g).to(torch.bfloat16)
    dYr = torch.randn(T, d, device="cuda", generator=g).to(torch.bfloat16)
    dYo = torch.empty_like(dYr)
    dgam = torch.empty(d, dtype=torch.float32, device="cuda")
    ws_b = resbm.workspace(desc, resbm.RESBM_OP_RMSNORM_BWD)
    Yl = Y.detach().clone().requires_grad_(True)
    gl = gamma.detach().clone().requires_grad_(True)

    def torch_bwd():
        n = torch.nn.functional.rms_norm(Yl, (d,), gl, eps)
        gy, gg = torch.autograd.grad(n, (Yl, gl), dN)
        return gy + dYr, gg

    bruns = {"norm_bwd_resbm": lambda: resbm.resbm_rmsnorm_bwd(desc, Y, gamma, eps, dN, dYr, dYo, dgam, ws_b),
             "norm_bwd_torch_then_add": torch_bwd}
    balg = {"norm_bwd_resbm": 4 * T * d * 2 + 2 * d + 4 * d, "norm_bwd_torch_then_add": None}
    for name, fn in bruns.items():
        for _ in range(warmup):
            fn()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(steps):
            fn()
        b.record()
        torch.cuda.synchronize()
        ms = a.elapsed_time(b) / steps
        res[name] = {"ms": ms}
        if balg[name]:
            gbs = balg[name] / (ms / 1e3) / 1e9
            res[name].update(alg_bytes=balg[name], GBps=gbs, frac=gbs / peaks["hbm_gbs"])
    return res


def pipeline_workload(torch, steps=3, warmup=2):
    """The simulated 4-stage pipeline: one training step (forward + backward) of the 24-layer
    transformer with three ResBM boundaries; the boundary kernels' share of the step time."""
    from paper_2604_11947_gb300 import pipeline
    cfg = pipeline.PIPELINE
    tokens = pipeline.synthetic_tokens(cfg)
    model = pipeline.PipelineModel(cfg)
    step_ms, bnd_ms, loss = pipeline.time_steps(model, tokens, steps, warmup)
    del model
    # the same model with the receiving blocks' RMSNorm run by torch after the decoder
    model = pipeline.PipelineModel(cfg.with_(fuse_norm=False))
    step_u, bnd_u, loss_u = pipeline.time_steps(model, tokens, steps, warmup)
    del model
    return {"workload": "%d-layer pre-norm decoder (d=%d, %d heads, SwiGLU %d, vocab %d, bf16) in %d "
                        "stages with a ResBM boundary (r=%d, m=%d, merge=1) between consecutive stages, "
                        "each receiving block's pre-attention RMSNorm fused into the decoder; "
                        "batch %d x seq %d uniform random token ids; one training step (forward + "
                        "backward, no optimizer update)"
                        % (cfg.layers, cfg.d, cfg.heads, cfg.ffn, cfg.vocab, cfg.stages, cfg.r, cfg.m,
                           cfg.batch, cfg.seq),
            "steps": steps, "warmup": warmup, "ms_per_step": step_ms,
            "value": cfg.tokens / (step_ms / 1e3), "unit": "tokens/s",
            "boundary_ms_per_step": bnd_ms, "boundary_share": bnd_ms / step_ms,
            "boundaries": cfg.stages - 1, "loss": loss,
            "unfused_norm": {"ms_per_step": step_u, "boundary_ms_per_step": bnd_u, "loss": loss_u},
            "timing": "CUDA events around the K steps and around every boundary C-ABI call "
                      "(12 per step: encode/decode forward and backward of 3 boundaries; with the fused "
                      "norm the decoder forward's call includes the norm)"}


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
    resbm.load()

    if args.rmsnorm_only:
        print(json.dumps(decode_rmsnorm_workload(resbm, torch, measured_peaks(), steps=max(args.steps, 1),
                                                 warmup=max(args.warmup, 0))), flush=True)
        return
    if args.hbm_forms_only:   # one GPU's memory system: rank 0 alone measures and prints
        if rank == 0:
            print(json.dumps(hbm_forms(resbm, torch, reps=max(args.steps, 1), warmup=max(args.warmup, 0),
                                       sampler=ClockSampler())), flush=True)
        if dist:
            dist.destroy_process_group()
        return
    if args.ffn_only:
        print(json.dumps(ffn_encode_workload(resbm, torch, steps=max(args.steps, 1), warmup=max(args.warmup, 0))),
              flush=True)
        return
    flags = resbm.RESBM_FLAG_GENERIC if args.generic else 0
    peaks = measured_peaks()
    dev = device_inputs(cfg, torch)
    w = Workload(cfg, flags, dev, resbm, torch)
    w.warm(args.warmup)

    props = torch.cuda.get_device_properties(local)
    uuid = getattr(props, "uuid", None)
    uuid = None if uuid is None else (str(uuid) if str(uuid).startswith("GPU-") else "GPU-" + str(uuid))
    clocks = ClockSampler(uuid)
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    clocks.start()
    time.sleep(0.15)
    # timed region: K boundary steps through the library's step call
    ms_total, launches = w.time_steps(args.steps)
    # second timed pass, same K steps as four op calls with events between them: the per-op
    # times of the roofline (these steps are a few percent slower than the ones above)
    op_ms = w.time_ops(args.steps)
    if dist:
        dist.barrier()
    clk = clocks.stop()
    ms_total = max_over_ranks(ms_total, dist, "cuda")
    ms_step = ms_total / max(args.steps, 1)
    value = job_throughput(cfg.T, world, args.steps, ms_total)

    bytes_ = op_bytes(cfg)
    per_op = per_op_table(cfg, op_ms, peaks)
    dom = max(OPS, key=lambda o: op_ms[o])
    worst = min(OPS, key=lambda o: per_op[o]["frac"])
    achieved = per_op[dom]["GBps"]
    step_bytes = sum(bytes_.values())
    roofline = {"bound": "hbm", "kernel": dom, "achieved": achieved, "peak": peaks["hbm_gbs"],
                "unit": "GB/s", "frac": achieved / peaks["hbm_gbs"],
                "frac_of_8TBps": achieved / NOMINAL_HBM_GBS,
                "traffic": traffic_for(dom, cfg),
                "peak_source": peaks["source"] + " copy bandwidth (MEASURED_PEAKS.json hbm_gbs)",
                "algorithmic_bytes_per_launch": bytes_[dom],
                "timing": "per-op CUDA events on the launching stream in a second timed pass "
                          "of the same K steps (op calls with events between them)",
                "min_op": worst, "min_op_frac": per_op[worst]["frac"],
                "min_op_frac_of_8TBps": per_op[worst]["frac_of_8TBps"],
                "target": "every op >= %.2f of peak HBM" % TARGET_FRAC,
                "target_met_of_measured": all(v["frac"] >= TARGET_FRAC for v in per_op.values()),
                "target_met_of_8TBps": all(v["frac_of_8TBps"] >= TARGET_FRAC for v in per_op.values()),
                "per_op": per_op,
                "step_GBps": step_bytes / (ms_step / 1e3) / 1e9}

    e2e = None
    if not args.no_e2e:
        e2e = run_e2e(args, cfg, w, resbm, torch, dist, world)
    del w

    extra = None
    if rank == 0 and world == 1 and not args.no_extra and not args.tokens:
        del dev
        torch.cuda.empty_cache()
        extra = {}
        k_extra, w_extra = max(3, min(args.steps, 50)), max(3, min(args.warmup, 5))
        extra["single_bf16"], _ = extra_workload("single_bf16", synth.CONFIGS["single_bf16"], flags, resbm,
                                                 torch, k_extra, w_extra, peaks)
        reuse = None
        for name in ("sweep_r32", "sweep_r64", "sweep_r128", "sweep_r512"):
            extra[name], reuse = extra_workload(name, synth.CONFIGS[name], flags, resbm, torch,
                                                k_extra, w_extra, peaks, reuse)
        del reuse
        torch.cuda.empty_cache()
        extra["ffn_down_encode"] = ffn_encode_workload(resbm, torch)
        torch.cuda.empty_cache()
        extra["decode_fwd_rmsnorm"] = decode_rmsnorm_workload(resbm, torch, peaks)
        torch.cuda.empty_cache()
        extra["pipeline"] = pipeline_workload(torch)
        torch.cuda.empty_cache()
        extra["hbm_forms"] = hbm_forms(resbm, torch)
        from paper_2604_11947_gb300 import pipeline
        conv = pipeline.convergence()
        conv["workload"] = ("loss curves (step, mean loss over the previous 25 steps) of a 4-layer "
                            "decoder (d=512, 8 heads, SwiGLU 1024, vocab 256) in 2 stages with one "
                            "ResBM boundary (r=16, 32x) wired as reading A (pad(b) + D(b) into the "
                            "block) and reading B (D(b) into the attention branch, pad(b) its skip), "
                            "and the same model in 1 stage (no boundary); AdamW lr 1e-3, batch 16 x "
                            "seq 256 of a seeded random Markov stream (4 successors per token)")
        extra["convergence"] = conv
        torch.cuda.empty_cache()

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
    if extra is not None:
        line["workloads"] = extra
    if rank == 0 and world == 1 and not args.no_cpu:
        line["cpu_baseline"] = cpu_baseline(cfg)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()


def hbm_forms(resbm, torch, gib=1, reps=10, warmup=3, sampler=None):
    """The HBM rate each access form of resbm_measure_hbm_form attains on this device: every form
    over `gib` GiB buffers (above the 129 MB L2, so no flush), `warmup` untimed launches, then
    `reps` launches each timed with CUDA events on the launching stream; GB/s of the bytes the
    form moves (reads + writes), median and best. `sampler`: a ClockSampler to run around it."""
    n = gib << 30
    a = torch.full((n,), 0x3C, dtype=torch.uint8, device="cuda")
    b = torch.zeros(n, dtype=torch.uint8, device="cuda")
    s = torch.cuda.current_stream()
    if sampler is not None:
        torch.cuda.synchronize()
        sampler.start()
        time.sleep(0.15)
    out = {}
    for name in resbm.HBM_FORMS:
        for _ in range(warmup):
            resbm.resbm_measure_hbm_form(name, a, b)
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(reps)]
        for e0, e1 in ev:
            e0.record(s)
            resbm.resbm_measure_hbm_form(name, a, b)
            e1.record(s)
        torch.cuda.synchronize()
        ms = sorted(e0.elapsed_time(e1) for e0, e1 in ev)
        moved = 2 * n if name.startswith("copy") else n
        out[name] = {"GBps_median": moved / (statistics.median(ms) / 1e3) / 1e9,
                     "GBps_best": moved / (ms[0] / 1e3) / 1e9, "ms_median": statistics.median(ms),
                     "moved_bytes": moved}
    res = {"forms": out, "buffer_bytes": n, "reps": reps, "warmup": warmup,
           "device_error": resbm.resbm_device_error(),
           "how": "one launch per timed rep, CUDA events on the launching stream; the forms are those of "
                  "include/resbm.h resbm_hbm_form"}
    if sampler is not None:
        res["clocks"] = sampler.stop()
    del a, b
    torch.cuda.empty_cache()
    return res


def host_link(torch, mib=512, reps=3):
    """The host link's copy rates with page-locked buffers (GB/s, best of `reps`): host to device
    and device to host alone on one stream, and both at once on two streams (the floor of the
    host-buffer step: its bytes each way over these rates)."""
    n = mib << 20
    h_in = torch.empty(n, dtype=torch.uint8).pin_memory()
    h_out = torch.empty(n, dtype=torch.uint8).pin_memory()
    d_in = torch.empty(n, dtype=torch.uint8, device="cuda")
    d_out = torch.empty(n, dtype=torch.uint8, device="cuda")
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()

    def timed(fn):
        best = float("inf")
        for _ in range(reps):
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            fn()
            torch.cuda.synchronize()
            best = min(best, time.perf_counter() - t0)
        return best

    t_h2d = timed(lambda: d_in.copy_(h_in, non_blocking=True))
    t_d2h = timed(lambda: h_out.copy_(d_out, non_blocking=True))

    def both():
        with torch.cuda.stream(s1):
            d_in.copy_(h_in, non_blocking=True)
        with torch.cuda.stream(s2):
            h_out.copy_(d_out, non_blocking=True)

    t_both = timed(both)
    return {"h2d_GBps": n / t_h2d / 1e9, "d2h_GBps": n / t_d2h / 1e9, "bidirectional_each_GBps": n / t_both / 1e9,
            "bytes": n, "how": "torch copies between page-locked host and device buffers, best of %d" % reps}


def run_e2e(args, cfg, w, resbm, torch, dist, world):
    """The same step through the C ABI with HOST buffers (resbm_boundary_step_host): inputs in
    pinned host memory, results back into pinned host memory, every copy inside the call and
    inside the timed region. The step is the one `value` times, dX[:, :r] += dB included (a
    pinned host dX whose first r columns travel in and back). Two calls are kept in flight (two
    streams, two device workspaces, two sets of host results), so one step's results travel back
    while the next step's inputs travel in, as a training loop fed from the host would run them."""
    desc, dev, out = w.desc, w.dev, w.out
    ins = ("X", "F", "dY", "We1", "We2", "Wd1", "Wd2")
    res = ("B", "Y", "dB", "dF", "dWe1", "dWe2", "dWd1", "dWd2")
    host_in = {k: dev[k].cpu().pin_memory() for k in ins}
    host_out = [{k: torch.empty(out[k].shape, dtype=out[k].dtype).pin_memory() for k in res}
                for _ in range(2)]
    for h in host_out:   # the residual gradient dX[:, :r] += dB accumulates into
        h["dX"] = torch.zeros(out["dX"].shape, dtype=out["dX"].dtype).pin_memory()
    wss = [resbm.workspace(desc, resbm.RESBM_OP_BOUNDARY_STEP_HOST) for _ in range(2)]
    streams = [torch.cuda.Stream() for _ in range(2)]
    # call k+1's copies in wait for call k's (resbm_step_args.wait_before_inputs / inputs_done):
    # one call's inputs travel in while the previous call's results travel out
    in_done = [torch.cuda.Event() for _ in range(2)]
    for ev, st in zip(in_done, streams):
        ev.record(st)
    es = host_in["F"].element_size()
    cols = cfg.T * cfg.r * es   # X[:, :r] and dX[:, :r]: the only columns of X and dX the step uses
    # what the call copies: X[:, :r], dX[:, :r], F, dY and the weights in; the results and
    # dX[:, :r] out
    h2d = 2 * cols + sum(host_in[k].numel() * es for k in ins if k != "X")
    d2h = cols + sum(host_out[0][k].numel() * host_out[0][k].element_size() for k in res)
    # 300 steps (≈2.3 s) whatever --steps is: the host link sometimes stalls for ~100 ms (seen as
    # 30-55 ms gaps between consecutive steps whose steady pace is 6.5 ms); a short window would
    # charge one such burst to a handful of steps, so the window is long enough to average them
    n = 300

    def step(i):
        b = i % 2
        resbm.resbm_boundary_step_host(desc, wss[b], stream=streams[b], wait_before_inputs=in_done[1 - b],
                                       inputs_done=in_done[b], **host_in, **host_out[b])

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
            "ms_per_step": ms / n, "host_link": host_link(torch),
            "api": "resbm_boundary_step_host (host buffers; copies inside the call; dX[:, :r] += dB)",
            "pipelined": "two calls in flight on two streams with two device workspaces, each call's "
                         "copies in chained after the previous call's (events); host wall clock from the "
                         "first copy to the last result on the host"}


if __name__ == "__main__":
    main()
