"""Seeded synthetic inputs for the ResBM boundary bottleneck.

This module holds no arithmetic of the bottleneck itself: it only draws the numbers that
both the CUDA path and the fp64 oracle consume.

Generator (counter-based, so any slice of any tensor can be drawn on its own and the result
does not depend on chunking or thread count):

  mix64(z)        the SplitMix64 output function (Steele, Lea & Flood, OOPSLA 2014):
                  z ^= z >> 30; z *= 0xBF58476D1CE4E5B9; z ^= z >> 27; z *= 0x94D049BB133111EB;
                  z ^= z >> 31                                   (all arithmetic mod 2^64)
  key(s, id)      mix64(mix64(s + G) + id * G),  G = 0x9E3779B97F4A7C15
  word(s, id, c)  mix64(key(s, id) + (c + 1) * G)                (the SplitMix64 stream at c)
  normal(s,id,i)  Box-Muller on the pair j = i // 2 of 53-bit uniforms:
                  u1 = ((word(2j) >> 11) + 1) * 2^-53 in (0, 1],  u2 = (word(2j+1) >> 11) * 2^-53
                  n  = sqrt(-2 ln u1) * cos(2 pi u2)  for even i,  ... * sin(2 pi u2)  for odd i

Tensors (row-major, element index i = row * cols + col):
  X, F   N(0,1); with token_scale, row t of both is multiplied by s_t = exp(0.5 * normal(s, 8, t))
         (a log-normal(0, 0.5) spread of per-token norms, like a residual stream)
  dY     N(0,1)                      dB, dX0 (stand-alone encoder backward inputs) N(0,1)
  We1 N(0,1/d)  We2 N(0,1/m)  Wd1 N(0,1/r)  Wd2 N(0,1/m)        (N(0, 1/fan_in))
Values are produced in fp64, rounded to fp32 and, for bf16 workloads, rounded to bf16
(round-to-nearest-even); they are returned as fp32 arrays holding exactly those values.
"""
from __future__ import annotations

import os
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, replace

import numpy as np

TENSOR_IDS = {"X": 1, "F": 2, "dY": 3, "We1": 4, "We2": 5, "Wd1": 6, "Wd2": 7,
              "scale": 8, "dB": 9, "dX0": 10, "matrix": 11, "gamma": 12}


def matrix(rows: int, cols: int, seed: int = 0) -> np.ndarray:
    """A rows x cols matrix of N(0,1) draws (fp64) for the weight-matrix utilities; seed selects
    the stream."""
    return normal(seed, TENSOR_IDS["matrix"], 0, rows * cols).reshape(rows, cols)

_G = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)


def _mix64_(z: np.ndarray) -> np.ndarray:
    """In-place SplitMix64 output function on a uint64 array."""
    t = z >> np.uint64(30)
    z ^= t
    z *= _M1
    np.right_shift(z, np.uint64(27), out=t)
    z ^= t
    z *= _M2
    np.right_shift(z, np.uint64(31), out=t)
    z ^= t
    return z


def _key(seed: int, tensor_id: int) -> np.uint64:
    s = np.array([seed], dtype=np.uint64)
    s += _G
    _mix64_(s)
    s += np.uint64((tensor_id * 0x9E3779B97F4A7C15) % (1 << 64))
    return _mix64_(s)[0]


def words(seed: int, tensor_id: int, c0: int, n: int) -> np.ndarray:
    """The raw 64-bit words word(seed, tensor_id, c) for c in [c0, c0 + n)."""
    z = np.arange(c0 + 1, c0 + 1 + n, dtype=np.uint64)
    z *= _G
    z += _key(seed, tensor_id)
    return _mix64_(z)


def _uniform53(w: np.ndarray, plus_one: bool) -> np.ndarray:
    w >>= np.uint64(11)
    if plus_one:
        w += np.uint64(1)
    u = w.astype(np.float64)
    u *= 2.0 ** -53
    return u


def normal(seed: int, tensor_id: int, i0: int, n: int) -> np.ndarray:
    """fp64 standard normals for element indices [i0, i0 + n) of one tensor."""
    if n <= 0:
        return np.empty(0, np.float64)
    j0, j1 = i0 // 2, (i0 + n - 1) // 2 + 1
    w = words(seed, tensor_id, 2 * j0, 2 * (j1 - j0))
    rad = _uniform53(w[0::2].copy(), True)
    np.log(rad, out=rad)
    rad *= -2.0
    np.sqrt(rad, out=rad)
    theta = _uniform53(w[1::2].copy(), False)
    theta *= 2.0 * np.pi
    out = np.empty(2 * (j1 - j0), np.float64)
    np.cos(theta, out=out[0::2])
    np.sin(theta, out=out[1::2])
    out[0::2] *= rad
    out[1::2] *= rad
    return out[i0 - 2 * j0: i0 - 2 * j0 + n]


def round_bf16(x32: np.ndarray) -> np.ndarray:
    """Round fp32 values to the nearest bf16 (ties to even); returned as fp32."""
    u = np.ascontiguousarray(x32, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = (u + np.uint64(0x7FFF) + ((u >> np.uint64(16)) & np.uint64(1))) & np.uint64(0xFFFF0000)
    return u.astype(np.uint32).view(np.float32)


@dataclass(frozen=True)
class BoundaryConfig:
    """One boundary workload: T tokens of width d compressed to r (hidden width m)."""
    name: str
    T: int
    d: int
    r: int
    m: int
    dtype: str = "bf16"          # "bf16" or "f32": I/O and weight dtype
    act: str = "silu"
    merge: int = 1
    token_scale: bool = True      # log-normal(0, 0.5) per-token spread of X and F
    seed: int = 0

    @property
    def compression(self) -> float:
        return self.d / self.r

    def with_(self, **kw) -> "BoundaryConfig":
        return replace(self, **kw)


# The workloads the boundary op is measured and checked on (m = r, see the design notes).
CONFIGS = {
    # batch 4 x seq 128, 128x compression, fp32 I/O
    "tiny_f32": BoundaryConfig("tiny_f32", T=512, d=256, r=2, m=2, dtype="f32", token_scale=False),
    # batch 8 x seq 2048, 128x
    "single_bf16": BoundaryConfig("single_bf16", T=16384, d=2048, r=16, m=16),
    # batch 32 x seq 2048, 128x: the headline roofline workload
    "large_bf16": BoundaryConfig("large_bf16", T=65536, d=4096, r=32, m=32),
    # compression-ratio sweep at d = 8192, T = 32768 (16x .. 256x)
    "sweep_r512": BoundaryConfig("sweep_r512", T=32768, d=8192, r=512, m=512),
    "sweep_r128": BoundaryConfig("sweep_r128", T=32768, d=8192, r=128, m=128),
    "sweep_r64": BoundaryConfig("sweep_r64", T=32768, d=8192, r=64, m=64),
    "sweep_r32": BoundaryConfig("sweep_r32", T=32768, d=8192, r=32, m=32),
}


def shapes(cfg: BoundaryConfig) -> dict:
    T, d, r, m = cfg.T, cfg.d, cfg.r, cfg.m
    return {"X": (T, d), "F": (T, d), "dY": (T, d), "dB": (T, r), "dX0": (T, d),
            "We1": (d, m), "We2": (m, r), "Wd1": (r, m), "Wd2": (m, d), "gamma": (1, d)}


def _std(cfg: BoundaryConfig, name: str) -> float:
    fan_in = {"We1": cfg.d, "We2": cfg.m, "Wd1": cfg.r, "Wd2": cfg.m}.get(name)
    return 1.0 if fan_in is None else 1.0 / np.sqrt(fan_in)


def _finish(cfg: BoundaryConfig, v64: np.ndarray) -> np.ndarray:
    v32 = v64.astype(np.float32)
    return round_bf16(v32) if cfg.dtype == "bf16" else v32


def token_scales(cfg: BoundaryConfig, t0: int, t1: int) -> np.ndarray:
    if not cfg.token_scale:
        return np.ones(t1 - t0, np.float64)
    return np.exp(0.5 * normal(cfg.seed, TENSOR_IDS["scale"], t0, t1 - t0))


def rows(cfg: BoundaryConfig, name: str, t0: int, t1: int) -> np.ndarray:
    """Rows [t0, t1) of one tensor, as fp32 holding I/O-dtype values."""
    nrows, ncols = shapes(cfg)[name]
    t1 = min(t1, nrows)
    v = normal(cfg.seed, TENSOR_IDS[name], t0 * ncols, (t1 - t0) * ncols).reshape(t1 - t0, ncols)
    if name in ("X", "F"):
        v *= token_scales(cfg, t0, t1)[:, None]
    elif name == "gamma":   # an RMSNorm weight: near 1, as trained norm weights sit
        v = 1.0 + 0.1 * v
    else:
        v *= _std(cfg, name)
    return _finish(cfg, v)


def rows_at(cfg: BoundaryConfig, name: str, idx) -> np.ndarray:
    """Selected rows (any order) of one tensor."""
    return np.concatenate([rows(cfg, name, int(t), int(t) + 1) for t in idx], axis=0)


def tensor(cfg: BoundaryConfig, name: str, threads: int | None = None,
           chunk_elems: int = 1 << 18, nrows: int | None = None) -> np.ndarray:
    """A whole tensor (or its first nrows rows), drawn in row chunks on a thread pool (numpy
    releases the GIL)."""
    full_rows, ncols = shapes(cfg)[name]
    nrows = full_rows if nrows is None else min(nrows, full_rows)
    step = max(1, chunk_elems // max(1, ncols))
    out = np.empty((nrows, ncols), np.float32)
    starts = list(range(0, nrows, step))

    def work(t0):
        t1 = min(t0 + step, nrows)
        out[t0:t1] = rows(cfg, name, t0, t1)

    if len(starts) == 1:
        work(0)
    else:
        with ThreadPoolExecutor(max_workers=threads or min(32, os.cpu_count() or 1)) as ex:
            list(ex.map(work, starts))
    return out


def inputs(cfg: BoundaryConfig, names=("X", "F", "dY", "We1", "We2", "Wd1", "Wd2")) -> dict:
    return {n: tensor(cfg, n) for n in names}
