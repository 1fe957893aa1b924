"""resbm_decode_fwd_rmsnorm (the decoder forward with the next block's pre-attention RMSNorm fused
in) through the C ABI against the oracle: Y = decode_fwd(B) and N = rmsnorm(Y as stored, gamma,
eps), on every path, with Y the same bits as resbm_decode_fwd's."""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import to_dev, to_host
from metrics import bf16_half_spacing, check
from paper_2604_11947_gb300 import resbm, synth

pytestmark = pytest.mark.gpu

PATHS = {"default": 0, "gemm": resbm.RESBM_FLAG_GEMM, "generic": resbm.RESBM_FLAG_GENERIC}
EPS = 1e-5

CASES = {
    # the fused kernels' widths (m = r in {16, 32, 64, 128}: NCH = 256 for m <= 32, else 128),
    # ragged token counts (a partial last tile), several tiles per CTA
    "r32": synth.BoundaryConfig("rn_r32", T=1000, d=512, r=32, m=32),
    "r16": synth.BoundaryConfig("rn_r16", T=777, d=768, r=16, m=16),
    "r64": synth.BoundaryConfig("rn_r64", T=300, d=256, r=64, m=64),
    "r128": synth.BoundaryConfig("rn_r128", T=260, d=512, r=128, m=128),
    "r32_gelu_merge0": synth.BoundaryConfig("rn_r32_g", T=515, d=1024, r=32, m=32, act="gelu_tanh", merge=0),
    # widths the fused kernels do not take: the GEMM chain / portable decoder, then the norm
    "r24_m40": synth.BoundaryConfig("rn_r24_m40", T=999, d=776, r=24, m=40),
    "odd": synth.BoundaryConfig("rn_odd", T=129, d=100, r=3, m=7),
    "f32": synth.BoundaryConfig("rn_f32", T=333, d=200, r=8, m=5, dtype="f32"),
    # one token, and a single partial tile
    "one_token": synth.BoundaryConfig("rn_one", T=1, d=512, r=32, m=32),
}


def _check_yn(cfg, Y, N, h, Wd2=None, eps=EPS):
    """Y and N against the oracle's exact chain (Y unrounded, N = rmsnorm(Y)). The GPU's N is
    rounded twice: Y to the output dtype before the norm reads it, then N. N's own rounding is
    the metric's h; Y's, carried through the row's factor rstd * gamma, is `allow`
    (bf16 only: fp32's rounding is far below its tolerance)."""
    wY, wN = oracle.decode_fwd_rmsnorm(h["B"], h["Wd1"], h["Wd2"] if Wd2 is None else Wd2, h["gamma"], eps,
                                       cfg.act, cfg.merge)
    check("Y", to_host(Y), wY, cfg.dtype)
    allow = None
    if cfg.dtype == "bf16":
        rstd = 1.0 / np.sqrt(np.mean(wY * wY, axis=1, keepdims=True) + eps)
        allow = bf16_half_spacing(wY) * np.abs(rstd * np.asarray(h["gamma"], np.float64)[None, :])
    check("N", to_host(N), wN, cfg.dtype, allow=allow)


def _inputs(cfg):
    B = synth.tensor(cfg, "dB")          # a T x r boundary tensor (the dB stream's draws)
    h = {"B": B, "Wd1": synth.tensor(cfg, "Wd1"), "Wd2": synth.tensor(cfg, "Wd2"),
         "gamma": synth.tensor(cfg, "gamma")[0]}
    dev = {k: to_dev(v, cfg) for k, v in h.items()}
    return h, dev


def _run(cfg, dev, flags=0, eps=EPS):
    desc = resbm.desc_from_config(cfg, flags)
    dt = torch.bfloat16 if cfg.dtype == "bf16" else torch.float32
    Y = torch.empty(cfg.T, cfg.d, dtype=dt, device="cuda")
    N = torch.empty(cfg.T, cfg.d, dtype=dt, device="cuda")
    ws = resbm.workspace(desc, resbm.RESBM_OP_DECODE_FWD_RMSNORM)
    resbm.resbm_decode_fwd_rmsnorm(desc, dev["B"], dev["Wd1"], dev["Wd2"], dev["gamma"], eps, Y, N, ws)
    torch.cuda.synchronize()
    return Y, N


@pytest.mark.parametrize("path", PATHS)
@pytest.mark.parametrize("name", CASES)
def test_decode_fwd_rmsnorm_matches_oracle(name, path):
    cfg = CASES[name]
    h, dev = _inputs(cfg)
    Y, N = _run(cfg, dev, PATHS[path])
    _check_yn(cfg, Y, N, h)
    # Y is the decoder forward's own output, bit for bit
    desc = resbm.desc_from_config(cfg, PATHS[path])
    Y2 = torch.empty_like(Y)
    resbm.resbm_decode_fwd(desc, dev["B"], dev["Wd1"], dev["Wd2"], Y2, resbm.workspace(desc, resbm.RESBM_OP_DECODE_FWD))
    torch.cuda.synchronize()
    assert torch.equal(Y, Y2)
    # and N is reproducible bit for bit (fixed-order row sums)
    _, N2 = _run(cfg, dev, PATHS[path])
    assert torch.equal(N, N2)
    assert resbm.resbm_device_error() == 0


def test_fused_and_unfused_norms_both_match_oracle():
    """The fused form (N from the recomputed fp32 values, the row RMS from fixed slots) and the GEMM
    chain's decoder followed by the norm over its stored Y, on the same inputs: both within the
    bound of the exact chain (they differ by the one rounding of Y the fused form skips)."""
    cfg = CASES["r32"]
    h, dev = _inputs(cfg)
    Yf, Nf = _run(cfg, dev, 0)
    Yg, Ng = _run(cfg, dev, resbm.RESBM_FLAG_GEMM)
    _check_yn(cfg, Yf, Nf, h)
    _check_yn(cfg, Yg, Ng, h)


def test_zero_second_layer_gives_normalised_identity_path():
    """Wd2 = 0 and merge = 1: Y = pad(B) exactly, N's first r columns B * rstd * gamma, the rest
    exactly zero."""
    cfg = CASES["r32"]
    h, dev = _inputs(cfg)
    dev["Wd2"] = torch.zeros_like(dev["Wd2"])
    Y, N = _run(cfg, dev, 0)
    r = cfg.r
    assert torch.equal(Y[:, :r], dev["B"]) and not torch.any(Y[:, r:])
    assert not torch.any(N[:, r:])
    _check_yn(cfg, Y, N, h, Wd2=np.zeros_like(h["Wd2"]))


def test_empty_token_count_is_a_no_op():
    cfg = synth.BoundaryConfig("rn_empty", T=0, d=512, r=32, m=32)
    desc = resbm.desc_from_config(cfg)
    w = {k: to_dev(synth.tensor(cfg, k), cfg) for k in ("Wd1", "Wd2")}
    g = to_dev(synth.tensor(cfg, "gamma")[0], cfg)
    e = torch.empty(0, device="cuda", dtype=torch.bfloat16)
    ws = resbm.workspace(desc, resbm.RESBM_OP_DECODE_FWD_RMSNORM)
    resbm.resbm_decode_fwd_rmsnorm(desc, e, w["Wd1"], w["Wd2"], g, EPS, e, e, ws)
    torch.cuda.synchronize()


@pytest.mark.slow
def test_headline_shape_every_element():
    """T = 65536, d = 4096, r = 32 (the bench's workload), in the launch configuration the bench
    times: every element of Y and N against the oracle."""
    cfg = synth.CONFIGS["large_bf16"]
    h, dev = _inputs(cfg)
    Y, N = _run(cfg, dev, 0)
    _check_yn(cfg, Y, N, h)
    assert resbm.resbm_device_error() == 0


@pytest.mark.parametrize("path", ["default", "generic"])
def test_linear_decoder_with_rmsnorm(path):
    """One linear layer per side (RESBM_FLAG_LINEAR: Y = pad(B) + B . Wd, Wd r x d; Wd1 absent):
    Y and N against the oracle's one-layer decoder followed by its norm."""
    cfg = synth.BoundaryConfig("rn_lin", T=700, d=512, r=32, m=32)
    flags = resbm.RESBM_FLAG_LINEAR | PATHS[path]
    B = synth.tensor(cfg, "dB")
    Wd = synth.tensor(cfg, "Wd2")[: cfg.r]          # r x d
    gamma = synth.tensor(cfg, "gamma")[0]
    desc = resbm.desc_from_config(cfg, flags)
    dB, dWd, dg = to_dev(B, cfg), to_dev(Wd, cfg), to_dev(gamma, cfg)
    Y = torch.empty(cfg.T, cfg.d, dtype=torch.bfloat16, device="cuda")
    N = torch.empty_like(Y)
    ws = resbm.workspace(desc, resbm.RESBM_OP_DECODE_FWD_RMSNORM)
    resbm.resbm_decode_fwd_rmsnorm(desc, dB, None, dWd, dg, EPS, Y, N, ws)
    torch.cuda.synchronize()
    wY = oracle.linear_decode_fwd(B, Wd, cfg.merge)
    check("Y", to_host(Y), wY, "bf16")
    rstd = 1.0 / np.sqrt(np.mean(wY * wY, axis=1, keepdims=True) + EPS)
    check("N", to_host(N), oracle.rmsnorm(wY, gamma, EPS), "bf16",
          allow=bf16_half_spacing(wY) * np.abs(rstd * np.asarray(gamma, np.float64)[None, :]))
    assert resbm.resbm_device_error() == 0
