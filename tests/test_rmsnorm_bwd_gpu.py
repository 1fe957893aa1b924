"""resbm_rmsnorm_bwd (the receiving block's RMSNorm backward with the residual gradient added)
through the C ABI against the oracle's chain rule, on the vector and the scalar paths, in place
and out of place, bitwise reproducible."""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import to_dev, to_host
from metrics import check
from paper_2604_11947_gb300 import resbm, synth

pytestmark = pytest.mark.gpu
EPS = 1e-5

CASES = {
    "d512": synth.BoundaryConfig("nb_d512", T=1000, d=512, r=32, m=32),
    "d2048_pipeline": synth.BoundaryConfig("nb_d2048", T=16384, d=2048, r=16, m=16),
    "d100_scalar": synth.BoundaryConfig("nb_d100", T=129, d=100, r=3, m=7),      # d % 8 != 0: one element a thread
    "f32": synth.BoundaryConfig("nb_f32", T=333, d=200, r=8, m=5, dtype="f32"),
    "d16384_max": synth.BoundaryConfig("nb_d16384", T=5, d=16384, r=32, m=32),
    "one_row": synth.BoundaryConfig("nb_one", T=1, d=64, r=32, m=32),
    "rows_lt_blocks": synth.BoundaryConfig("nb_300", T=300, d=768, r=16, m=16),   # fewer rows than blocks
    # rows held in registers with 1, 2 and 4 vectors a thread (d = 2048 above: 1), the last one partial
    "d3000_two_vectors": synth.BoundaryConfig("nb_d3000", T=777, d=3000, r=8, m=8),
    "d6144_four_vectors": synth.BoundaryConfig("nb_d6144", T=77, d=6144, r=32, m=32),
}


def _inputs(cfg):
    h = {"Y": synth.tensor(cfg, "X"), "dN": synth.tensor(cfg, "dY"), "dY": synth.tensor(cfg, "dX0"),
         "gamma": synth.tensor(cfg, "gamma")[0]}
    return h, {k: to_dev(v, cfg) for k, v in h.items()}


def _run(cfg, dev, dY="given", out=None):
    desc = resbm.desc_from_config(cfg)
    dY_in = dev["dY"] if dY == "given" else None
    dY_out = torch.empty_like(dev["Y"]) if out is None else out
    dg = torch.empty(cfg.d, dtype=torch.float32, device="cuda")
    ws = resbm.workspace(desc, resbm.RESBM_OP_RMSNORM_BWD)
    resbm.resbm_rmsnorm_bwd(desc, dev["Y"], dev["gamma"], EPS, dev["dN"], dY_in, dY_out, dg, ws)
    torch.cuda.synchronize()
    return dY_out, dg


@pytest.mark.parametrize("name", CASES)
def test_rmsnorm_bwd_matches_oracle(name):
    cfg = CASES[name]
    h, dev = _inputs(cfg)
    dYo, dg = _run(cfg, dev)
    wdY, wdg = oracle.rmsnorm_bwd(h["Y"], h["gamma"], EPS, h["dN"], h["dY"])
    check("dY_out", to_host(dYo), wdY, cfg.dtype)
    check("dgamma", to_host(dg), wdg, cfg.dtype)
    # without an incoming gradient; then in place over a copy of dY; and reproducible
    dYo0, dg0 = _run(cfg, dev, dY=None)
    check("dY_out", to_host(dYo0), oracle.rmsnorm_bwd(h["Y"], h["gamma"], EPS, h["dN"])[0], cfg.dtype)
    assert torch.equal(dg0, dg)
    buf = dev["dY"].clone()
    dev_inplace = dict(dev, dY=buf)
    dYi, dgi = _run(cfg, dev_inplace, out=buf)
    assert torch.equal(dYi, dYo) and torch.equal(dgi, dg)
    dYo2, dg2 = _run(cfg, dev)
    assert torch.equal(dYo2, dYo) and torch.equal(dg2, dg)
    assert resbm.resbm_device_error() == 0


@pytest.mark.slow
def test_rmsnorm_bwd_headline_shape():
    """T = 65536, d = 4096: every element of dY_out and dgamma against the oracle."""
    cfg = synth.CONFIGS["large_bf16"]
    h, dev = _inputs(cfg)
    dYo, dg = _run(cfg, dev)
    wdY, wdg = oracle.rmsnorm_bwd(h["Y"], h["gamma"], EPS, h["dN"], h["dY"])
    check("dY_out", to_host(dYo), wdY, "bf16")
    check("dgamma", to_host(dg), wdg, "bf16")
