"""resbm_ffn_down_encode_fwd (the encoder fused into the FFN down-projection) through the C ABI
against the oracle (the down-projection in float64, rounded to bf16, then the encoder)."""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import to_host
from metrics import check
from paper_2604_11947_gb300 import resbm, synth

pytestmark = pytest.mark.gpu

CASES = {
    # T, f, d, r, m
    "small": (1000, 1024, 512, 32, 32),
    "odd": (333, 200, 776, 24, 16),              # partial tiles along T, d and the FFN width
    "pipeline": (16384, 5632, 2048, 16, 16),     # the fifth workload's boundary: d = 2048, SwiGLU 5632
}


def _inputs(T, f, d, r, m):
    cfg = synth.BoundaryConfig("ffn", T=T, d=d, r=r, m=m)
    bf = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to("cuda").to(torch.bfloat16)
    H = bf(synth.matrix(T, f, seed=11) * 0.5)
    W2 = bf(synth.matrix(f, d, seed=12) / np.sqrt(f))
    return cfg, H, W2, bf(synth.tensor(cfg, "X")), bf(synth.tensor(cfg, "We1")), bf(synth.tensor(cfg, "We2"))


@pytest.mark.parametrize("case", CASES)
def test_fused_down_projection_encoder_matches_oracle(case):
    T, f, d, r, m = CASES[case]
    cfg, H, W2, X, We1, We2 = _inputs(T, f, d, r, m)
    desc = resbm.desc_from_config(cfg)
    ws = resbm.ffn_down_encode_workspace(desc, f)
    B = torch.empty(T, r, dtype=torch.bfloat16, device="cuda")
    P = torch.empty(T, m, dtype=torch.float32, device="cuda")
    F = torch.empty(T, d, dtype=torch.bfloat16, device="cuda")
    resbm.resbm_ffn_down_encode_fwd(desc, H, W2, X, We1, We2, B, P, F, ws)
    # without F_out and P: the same B bit for bit (F never leaves the chip)
    B2 = torch.empty_like(B)
    resbm.resbm_ffn_down_encode_fwd(desc, H, W2, X, We1, We2, B2, None, None, ws)
    torch.cuda.synchronize()
    assert torch.equal(B, B2)
    wB, wP, wF = oracle.ffn_down_encode_fwd(to_host(H), to_host(W2), to_host(X), to_host(We1), to_host(We2), cfg.act)
    check("F", to_host(F), wF, "bf16")
    check("B", to_host(B), wB, "bf16")
    # P: fp32 sums of F . We1 (d terms) from the GPU's bf16 F. F's fp32 down-projection error is
    # relative to the size of its f terms, not to F, so on the elements that cancel toward zero it
    # moves F's bf16 rounding to the neighbouring value: measured on ~20 % of F (one spacing,
    # 2^-8 of the element). Carried through We1 that is sqrt(0.2 d) x 2^-8 x E|F| x rms(We1) ~ 1.4e-3
    # of P's RMS per element, ~6e-3 for the largest of 2.6e5 (measured up to 2e-3): bound 1e-2
    check("P", to_host(P), wP, "f32", tol=1e-2)
    assert resbm.resbm_device_error() == 0
