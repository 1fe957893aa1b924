"""Shared helpers of the GPU parity tests: run the CUDA path through the C ABI and the oracle
on the same seeded inputs."""
import numpy as np
import torch

import oracle
from paper_2604_11947_gb300 import resbm, synth

INPUTS = ("X", "F", "dY", "We1", "We2", "Wd1", "Wd2")


def torch_dtype(cfg):
    return torch.bfloat16 if cfg.dtype == "bf16" else torch.float32


def to_dev(a, cfg):
    return torch.from_numpy(np.ascontiguousarray(a)).to("cuda").to(torch_dtype(cfg))


def to_host(t):
    return t.detach().float().cpu().numpy().astype(np.float64)


def host_inputs(cfg, names=INPUTS):
    return {n: synth.tensor(cfg, n) for n in names}


def gpu_step(cfg, dev, flags=0, with_dX=True, with_P=True, dX0=None):
    """One resbm_boundary_step on device inputs `dev` (dict of torch tensors)."""
    desc = resbm.desc_from_config(cfg, flags)
    out = resbm.step_outputs(desc, with_dX=with_dX)
    if with_dX and dX0 is not None:
        out["dX"].copy_(dX0)
    if not with_P:
        out.pop("P")
    ws = resbm.workspace(desc, resbm.RESBM_OP_BOUNDARY_STEP)
    resbm.resbm_boundary_step(desc, ws, **{k: dev[k] for k in INPUTS}, **out)
    torch.cuda.synchronize()
    return out


def oracle_step(cfg, h):
    """The oracle's boundary step; B and dB cross the boundary rounded to the I/O dtype."""
    return oracle.boundary_step(h["X"], h["F"], h["dY"], h["We1"], h["We2"], h["Wd1"], h["Wd2"],
                                act=cfg.act, merge=cfg.merge, transfer=cfg.dtype)


def check_output(name, got, want, cfg, dX0=None):
    """Compare one step output (torch tensor) with the oracle's (numpy). dX is compared on its
    first r columns (the identity-path gradient); its other columns must be untouched."""
    from metrics import check
    g = to_host(got)
    if name == "dX":
        base = np.zeros_like(g) if dX0 is None else np.asarray(dX0, np.float64)
        assert np.array_equal(g[:, cfg.r:], base[:, cfg.r:]), "dX columns >= r were modified"
        return check(name, g[:, :cfg.r], base[:, :cfg.r] + want[:, :cfg.r], cfg.dtype)
    return check(name, g, want, cfg.dtype)


def _ws(desc, op):
    return resbm.workspace(desc, op)


def gpu_stages(cfg, dev, want, flags=0, dX0=None):
    """The decoder (fwd + bwd) and the encoder backward run alone on the tensors that crossed the
    boundary in the oracle's step (its B and dB, already rounded to the I/O dtype), so that both
    sides take the transfer rounding of Appendix A.3 on the same values. Returns their outputs."""
    desc = resbm.desc_from_config(cfg, flags)
    T, d, r, m = cfg.T, cfg.d, cfg.r, cfg.m
    io = torch_dtype(cfg)
    B = to_dev(want["B"], cfg)
    dB_in = to_dev(want["dB"], cfg)
    out = dict(Y=torch.empty(T, d, dtype=io, device="cuda"), dB=torch.empty(T, r, dtype=io, device="cuda"),
               dWd1=torch.empty(r, m, device="cuda"), dWd2=torch.empty(m, d, device="cuda"),
               dF=torch.empty(T, d, dtype=io, device="cuda"),
               dX=torch.zeros(T, d, dtype=io, device="cuda") if dX0 is None else dX0.clone(),
               dWe1=torch.empty(d, m, device="cuda"), dWe2=torch.empty(m, r, device="cuda"))
    resbm.resbm_decode_fwd(desc, B, dev["Wd1"], dev["Wd2"], out["Y"], _ws(desc, resbm.RESBM_OP_DECODE_FWD))
    resbm.resbm_decode_bwd(desc, dev["dY"], B, dev["Wd1"], dev["Wd2"], out["dB"], out["dWd1"], out["dWd2"],
                           _ws(desc, resbm.RESBM_OP_DECODE_BWD))
    resbm.resbm_encode_bwd(desc, dB_in, dev["F"], None, dev["We1"], dev["We2"], out["dF"], out["dX"],
                           out["dWe1"], out["dWe2"], _ws(desc, resbm.RESBM_OP_ENCODE_BWD))
    torch.cuda.synchronize()
    return out


def assert_step_is_its_stages(cfg, dev, got, flags=0, dX0=None):
    """The boundary step hands its own B to the decoder and its own dB to the encoder backward:
    running those ops alone on the step's B and dB gives the step's outputs bit for bit."""
    desc = resbm.desc_from_config(cfg, flags)
    T, d, r, m = cfg.T, cfg.d, cfg.r, cfg.m
    io = torch_dtype(cfg)
    Y = torch.empty(T, d, dtype=io, device="cuda")
    resbm.resbm_decode_fwd(desc, got["B"], dev["Wd1"], dev["Wd2"], Y, _ws(desc, resbm.RESBM_OP_DECODE_FWD))
    dB = torch.empty(T, r, dtype=io, device="cuda")
    dWd1, dWd2 = torch.empty(r, m, device="cuda"), torch.empty(m, d, device="cuda")
    resbm.resbm_decode_bwd(desc, dev["dY"], got["B"], dev["Wd1"], dev["Wd2"], dB, dWd1, dWd2,
                           _ws(desc, resbm.RESBM_OP_DECODE_BWD))
    dF = torch.empty(T, d, dtype=io, device="cuda")
    dX = torch.zeros(T, d, dtype=io, device="cuda") if dX0 is None else dX0.clone()
    dWe1, dWe2 = torch.empty(d, m, device="cuda"), torch.empty(m, r, device="cuda")
    resbm.resbm_encode_bwd(desc, got["dB"], dev["F"], got.get("P"), dev["We1"], dev["We2"], dF,
                           dX if "dX" in got else None, dWe1, dWe2, _ws(desc, resbm.RESBM_OP_ENCODE_BWD))
    torch.cuda.synchronize()
    mine = dict(Y=Y, dB=dB, dWd1=dWd1, dWd2=dWd2, dF=dF, dX=dX, dWe1=dWe1, dWe2=dWe2)
    for k, v in mine.items():
        if k in got:
            assert torch.equal(v, got[k]), "step output %s differs from its stage run alone" % k
