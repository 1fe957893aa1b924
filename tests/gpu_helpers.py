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


def sample_tokens(T, n, seed=0, tile=128):
    """Tokens to check at full size: the ends, both sides of tile edges, and random ones."""
    rng = np.random.default_rng(seed)
    fixed = {0, 1, T - 1, T - 2}
    for t in (tile - 1, tile, 2 * tile - 1, T // 2, T // 2 + 1, T - tile, T - tile - 1):
        if 0 <= t < T:
            fixed.add(t)
    rest = rng.choice(T, size=min(T, max(0, n - len(fixed))), replace=False)
    return np.array(sorted(fixed | set(int(x) for x in rest)))
