"""resbm_boundary_step_host (every tensor in host memory) against resbm_boundary_step on device
copies of the same seeded inputs: the same kernels run on the same values, so every output
must agree bit for bit, and the parts of dX the step does not own must come back untouched."""
import numpy as np
import pytest
import torch

from gpu_helpers import host_inputs
from paper_2604_11947_gb300 import resbm, synth

pytestmark = pytest.mark.gpu

CASES = {
    # tensor-core kernels, several tiles and a ragged tail
    "bf16_tc": (synth.BoundaryConfig("hs_bf16", T=1000, d=512, r=32, m=32), 0),
    # portable kernels, fp32, odd sizes
    "f32_generic": (synth.BoundaryConfig("hs_f32", T=333, d=200, r=8, m=5, dtype="f32"), 0),
    # one linear layer per side (second-layer pointers NULL)
    "bf16_linear": (synth.BoundaryConfig("hs_lin", T=777, d=384, r=16, m=16), resbm.RESBM_FLAG_LINEAR),
}


def _io(cfg):
    return torch.bfloat16 if cfg.dtype == "bf16" else torch.float32


def _host_args(cfg, desc, flags, pinned, with_dX=True, with_P=True, seed=5):
    io = _io(cfg)
    h = {k: torch.from_numpy(np.ascontiguousarray(v)).to(io) for k, v in host_inputs(cfg).items()}
    out = {k: v.cpu() for k, v in resbm.step_outputs(desc, with_dX=with_dX).items()}
    if with_dX:
        g = torch.Generator().manual_seed(seed)
        out["dX"] = torch.randn(cfg.T, cfg.d, generator=g).to(io)
    if not with_P:
        out.pop("P")
    if flags & resbm.RESBM_FLAG_LINEAR:
        for k in ("We2", "Wd1"):
            h.pop(k)
        for k in ("dWe2", "dWd1"):
            out.pop(k)
    if pinned:
        h = {k: v.pin_memory() for k, v in h.items()}
        out = {k: v.pin_memory() for k, v in out.items()}
    return h, out


def _device_reference(desc, h, out0):
    dev = {k: v.to("cuda") for k, v in h.items()}
    out = {k: v.to("cuda") for k, v in out0.items()}
    ws = resbm.workspace(desc, resbm.RESBM_OP_BOUNDARY_STEP)
    resbm.resbm_boundary_step(desc, ws, **dev, **out)
    torch.cuda.synchronize()
    return {k: v.cpu() for k, v in out.items()}


def _same(got, want, dX0=None, r=None):
    for k in want:
        assert torch.equal(got[k], want[k]), k
    if dX0 is not None:
        assert torch.equal(got["dX"][:, r:], dX0[:, r:]), "dX columns >= r changed"


@pytest.mark.parametrize("pinned", [True, False], ids=["pinned", "pageable"])
@pytest.mark.parametrize("case", CASES)
def test_host_step_matches_device_step(case, pinned):
    cfg, flags = CASES[case]
    desc = resbm.desc_from_config(cfg, flags)
    h, out = _host_args(cfg, desc, flags, pinned)
    dX0 = out["dX"].clone()
    want = _device_reference(desc, h, out)
    ws = resbm.workspace(desc, resbm.RESBM_OP_BOUNDARY_STEP_HOST)
    resbm.resbm_boundary_step_host(desc, ws, **h, **out)
    torch.cuda.synchronize()
    _same(out, want, dX0, cfg.r)
    assert resbm.resbm_device_error() == 0


def test_host_step_without_dX_and_P():
    cfg, flags = CASES["bf16_tc"]
    desc = resbm.desc_from_config(cfg, flags)
    h, out = _host_args(cfg, desc, flags, True, with_dX=False, with_P=False)
    want = _device_reference(desc, h, out)
    ws = resbm.workspace(desc, resbm.RESBM_OP_BOUNDARY_STEP_HOST)
    resbm.resbm_boundary_step_host(desc, ws, **h, **out)
    torch.cuda.synchronize()
    _same(out, want)


def test_host_steps_on_two_streams_at_once():
    """Two calls in flight together (own streams, own workspaces, own host outputs), each
    followed by a second call on the same stream that must wait for the first."""
    cfg, flags = CASES["bf16_tc"]
    desc = resbm.desc_from_config(cfg, flags)
    runs = [_host_args(cfg, desc, flags, True, seed=s) for s in (1, 2)]
    wants = [_device_reference(desc, h, out) for h, out in runs]
    streams = [torch.cuda.Stream() for _ in runs]
    wss = [resbm.workspace(desc, resbm.RESBM_OP_BOUNDARY_STEP_HOST) for _ in runs]
    dX0 = [out["dX"].clone() for _, out in runs]
    for rep in range(2):
        for (h, out), st, ws, x0 in zip(runs, streams, wss, dX0):
            out["dX"].copy_(x0)   # host write: the previous call on this stream has finished
            resbm.resbm_boundary_step_host(desc, ws, stream=st, **h, **out)
        for st in streams:
            st.synchronize()
        for (h, out), want, x0 in zip(runs, wants, dX0):
            _same(out, want, x0, cfg.r)


def test_host_steps_chained_by_events():
    """Calls on two streams whose host-to-device phases are chained (call k+1 waits for call k's
    inputs_done): every call still gives the device step's results bit for bit."""
    cfg, flags = CASES["bf16_tc"]
    desc = resbm.desc_from_config(cfg, flags)
    runs = [_host_args(cfg, desc, flags, True, seed=s) for s in (3, 4)]
    wants = [_device_reference(desc, h, out) for h, out in runs]
    streams = [torch.cuda.Stream() for _ in runs]
    wss = [resbm.workspace(desc, resbm.RESBM_OP_BOUNDARY_STEP_HOST) for _ in runs]
    evs = [torch.cuda.Event() for _ in runs]
    for e, st in zip(evs, streams):
        e.record(st)          # gives each event its CUDA handle
    dX0 = [out["dX"].clone() for _, out in runs]
    prev = None
    for i in range(6):
        b = i % 2
        h, out = runs[b]
        streams[b].synchronize()   # the previous call on this stream has finished with out["dX"]
        out["dX"].copy_(dX0[b])
        resbm.resbm_boundary_step_host(desc, wss[b], stream=streams[b], wait_before_inputs=prev, inputs_done=evs[b],
                                       **h, **out)
        prev = evs[b]
    for st in streams:
        st.synchronize()
    for (h, out), want, x0 in zip(runs, wants, dX0):
        _same(out, want, x0, cfg.r)
    assert resbm.resbm_device_error() == 0


def test_host_step_empty_batch():
    """T = 0: nothing to copy in; the weight gradients come back as zeros."""
    cfg = synth.BoundaryConfig("hs_empty", T=0, d=256, r=16, m=16)
    desc = resbm.desc_from_config(cfg, 0)
    h, out = _host_args(cfg, desc, 0, True, with_dX=False)
    for k in ("dWe1", "dWe2", "dWd1", "dWd2"):
        out[k].fill_(7.0)
    ws = resbm.workspace(desc, resbm.RESBM_OP_BOUNDARY_STEP_HOST)
    resbm.resbm_boundary_step_host(desc, ws, **h, **out)
    torch.cuda.synchronize()
    for k in ("dWe1", "dWe2", "dWd1", "dWd2"):
        assert torch.count_nonzero(out[k]) == 0, k


def test_pinned_columns_move_through_the_host_mapping():
    """With page-locked host buffers the r-column copies of X and dX run as a kernel on the host
    mapping (three launches: X in, dX in, dX out); pageable buffers take strided copies. The
    results are the same either way (test_host_step_matches_device_step)."""
    cfg, flags = CASES["bf16_tc"]
    desc = resbm.desc_from_config(cfg, flags)
    ws = resbm.workspace(desc, resbm.RESBM_OP_BOUNDARY_STEP_HOST)
    launches = {}
    for pinned in (True, False):
        h, out = _host_args(cfg, desc, flags, pinned)
        torch.cuda.synchronize()
        n0 = resbm.resbm_kernel_launches()
        resbm.resbm_boundary_step_host(desc, ws, **h, **out)
        torch.cuda.synchronize()
        launches[pinned] = resbm.resbm_kernel_launches() - n0
    assert launches[True] == launches[False] + 3, launches
