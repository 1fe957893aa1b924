"""resbm_decode_bwd_noalloc, the decoder backward that takes its scratch from the library's fixed
device array instead of a caller workspace, against resbm_decode_bwd on the same inputs.

This file is named so that it is collected after the other test files: the fixed array is shared
by every call on a device, and the tests must pass both alone and after everything else ran."""
import ctypes

import pytest
import torch

from gpu_helpers import host_inputs, to_dev
from paper_2604_11947_gb300 import build, resbm, synth

CASES = {
    # tensor-core kernels: several tiles per CTA and a ragged tail
    "bf16_tc": (synth.BoundaryConfig("na_bf16", T=3001, d=1024, r=32, m=32), 0),
    # portable kernels (fp32 I/O, odd sizes)
    "f32_generic": (synth.BoundaryConfig("na_f32", T=333, d=200, r=8, m=5, dtype="f32"), 0),
    # bf16 forced onto the portable kernels
    "bf16_generic": (synth.BoundaryConfig("na_bf16_g", T=777, d=384, r=16, m=16),
                     resbm.RESBM_FLAG_GENERIC),
}


def _outputs(cfg):
    T, d, r, m = cfg.T, cfg.d, cfg.r, cfg.m
    io = torch.bfloat16 if cfg.dtype == "bf16" else torch.float32
    return (torch.empty(T, r, dtype=io, device="cuda"), torch.empty(r, m, device="cuda"),
            torch.empty(m, d, device="cuda"))


@pytest.mark.gpu
@pytest.mark.parametrize("case", CASES)
def test_noalloc_matches_decode_bwd_two_calls_in_a_row(case):
    cfg, flags = CASES[case]
    desc = resbm.desc_from_config(cfg, flags)
    assert resbm.resbm_workspace_bytes(desc, resbm.RESBM_OP_DECODE_BWD) <= resbm.RESBM_STATIC_SCRATCH_BYTES
    h = host_inputs(cfg, ("dY", "Wd1", "Wd2"))
    dev = {k: to_dev(v, cfg) for k, v in h.items()}
    dev["B"] = to_dev(synth.tensor(cfg, "dB"), cfg)      # any seeded T x r tensor serves as B
    dY2 = (dev["dY"].float() * -0.5).to(dev["dY"].dtype)  # second call: different upstream gradient
    ws = resbm.workspace(desc, resbm.RESBM_OP_DECODE_BWD)
    for dY in (dev["dY"], dY2):
        want = _outputs(cfg)
        resbm.resbm_decode_bwd(desc, dY, dev["B"], dev["Wd1"], dev["Wd2"], *want, ws)
        got = _outputs(cfg)
        resbm.resbm_decode_bwd_noalloc(desc, dY, dev["B"], dev["Wd1"], dev["Wd2"], *got)
        torch.cuda.synchronize()
        # the same kernels on the same inputs with the same launch shapes: only the scratch
        # address differs, so every output must match bit for bit
        for name, g, w in zip(("dB", "dWd1", "dWd2"), got, want):
            assert torch.equal(g, w), "%s differs from resbm_decode_bwd (max |diff| %.3e)" % (
                name, float((g.float() - w.float()).abs().max()))
    assert resbm.resbm_device_error() == 0


@pytest.mark.gpu
def test_noalloc_reserves_no_device_memory_per_call():
    cfg, flags = CASES["bf16_tc"]
    desc = resbm.desc_from_config(cfg, flags)
    h = host_inputs(cfg, ("dY", "Wd1", "Wd2"))
    dev = {k: to_dev(v, cfg) for k, v in h.items()}
    B = to_dev(synth.tensor(cfg, "dB"), cfg)
    out = _outputs(cfg)
    resbm.resbm_decode_bwd_noalloc(desc, dev["dY"], B, dev["Wd1"], dev["Wd2"], *out)
    torch.cuda.synchronize()
    # torch's caching allocator sees no request (the library never calls into torch), and the
    # device's free memory does not move (the library calls no cudaMalloc either)
    alloc0, reserved0 = torch.cuda.memory_allocated(), torch.cuda.memory_reserved()
    free0, _ = torch.cuda.mem_get_info()
    for _ in range(3):
        resbm.resbm_decode_bwd_noalloc(desc, dev["dY"], B, dev["Wd1"], dev["Wd2"], *out)
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert torch.cuda.memory_allocated() == alloc0
    assert torch.cuda.memory_reserved() == reserved0
    assert free1 == free0


def test_noalloc_rejects_scratch_beyond_the_fixed_size():
    """A shape whose scratch exceeds the fixed array is refused before anything touches the
    device (fake, aligned, non-overlapping pointers)."""
    build.build()
    lib = resbm.load()
    d = resbm.make_desc(65536, 4096, 32, 32, dtype="bf16")
    assert resbm.resbm_workspace_bytes(d, resbm.RESBM_OP_DECODE_BWD) > resbm.RESBM_STATIC_SCRATCH_BYTES
    big, A = 1 << 32, 1 << 40
    st = lib.resbm_decode_bwd_noalloc(ctypes.byref(d), *[A + i * big for i in range(7)], None)
    assert st == resbm.RESBM_ERR_WORKSPACE
    # argument errors still come first
    st = lib.resbm_decode_bwd_noalloc(ctypes.byref(d), None, *[A + i * big for i in range(6)], None)
    assert st == resbm.RESBM_ERR_INVALID_ARG
