"""The CUDA path (through the C ABI) against the fp64 oracle on the same seeded inputs."""
import numpy as np
import pytest
import torch

from gpu_helpers import (INPUTS, assert_step_is_its_stages, check_output, gpu_stages, gpu_step,
                         host_inputs, oracle_step, to_dev, to_host)
from metrics import TOL, check
from paper_2604_11947_gb300 import resbm, synth

import oracle

pytestmark = pytest.mark.gpu

# default: the fused tensor-core kernels where they take the shape, else the tensor-core GEMM
# chain, else the portable kernels; gemm: the GEMM chain wherever it takes the shape (bf16, d, r, m
# multiples of 8); generic: the portable CUDA-core kernels
PATHS = {"default": 0, "gemm": resbm.RESBM_FLAG_GEMM, "generic": resbm.RESBM_FLAG_GENERIC}
OUTS = ("B", "Y", "dB", "dF", "dX", "dWe1", "dWe2", "dWd1", "dWd2")

SMALL = {
    # name: config (ragged token counts, several 128-token tiles, r and m around the tiles)
    "tiny_f32": synth.CONFIGS["tiny_f32"],
    "ragged_bf16_r32": synth.BoundaryConfig("ragged_bf16_r32", T=1000, d=512, r=32, m=32),
    "ragged_bf16_r16": synth.BoundaryConfig("ragged_bf16_r16", T=777, d=384, r=16, m=16),
    "bf16_r64": synth.BoundaryConfig("bf16_r64", T=300, d=256, r=64, m=64),
    "bf16_m_ne_r": synth.BoundaryConfig("bf16_m_ne_r", T=515, d=320, r=16, m=48),
    "bf16_r128": synth.BoundaryConfig("bf16_r128", T=260, d=512, r=128, m=128),
    "f32_ragged": synth.BoundaryConfig("f32_ragged", T=333, d=200, r=8, m=5, dtype="f32"),
    "bf16_odd_d": synth.BoundaryConfig("bf16_odd_d", T=129, d=100, r=3, m=7),
    "bf16_no_compression": synth.BoundaryConfig("bf16_no_compression", T=200, d=64, r=64, m=16),
    "bf16_r1": synth.BoundaryConfig("bf16_r1", T=64, d=128, r=1, m=1),
    # ~1000 tokens per CTA: several groups of tiles per CTA in the backward kernels (whose
    # grids on a 152-SM GB300 are 144 CTAs in clusters of 4; the decoder backward's balanced grid
    # keeps the most tiles per CTA on fewer clusters: 132 CTAs here)
    "bf16_multi_group": synth.BoundaryConfig("bf16_multi_group", T=150001, d=128, r=32, m=32),
    # 618 (585) tiles on 144 backward CTAs: 4 or 5 tiles per CTA, cut into 2 + 2 or 3 + 2, so
    # the CTAs of a cluster have different group sizes but the same number of groups
    "bf16_uneven_groups": synth.BoundaryConfig("bf16_uneven_groups", T=79031, d=256, r=32, m=32),
    "bf16_uneven_groups_144": synth.BoundaryConfig("bf16_uneven_groups_144", T=74871, d=256, r=32, m=32),
    # one partial tile: a single CTA (pairs of the encoder forward: the forced-cluster cases)
    "bf16_single_ctas": synth.BoundaryConfig("bf16_single_ctas", T=40, d=256, r=32, m=32),
    # one 64-column chunk per tile and three; the other stages run on the portable kernels at
    # these widths
    "bf16_d64": synth.BoundaryConfig("bf16_d64", T=1000, d=64, r=32, m=32),
    "bf16_d192": synth.BoundaryConfig("bf16_d192", T=300, d=192, r=32, m=32),
    # widths the fused kernels do not take run as the tensor-core GEMM chain by default: m = r =
    # 512 (two 256-column output blocks, split-K weight gradients at this T), and odd multiples
    # of 8 (d = 776 = 3 x 256 + 8 leaves an 8-column output block and a 8-deep K tail; r = 24 and
    # m = 40 a partial 32-column epilogue chunk)
    "bf16_r512": synth.BoundaryConfig("bf16_r512", T=700, d=1024, r=512, m=512),
    # nine 128-row blocks: the GEMM's CTA pairs (B shared by multicast) end with a partner whose
    # row block lies past T (it loads zeros and stores nothing)
    "bf16_r512_odd_blocks": synth.BoundaryConfig("bf16_r512_odd_blocks", T=1100, d=1024, r=512, m=512),
    "bf16_r24_m40": synth.BoundaryConfig("bf16_r24_m40", T=999, d=776, r=24, m=40),
    # K = d = 2304 and K = T = 2300: the long-K products (P = F . We1, dQ = dY . Wd2^T and the
    # weight gradients) where the GEMM may take 256-row units; m = 384 leaves a 128-column output
    # block, T a 252-row last unit (its second half partly past T)
    "bf16_r384_long_k": synth.BoundaryConfig("bf16_r384_long_k", T=2300, d=2304, r=384, m=384),
}

# Backward grids under each forced cluster size (RESBM_CLUSTER), one CTA per 128-token
# tile at most: 8 tiles -> 8 CTAs in pairs or fours; 16 -> 16; 17 -> 16 in pairs or fours (one
# idle SM); 18 -> 18 in pairs, no fours (16 < 15/16 x 18); 3 -> single CTAs (fours do not fit,
# pairs leave too many idle); uneven tile groups inside clusters. The decoder backward then
# shrinks that grid to the fewest clusters that keep its most tiles per CTA (17 tiles: 12 CTAs in
# fours, two tiles each but one; test_decoder_backward_grid_rules_match_oracle runs both rules).
CLUSTER_CASES = {
    "t8_r32": synth.BoundaryConfig("cl_t8_r32", T=1000, d=512, r=32, m=32),
    "t16_r32": synth.BoundaryConfig("cl_t16_r32", T=2000, d=384, r=32, m=32),
    "t16_r16": synth.BoundaryConfig("cl_t16_r16", T=1990, d=256, r=16, m=16),
    "t17_r32": synth.BoundaryConfig("cl_t17_r32", T=2100, d=256, r=32, m=32),
    "t18_r32": synth.BoundaryConfig("cl_t18_r32", T=2260, d=256, r=32, m=32),
    "t3_r32": synth.BoundaryConfig("cl_t3_r32", T=280, d=256, r=32, m=32),
    "uneven_r32": synth.BoundaryConfig("cl_uneven_r32", T=79031, d=256, r=32, m=32),
    # 321 tiles on 152 CTAs (144 in fours): two or three tiles per CTA, the last one partial
    # (77 tokens)
    "t321_r32": synth.BoundaryConfig("cl_t321_r32", T=41037, d=256, r=32, m=32),
    # 235 tiles: one or two per CTA, the last partial (48 tokens); three d chunks
    "t235_d384_r16": synth.BoundaryConfig("cl_t235_d384_r16", T=30000, d=384, r=16, m=16),
    # the encoder forward's pairs where it has no more tiles than SMs (single CTAs by default):
    # one partial tile split by a pair; one 64-column chunk per tile (the split always falls on a
    # tile boundary) and three (a pair's single tile split 1 + 2)
    "t1_partial": synth.BoundaryConfig("cl_t1_partial", T=40, d=256, r=32, m=32),
    "d64": synth.BoundaryConfig("cl_d64", T=1000, d=64, r=32, m=32),
    "d192": synth.BoundaryConfig("cl_d192", T=300, d=192, r=32, m=32),
}
_ORACLE_CACHE = {}


@pytest.mark.parametrize("cluster", ["1", "2", "4"])
@pytest.mark.parametrize("name", CLUSTER_CASES)
def test_forced_cluster_sizes_match_oracle(name, cluster, monkeypatch):
    """The backward kernels with every cluster size forced (1, 2, 4 CTAs), where it fits."""
    monkeypatch.setenv("RESBM_CLUSTER", cluster)
    cfg = CLUSTER_CASES[name]
    h = host_inputs(cfg)
    dev = {k: to_dev(v, cfg) for k, v in h.items()}
    got = gpu_step(cfg, dev)
    if name not in _ORACLE_CACHE:
        _ORACLE_CACHE[name] = oracle_step(cfg, h)
    _compare_all(cfg, got, _ORACLE_CACHE[name], dev)
    assert resbm.resbm_device_error() == 0


@pytest.mark.parametrize("balance", ["0", "1"])
@pytest.mark.parametrize("name", ["t321_r32", "uneven_r32"])
def test_decoder_backward_grid_rules_match_oracle(name, balance, monkeypatch):
    """The decoder backward on its balanced grid (the fewest clusters that keep the most tiles a
    CTA gets: 321 tiles on 108 CTAs instead of 144, 618 on 124) and on the cluster rule's full
    grid (RESBM_BWD_BALANCE=0): both against the oracle."""
    monkeypatch.setenv("RESBM_BWD_BALANCE", balance)
    cfg = CLUSTER_CASES[name]
    h = host_inputs(cfg)
    dev = {k: to_dev(v, cfg) for k, v in h.items()}
    got = gpu_step(cfg, dev)
    if name not in _ORACLE_CACHE:
        _ORACLE_CACHE[name] = oracle_step(cfg, h)
    _compare_all(cfg, got, _ORACLE_CACHE[name], dev)
    assert resbm.resbm_device_error() == 0


def _compare_all(cfg, got, want, dev, flags=0):
    """The step's boundary tensors (B and dB, after the transfer rounding) against the oracle's;
    every later output against the oracle with the stage that produces it run on the oracle's
    transferred tensor (gpu_stages); and the step against its own stages, bit for bit."""
    errs = {k: check_output(k, got[k], want[k], cfg) for k in ("B", "dB")}
    stages = gpu_stages(cfg, dev, want, flags)
    for k in OUTS:
        if k not in ("B",):
            errs["stage_" + k] = check_output(k, stages[k], want[k], cfg)
    assert_step_is_its_stages(cfg, dev, got, flags)
    return errs


@pytest.mark.parametrize("path", PATHS)
@pytest.mark.parametrize("name", SMALL)
def test_small_configs_match_oracle(name, path):
    cfg = SMALL[name]
    h = host_inputs(cfg)
    dev = {k: to_dev(v, cfg) for k, v in h.items()}
    got = gpu_step(cfg, dev, flags=PATHS[path])
    want = oracle_step(cfg, h)
    _compare_all(cfg, got, want, dev, PATHS[path])
    # the saved pre-activation P = F . We1 is an fp32 output: fp32 accumulation error only
    check("P", to_host(got["P"]), want["P"], "f32", tol=1e-4)


@pytest.mark.parametrize("bm2", ["0", "1"])
@pytest.mark.parametrize("name", ["bf16_r384_long_k", "bf16_r512_odd_blocks", "bf16_r24_m40"])
def test_gemm_row_units_match_oracle(name, bm2, monkeypatch):
    """The GEMM chain with 256-row units forced wherever the shape allows them (RESBM_GEMM_BM2=1)
    and with 128-row units only (=0): both against the oracle, and the forward outputs (single
    products, no split over K) the same bits either way."""
    cfg = SMALL[name]
    h = host_inputs(cfg)
    dev = {k: to_dev(v, cfg) for k, v in h.items()}
    monkeypatch.setenv("RESBM_GEMM_BM2", bm2)
    got = gpu_step(cfg, dev)
    if name not in _ORACLE_CACHE:
        _ORACLE_CACHE[name] = oracle_step(cfg, h)
    _compare_all(cfg, got, _ORACLE_CACHE[name], dev)
    check("P", to_host(got["P"]), _ORACLE_CACHE[name]["P"], "f32", tol=1e-4)
    monkeypatch.setenv("RESBM_GEMM_BM2", "1" if bm2 == "0" else "0")
    other = gpu_step(cfg, dev)
    for k in ("B", "Y", "P"):
        assert torch.equal(got[k], other[k]), k
    assert resbm.resbm_device_error() == 0


@pytest.mark.parametrize("name", ["bf16_r512_odd_blocks", "bf16_r24_m40", "bf16_r384_long_k"])
def test_gemm_tma_store_epilogue_same_bits(name, monkeypatch):
    """The GEMM chain's TMA-store epilogue for Y and dF (on by default) against per-thread stores
    (RESBM_GEMM_TS=0): every output of the step the same bits (d = 776 leaves an 8-column last
    box, T = 999 and 1100 partial row blocks and a pair partner past T; m = 40 takes dF from a
    hi + lo dP)."""
    cfg = SMALL[name]
    h = host_inputs(cfg)
    dev = {k: to_dev(v, cfg) for k, v in h.items()}
    got = gpu_step(cfg, dev, flags=resbm.RESBM_FLAG_GEMM)
    monkeypatch.setenv("RESBM_GEMM_TS", "0")
    ref = gpu_step(cfg, dev, flags=resbm.RESBM_FLAG_GEMM)
    for k in OUTS:
        assert torch.equal(got[k], ref[k]), k
    assert resbm.resbm_device_error() == 0


@pytest.mark.parametrize("act", ["gelu_tanh", "identity"])
@pytest.mark.parametrize("merge", [0, 1])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_activation_and_merge_variants(act, merge, dtype):
    cfg = synth.BoundaryConfig("v", T=400, d=256, r=16, m=24, dtype=dtype, act=act, merge=merge)
    h = host_inputs(cfg)
    dev = {k: to_dev(v, cfg) for k, v in h.items()}
    want = oracle_step(cfg, h)
    for flags in PATHS.values():
        _compare_all(cfg, gpu_step(cfg, dev, flags=flags), want, dev, flags)


def test_single_bf16_config_full():
    """T = 16384, d = 2048, r = 16 (batch 8 x seq 2048, 128x): every element of every output."""
    cfg = synth.CONFIGS["single_bf16"]
    h = host_inputs(cfg)
    dev = {k: to_dev(v, cfg) for k, v in h.items()}
    got = gpu_step(cfg, dev)
    want = oracle_step(cfg, h)
    _compare_all(cfg, got, want, dev)


def _full_size_every_element(cfg):
    """Full-size launch (the benchmarked shapes, the grids and cluster sizes the bench runs)
    against one oracle step over all T tokens: every element of B, Y, dB, dF, dX[:, :r] and of
    the four weight gradients, each compared with the stage run on the oracle's transferred
    tensor as in the small cases, and the step against its own stages bit for bit."""
    h = host_inputs(cfg)
    dev = {k: to_dev(v, cfg) for k, v in h.items()}
    got = gpu_step(cfg, dev)
    want = oracle_step(cfg, h)
    del h
    errs = _compare_all(cfg, got, want, dev)
    assert resbm.resbm_device_error() == 0
    return errs


@pytest.mark.slow
def test_large_bf16_full_size():
    """T = 65536, d = 4096, r = 32 (batch 32 x seq 2048, 128x): the headline workload."""
    _full_size_every_element(synth.CONFIGS["large_bf16"])


@pytest.mark.slow
@pytest.mark.parametrize("name", ["sweep_r512", "sweep_r128", "sweep_r64", "sweep_r32"])
def test_sweep_full_size(name):
    """d = 8192, T = 32768, r in {512, 128, 64, 32} (16x .. 256x compression)."""
    _full_size_every_element(synth.CONFIGS[name])


# ---------------------------------------------------------------------------------------------
# The single ops, their optional arguments, and edge cases.
# ---------------------------------------------------------------------------------------------

def _ws(desc, op):
    return resbm.workspace(desc, op)


@pytest.mark.parametrize("path", PATHS)
def test_single_ops_and_optional_arguments(path):
    cfg = synth.BoundaryConfig("ops", T=700, d=384, r=32, m=32)
    flags = PATHS[path]
    h = host_inputs(cfg, INPUTS + ("dB", "dX0"))
    dev = {k: to_dev(v, cfg) for k, v in h.items()}
    desc = resbm.desc_from_config(cfg, flags)
    T, d, r, m = cfg.T, cfg.d, cfg.r, cfg.m
    bf = torch.bfloat16
    B = torch.empty(T, r, dtype=bf, device="cuda")
    P = torch.empty(T, m, dtype=torch.float32, device="cuda")
    resbm.resbm_encode_fwd(desc, dev["X"], dev["F"], dev["We1"], dev["We2"], B, None,
                           _ws(desc, resbm.RESBM_OP_ENCODE_FWD))
    wantB, wantP = oracle.encode_fwd(h["X"], h["F"], h["We1"], h["We2"], cfg.act)
    check("B", to_host(B), wantB, "bf16")
    B2 = torch.empty_like(B)
    resbm.resbm_encode_fwd(desc, dev["X"], dev["F"], dev["We1"], dev["We2"], B2, P,
                           _ws(desc, resbm.RESBM_OP_ENCODE_FWD))
    torch.cuda.synchronize()
    assert torch.equal(B, B2)
    check("P", to_host(P), wantP, "f32", tol=1e-4)
    # X aliasing F (single-input variant)
    resbm.resbm_encode_fwd(desc, dev["F"], dev["F"], dev["We1"], dev["We2"], B2, None,
                           _ws(desc, resbm.RESBM_OP_ENCODE_FWD))
    check("B", to_host(B2), oracle.encode_fwd(h["F"], h["F"], h["We1"], h["We2"], cfg.act)[0], "bf16")
    # encode bwd with a given dB, with and without P_save, with and without dX
    dF = torch.empty(T, d, dtype=bf, device="cuda")
    dX = dev["dX0"].clone()
    dWe1 = torch.empty(d, m, device="cuda")
    dWe2 = torch.empty(m, r, device="cuda")
    wdF, wdX, wdWe1, wdWe2 = oracle.encode_bwd(h["dB"], h["F"], h["We1"], h["We2"], cfg.act)
    dF_with_P = None
    for Psave in (P, None):
        dX.copy_(dev["dX0"])
        resbm.resbm_encode_bwd(desc, dev["dB"], dev["F"], Psave, dev["We1"], dev["We2"], dF, dX,
                               dWe1, dWe2, _ws(desc, resbm.RESBM_OP_ENCODE_BWD))
        check("dF", to_host(dF), wdF, "bf16")
        check("dWe1", to_host(dWe1), wdWe1, "bf16")
        check("dWe2", to_host(dWe2), wdWe2, "bf16")
        # dX[:, :r] += dB in bf16, other columns untouched
        expect = h["dX0"].astype(np.float64) + wdX
        check("dX", to_host(dX), expect, "bf16")
        assert torch.equal(dX[:, r:], dev["dX0"][:, r:])
        if Psave is not None:
            dF_with_P = dF.clone()
    # leaving out dX changes nothing else
    dF2 = torch.empty_like(dF)
    resbm.resbm_encode_bwd(desc, dev["dB"], dev["F"], P, dev["We1"], dev["We2"], dF2, None,
                           dWe1, dWe2, _ws(desc, resbm.RESBM_OP_ENCODE_BWD))
    torch.cuda.synchronize()
    assert torch.equal(dF_with_P, dF2)
    # decode fwd / bwd alone
    Y = torch.empty(T, d, dtype=bf, device="cuda")
    resbm.resbm_decode_fwd(desc, dev["dB"], dev["Wd1"], dev["Wd2"], Y, _ws(desc, resbm.RESBM_OP_DECODE_FWD))
    check("Y", to_host(Y), oracle.decode_fwd(h["dB"], h["Wd1"], h["Wd2"], cfg.act, cfg.merge), "bf16")
    dB = torch.empty(T, r, dtype=bf, device="cuda")
    dWd1 = torch.empty(r, m, device="cuda")
    dWd2 = torch.empty(m, d, device="cuda")
    resbm.resbm_decode_bwd(desc, dev["dY"], dev["dB"], dev["Wd1"], dev["Wd2"], dB, dWd1, dWd2,
                           _ws(desc, resbm.RESBM_OP_DECODE_BWD))
    wdB, wdWd1, wdWd2 = oracle.decode_bwd(h["dY"], h["dB"], h["Wd1"], h["Wd2"], cfg.act, cfg.merge)
    check("dB", to_host(dB), wdB, "bf16")
    check("dWd1", to_host(dWd1), wdWd1, "bf16")
    check("dWd2", to_host(dWd2), wdWd2, "bf16")


@pytest.mark.parametrize("path", PATHS)
def test_zero_learned_weights_give_identity_path_bitwise(path):
    """The identity path alone (Sec. 3.3): with zero second-layer weights B = X[:, :r] and
    Y = pad(B) exactly; backward gives dB = dY[:, :r], dF = 0 exactly."""
    cfg = synth.BoundaryConfig("zero", T=300, d=256, r=16, m=16)
    h = host_inputs(cfg)
    h["We2"] = np.zeros_like(h["We2"])
    h["Wd2"] = np.zeros_like(h["Wd2"])
    dev = {k: to_dev(v, cfg) for k, v in h.items()}
    got = gpu_step(cfg, dev, flags=PATHS[path])
    r = cfg.r
    assert torch.equal(got["B"], dev["X"][:, :r])
    assert torch.equal(got["Y"][:, :r], got["B"]) and not torch.any(got["Y"][:, r:])
    assert torch.equal(got["dB"], dev["dY"][:, :r])
    assert not torch.any(got["dF"])
    assert torch.equal(got["dX"][:, :r], dev["dY"][:, :r]) and not torch.any(got["dX"][:, r:])


def test_no_compression_zero_weights_is_vanilla_residual():
    """r = d (c = C, Sec. 3.3) with zero learned weights: Y == X bit for bit."""
    cfg = synth.BoundaryConfig("vanilla", T=256, d=64, r=64, m=16)
    h = host_inputs(cfg)
    h["We2"] = np.zeros_like(h["We2"])
    h["Wd2"] = np.zeros_like(h["Wd2"])
    dev = {k: to_dev(v, cfg) for k, v in h.items()}
    for flags in PATHS.values():
        got = gpu_step(cfg, dev, flags=flags)
        assert torch.equal(got["Y"], dev["X"])


@pytest.mark.parametrize("path", PATHS)
def test_empty_batch_zeroes_weight_grads(path):
    cfg = synth.BoundaryConfig("empty", T=0, d=128, r=8, m=8)
    desc = resbm.desc_from_config(cfg, PATHS[path])
    w = {k: to_dev(synth.tensor(cfg, k), cfg) for k in ("We1", "We2", "Wd1", "Wd2")}
    empty = torch.empty(0, cfg.d, dtype=torch.bfloat16, device="cuda")
    out = resbm.step_outputs(desc)
    for k in ("dWe1", "dWe2", "dWd1", "dWd2"):
        out[k].fill_(7.0)
    ws = resbm.workspace(desc, resbm.RESBM_OP_BOUNDARY_STEP)
    resbm.resbm_boundary_step(desc, ws, X=empty, F=empty, dY=empty, **w, **out)
    torch.cuda.synchronize()
    for k in ("dWe1", "dWe2", "dWd1", "dWd2"):
        assert not torch.any(out[k]), k


@pytest.mark.parametrize("path", PATHS)
def test_deterministic(path):
    cfg = synth.BoundaryConfig("det", T=2048, d=512, r=32, m=32)
    h = host_inputs(cfg)
    dev = {k: to_dev(v, cfg) for k, v in h.items()}
    a = gpu_step(cfg, dev, flags=PATHS[path])
    b = gpu_step(cfg, dev, flags=PATHS[path])
    for k in OUTS + ("P",):
        assert torch.equal(a[k], b[k]), k


def test_workspace_too_small_is_reported_on_device():
    cfg = synth.BoundaryConfig("ws", T=256, d=256, r=16, m=16)
    desc = resbm.desc_from_config(cfg)
    h = host_inputs(cfg)
    dev = {k: to_dev(v, cfg) for k, v in h.items()}
    out = resbm.step_outputs(desc)
    need = resbm.resbm_workspace_bytes(desc, resbm.RESBM_OP_BOUNDARY_STEP)
    ws = torch.empty(max(need - 256, 1), dtype=torch.uint8, device="cuda")
    with pytest.raises(resbm.ResbmError) as e:
        resbm.resbm_boundary_step(desc, ws, **dev, **out)
    assert e.value.status == resbm.RESBM_ERR_WORKSPACE


def test_runs_on_a_side_stream():
    cfg = synth.BoundaryConfig("stream", T=512, d=256, r=16, m=16)
    h = host_inputs(cfg)
    dev = {k: to_dev(v, cfg) for k, v in h.items()}
    ref = gpu_step(cfg, dev)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        got = gpu_step(cfg, dev)
    torch.cuda.synchronize()
    for k in OUTS:
        assert torch.equal(ref[k], got[k]), k


def test_no_kernel_reported_a_timeout():
    """The tensor-core kernels' bounded waits never gave up during this test session."""
    assert resbm.resbm_device_error() == 0


# ---------------------------------------------------------------------------------------------
# One linear layer per side (RESBM_FLAG_LINEAR): We1 is d x r, Wd2 is r x d, no We2 / Wd1.
# ---------------------------------------------------------------------------------------------

LINEAR = {
    "bf16_r32": synth.BoundaryConfig("lin_bf16", T=1000, d=512, r=32, m=32),
    "bf16_r16_merge0": synth.BoundaryConfig("lin_bf16_m0", T=777, d=384, r=16, m=16, merge=0),
    "f32_r8": synth.BoundaryConfig("lin_f32", T=333, d=200, r=8, m=8, dtype="f32"),
}


@pytest.mark.parametrize("path", PATHS)
@pytest.mark.parametrize("name", LINEAR)
def test_linear_mode_matches_oracle(name, path):
    cfg = LINEAR[name]
    flags = PATHS[path] | resbm.RESBM_FLAG_LINEAR
    desc = resbm.desc_from_config(cfg, flags)
    T, d, r = cfg.T, cfg.d, cfg.r
    h = host_inputs(cfg, ("X", "F", "dY", "We1", "Wd2"))
    dev = {k: to_dev(v, cfg) for k, v in h.items()}
    io = torch.bfloat16 if cfg.dtype == "bf16" else torch.float32
    want = oracle.linear_boundary_step(h["X"], h["F"], h["dY"], h["We1"], h["Wd2"], cfg.merge,
                                       transfer=cfg.dtype)
    # the whole step through the C ABI (second-layer tensors absent)
    out = dict(B=torch.empty(T, r, dtype=io, device="cuda"), Y=torch.empty(T, d, dtype=io, device="cuda"),
               dB=torch.empty(T, r, dtype=io, device="cuda"), dF=torch.empty(T, d, dtype=io, device="cuda"),
               dX=torch.zeros(T, d, dtype=io, device="cuda"), dWe1=torch.empty(d, r, device="cuda"),
               dWd2=torch.empty(r, d, device="cuda"))
    ws = resbm.workspace(desc, resbm.RESBM_OP_BOUNDARY_STEP)
    resbm.resbm_boundary_step(desc, ws, X=dev["X"], F=dev["F"], dY=dev["dY"], We1=dev["We1"],
                              Wd2=dev["Wd2"], **out)
    torch.cuda.synchronize()
    for k in ("B", "dB"):
        check_output(k, out[k], want[k], cfg)
    # each later stage on the oracle's transferred tensor, against the oracle
    B = to_dev(want["B"], cfg)
    Y = torch.empty_like(out["Y"])
    resbm.resbm_decode_fwd(desc, B, None, dev["Wd2"], Y, resbm.workspace(desc, resbm.RESBM_OP_DECODE_FWD))
    dB = torch.empty_like(out["dB"])
    dWd2 = torch.empty_like(out["dWd2"])
    resbm.resbm_decode_bwd(desc, dev["dY"], B, None, dev["Wd2"], dB, None, dWd2,
                           resbm.workspace(desc, resbm.RESBM_OP_DECODE_BWD))
    dF = torch.empty_like(out["dF"])
    dX = torch.zeros_like(out["dX"])
    dWe1 = torch.empty_like(out["dWe1"])
    resbm.resbm_encode_bwd(desc, to_dev(want["dB"], cfg), dev["F"], None, dev["We1"], None, dF, dX,
                           dWe1, None, resbm.workspace(desc, resbm.RESBM_OP_ENCODE_BWD))
    torch.cuda.synchronize()
    for k, v in dict(Y=Y, dB=dB, dWd2=dWd2, dF=dF, dX=dX, dWe1=dWe1).items():
        check_output(k, v, want[k], cfg)
    # the step is its own stages, bit for bit
    resbm.resbm_decode_fwd(desc, out["B"], None, dev["Wd2"], Y, resbm.workspace(desc, resbm.RESBM_OP_DECODE_FWD))
    resbm.resbm_decode_bwd(desc, dev["dY"], out["B"], None, dev["Wd2"], dB, None, dWd2,
                           resbm.workspace(desc, resbm.RESBM_OP_DECODE_BWD))
    dX.zero_()
    resbm.resbm_encode_bwd(desc, out["dB"], dev["F"], None, dev["We1"], None, dF, dX, dWe1, None,
                           resbm.workspace(desc, resbm.RESBM_OP_ENCODE_BWD))
    torch.cuda.synchronize()
    for k, v in dict(Y=Y, dB=dB, dWd2=dWd2, dF=dF, dX=dX, dWe1=dWe1).items():
        assert torch.equal(v, out[k]), k


def test_linear_zero_weights_give_identity_path_bitwise():
    cfg = synth.BoundaryConfig("lin_zero", T=300, d=256, r=16, m=16)
    desc = resbm.desc_from_config(cfg, resbm.RESBM_FLAG_LINEAR)
    h = host_inputs(cfg, ("X", "F", "dY"))
    dev = {k: to_dev(v, cfg) for k, v in h.items()}
    T, d, r = cfg.T, cfg.d, cfg.r
    bf = torch.bfloat16
    zero_e, zero_d = torch.zeros(d, r, dtype=bf, device="cuda"), torch.zeros(r, d, dtype=bf, device="cuda")
    out = dict(B=torch.empty(T, r, dtype=bf, device="cuda"), Y=torch.empty(T, d, dtype=bf, device="cuda"),
               dB=torch.empty(T, r, dtype=bf, device="cuda"), dF=torch.empty(T, d, dtype=bf, device="cuda"),
               dWe1=torch.empty(d, r, device="cuda"), dWd2=torch.empty(r, d, device="cuda"))
    resbm.resbm_boundary_step(desc, resbm.workspace(desc, resbm.RESBM_OP_BOUNDARY_STEP), X=dev["X"],
                              F=dev["F"], dY=dev["dY"], We1=zero_e, Wd2=zero_d, **out)
    torch.cuda.synchronize()
    assert torch.equal(out["B"], dev["X"][:, :r])
    assert torch.equal(out["Y"][:, :r], out["B"]) and not torch.any(out["Y"][:, r:])
    assert torch.equal(out["dB"], dev["dY"][:, :r])
    assert not torch.any(out["dF"])
