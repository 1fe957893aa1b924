"""The simulated pipeline (a decoder-only transformer in stages with ResBM boundaries, Sec. 3.2
placement): one training step through the C ABI, and every boundary's tensors of that step
against the fp64 oracle run on the same inputs."""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import to_host
from metrics import bf16_half_spacing, check
from paper_2604_11947_gb300 import pipeline, resbm

pytestmark = pytest.mark.gpu


def _check_boundary(cap, bnd, cfg, merge):
    """Each op of one boundary against the oracle on the inputs the step gave it."""
    X, F, dY = to_host(cap["X"]), to_host(cap["F"]), to_host(cap["dY"])
    w = {k: to_host(getattr(bnd, k)) for k in ("We1", "We2", "Wd1", "Wd2")}
    B, dB = to_host(cap["B"]), to_host(cap["dB"])
    assert torch.equal(cap["B"], cap["B_dec"])          # the handoff is the tensor itself
    if merge:
        # reading A: b has one consumer, so the encoder receives the decoder's dB itself (its
        # identity-path term included); reading B adds the pad skip's gradient to it
        assert torch.equal(cap["dB"], cap["dB_in"])
    dB_in = to_host(cap["dB_in"])
    wantB, _ = oracle.encode_fwd(X, F, w["We1"], w["We2"], cfg.act)
    check("B", B, wantB, "bf16")
    check("Y", to_host(cap["Y"]), oracle.decode_fwd(B, w["Wd1"], w["Wd2"], cfg.act, merge), "bf16")
    wdB, wdWd1, wdWd2 = oracle.decode_bwd(dY, B, w["Wd1"], w["Wd2"], cfg.act, merge)
    check("dB", dB, wdB, "bf16")
    if "N" in cap:   # the receiving block's attention input, from the fused decoder + RMSNorm
        gamma = to_host(cap["gamma"])
        wY2, wN = oracle.decode_fwd_rmsnorm(B, w["Wd1"], w["Wd2"], gamma, pipeline.NORM_EPS, cfg.act, merge)
        rstd = 1.0 / np.sqrt(np.mean(wY2 * wY2, axis=1, keepdims=True) + pipeline.NORM_EPS)
        check("N", to_host(cap["N"]), wN, "bf16", allow=bf16_half_spacing(wY2) * np.abs(rstd * gamma[None, :]))
    check("dWd1", to_host(cap["dWd1"]), wdWd1, "bf16")
    check("dWd2", to_host(cap["dWd2"]), wdWd2, "bf16")
    wdF, wdX, wdWe1, wdWe2 = oracle.encode_bwd(dB_in, F, w["We1"], w["We2"], cfg.act)
    check("dF", to_host(cap["dF"]), wdF, "bf16")
    dX = to_host(cap["dX"])
    r = bnd.r
    assert not np.any(dX[:, r:]), "the identity path's gradient reaches only the first r columns"
    check("dX", dX[:, :r], wdX[:, :r], "bf16")
    check("dWe1", to_host(cap["dWe1"]), wdWe1, "bf16")
    check("dWe2", to_host(cap["dWe2"]), wdWe2, "bf16")


def _run(cfg):
    model = pipeline.PipelineModel(cfg)
    caps = []
    for bnd in model.bounds:
        bnd.capture = {}
        caps.append(bnd.capture)
    tokens = pipeline.synthetic_tokens(cfg)
    loss = pipeline.train_step(model, tokens)
    torch.cuda.synchronize()
    assert torch.isfinite(loss)
    for p in model.parameters():
        assert p.grad is not None and torch.isfinite(p.grad.float()).all()
    return model, caps


def test_four_stage_pipeline_boundaries_match_oracle():
    """24 layers, d = 2048, 16 heads, SwiGLU 5632, vocabulary 32000, 4 stages, r = 16, batch 8 x
    seq 2048: every one of the three boundaries, forward and backward, against the oracle."""
    cfg = pipeline.PIPELINE
    model, caps = _run(cfg)
    assert len(caps) == 3
    for cap, bnd in zip(caps, model.bounds):
        assert cap["X"].shape == (cfg.tokens, cfg.d) and cap["B"].shape == (cfg.tokens, bnd.r)
        _check_boundary(cap, bnd, cfg, merge=1)
    assert resbm.resbm_device_error() == 0


def test_reading_b_wiring_boundaries_match_oracle():
    """The decoder inside the attention branch (merge_identity = 0; pad(b) is the attention's
    skip), on a small model."""
    cfg = pipeline.PipelineConfig(layers=4, d=512, heads=4, ffn=1024, vocab=1000, stages=2, r=16, m=16,
                                  batch=2, seq=256, wiring="B")
    model, caps = _run(cfg)
    _check_boundary(caps[0], model.bounds[0], cfg, merge=0)


def test_non_uniform_bottleneck_widths():
    """A different r (and m) at each boundary (the paper allows the compression to vary per
    boundary): r = 16, 32, 64 over three boundaries, every boundary against the oracle."""
    cfg = pipeline.PipelineConfig(layers=4, d=512, heads=4, ffn=1024, vocab=1000, stages=4, r=(16, 32, 64),
                                  m=(16, 32, 64), batch=2, seq=256)
    model, caps = _run(cfg)
    assert [b.r for b in model.bounds] == [16, 32, 64]
    for cap, bnd in zip(caps, model.bounds):
        assert cap["B"].shape == (cfg.tokens, bnd.r)
        _check_boundary(cap, bnd, cfg, merge=1)
    assert resbm.resbm_device_error() == 0


def test_boundary_share_is_measured():
    cfg = pipeline.PipelineConfig(layers=4, d=512, heads=4, ffn=1024, vocab=1000, stages=4, r=16, m=16,
                                  batch=2, seq=256)
    model = pipeline.PipelineModel(cfg)
    step_ms, bnd_ms, loss = pipeline.time_steps(model, pipeline.synthetic_tokens(cfg), steps=2, warmup=1)
    assert 0 < bnd_ms < step_ms and np.isfinite(loss)


def test_both_wirings_learn_the_markov_stream():
    """Reading A and reading B of the receive side, and the uncompressed model, trained with AdamW
    on a learnable stream: every loss curve falls well below its start (ln 256 = 5.5) toward the
    stream's entropy rate."""
    res = pipeline.convergence(steps=150)
    for name in ("A", "B", "uncompressed"):
        curve = res[name]
        first, last = curve[0][1], curve[-1][1]
        assert np.isfinite(last) and last < 0.6 * first, (name, curve)
    assert resbm.resbm_device_error() == 0


@pytest.mark.parametrize("wiring", ["A", "B"])
def test_fused_norm_matches_the_unfused_model(wiring):
    """The same model with the receiving block's RMSNorm fused into the decoder and without: the
    loss and every gradient agree to bf16 noise (the fused N skips one rounding of y)."""
    cfg = pipeline.PipelineConfig(layers=4, d=512, heads=4, ffn=1024, vocab=1000, stages=2, r=16, m=16,
                                  batch=2, seq=256, wiring=wiring)
    tokens = pipeline.synthetic_tokens(cfg)
    grads, losses = [], []
    for fuse in (True, False):
        model = pipeline.PipelineModel(cfg.with_(fuse_norm=fuse))
        losses.append(float(pipeline.train_step(model, tokens)))
        grads.append({k: p.grad.float().clone() for k, p in model.named_parameters()})
    assert abs(losses[0] - losses[1]) < 1e-3 * abs(losses[1])
    for k in grads[1]:
        a, b = grads[0][k], grads[1][k]
        rel = float((a - b).norm() / b.norm().clamp_min(1e-30))
        assert rel < 3e-2, (k, rel)
    assert resbm.resbm_device_error() == 0
