"""Host-side pieces of the simulated pipeline (no GPU): the model's structure and the learnable
synthetic token stream of the convergence comparison."""
import math

import numpy as np
import torch

from paper_2604_11947_gb300 import pipeline


def test_markov_stream_follows_its_chain():
    cfg = pipeline.CONVERGENCE
    t, rate = pipeline.markov_batches(cfg, 2, device="cpu")
    assert t.shape == (2, cfg.batch, cfg.seq) and int(t.min()) >= 0 and int(t.max()) < cfg.vocab
    # the same seed gives the same stream; each token has at most `branching` successors
    t2, _ = pipeline.markov_batches(cfg, 2, device="cpu")
    assert torch.equal(t, t2)
    a = t.reshape(-1, cfg.seq).numpy()
    succ = {}
    for row in a:
        for x, y in zip(row[:-1], row[1:]):
            succ.setdefault(int(x), set()).add(int(y))
    assert max(len(v) for v in succ.values()) <= 4
    # the entropy rate lies between 0 and log(branching), far below the uniform log(vocab)
    assert 0.0 < rate < math.log(4) < math.log(cfg.vocab)


def test_model_structure():
    cfg = pipeline.PipelineConfig(layers=4, d=64, heads=4, ffn=128, vocab=50, stages=2, r=8, m=8, batch=2, seq=16)
    m = pipeline.PipelineModel(cfg, device="cpu")
    assert len(m.blocks) == 4 and len(m.bounds) == 1
    b = m.bounds[0]
    assert b.We1.shape == (64, 8) and b.We2.shape == (8, 8) and b.Wd1.shape == (8, 8) and b.Wd2.shape == (8, 64)
    assert b.merge == 1 and pipeline.PipelineModel(cfg.with_(wiring="B"), device="cpu").bounds[0].merge == 0
    # the full workload: 24 layers in 4 stages, three boundaries of 128x compression
    full = pipeline.PIPELINE
    assert full.layers // full.stages == 6 and full.d // full.r == 128 and full.tokens == 16384


def test_per_boundary_widths():
    cfg = pipeline.PipelineConfig(layers=4, d=64, heads=4, ffn=128, vocab=50, stages=4, r=(8, 16, 32), m=(8, 16, 32),
                                  batch=2, seq=16)
    assert [cfg.boundary_widths(k) for k in range(3)] == [(8, 8), (16, 16), (32, 32)]
    m = pipeline.PipelineModel(cfg, device="cpu")
    assert [(b.r, b.m) for b in m.bounds] == [(8, 8), (16, 16), (32, 32)]
    assert m.bounds[2].We2.shape == (32, 32) and m.bounds[0].Wd2.shape == (8, 64)
    assert pipeline.PIPELINE.boundary_widths(2) == (16, 16)
