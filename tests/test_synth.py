"""The seeded input generator (no GPU)."""
import numpy as np
import torch

from paper_2604_11947_gb300 import synth


def test_splitmix64_published_sequence():
    # SplitMix64 seeded with 0 starts 0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F
    z = np.array([1, 2, 3], dtype=np.uint64) * synth._G
    got = [int(v) for v in synth._mix64_(z)]
    assert got == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]


def test_slices_are_chunking_independent():
    a = synth.normal(0, 2, 0, 1001)
    for i0, n in [(0, 1), (1, 1), (5, 7), (6, 3), (999, 2)]:
        np.testing.assert_array_equal(synth.normal(0, 2, i0, n), a[i0:i0 + n])
    cfg = synth.CONFIGS["single_bf16"].with_(T=300, d=64)
    full = synth.tensor(cfg, "F", chunk_elems=1000)
    np.testing.assert_array_equal(full[17:40], synth.rows(cfg, "F", 17, 40))
    np.testing.assert_array_equal(full[[5, 250]], synth.rows_at(cfg, "F", [5, 250]))


def test_normal_moments_and_streams_differ():
    a = synth.normal(0, 1, 0, 400000)
    assert abs(a.mean()) < 0.01 and abs(a.std() - 1) < 0.01
    assert abs(np.mean(a ** 4) - 3) < 0.05
    b = synth.normal(0, 2, 0, 400000)
    assert abs(np.corrcoef(a, b)[0, 1]) < 0.01
    c = synth.normal(1, 1, 0, 400000)
    assert abs(np.corrcoef(a, c)[0, 1]) < 0.01


def test_bf16_rounding_matches_torch():
    x = (synth.normal(0, 3, 0, 100000) * 50).astype(np.float32)
    mine = synth.round_bf16(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).float().numpy()
    np.testing.assert_array_equal(mine, ref)


def test_weight_scale_and_token_spread():
    cfg = synth.CONFIGS["single_bf16"].with_(T=4096, d=256, r=16, m=16)
    w = synth.tensor(cfg, "We1")
    assert abs(w.std() * np.sqrt(cfg.d) - 1) < 0.02
    s = synth.token_scales(cfg, 0, cfg.T)
    assert abs(np.log(s).std() - 0.5) < 0.02          # log-normal(0, 0.5)
    X = synth.tensor(cfg, "X")
    F = synth.tensor(cfg, "F")
    rx = np.sqrt((X.astype(np.float64) ** 2).mean(1))
    rf = np.sqrt((F.astype(np.float64) ** 2).mean(1))
    assert np.corrcoef(np.log(rx), np.log(rf))[0, 1] > 0.9   # same per-token scale
    assert not np.array_equal(X, F)
