"""Host logic of bench.py that needs no GPU: the roofline's `traffic` comes from the committed
ncu summary only while the kernel sources hash to the value it was captured on, and the
algorithmic-byte model it is compared with."""
import json
import os

import pytest

import bench
from paper_2604_11947_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_traffic_is_read_for_the_sources_it_was_captured_on():
    with open(os.path.join(ROOT, "profiles", "dram_traffic.json")) as f:
        j = json.load(f)
    cfg = synth.CONFIGS["large_bf16"]
    if j["kernel_sources_sha"] != bench.kernel_sources_sha():
        # allowed (the bench then reports traffic as null), but worth knowing
        pytest.skip("profiles/dram_traffic.json was captured on other kernel sources")
    for op in ("enc_fwd", "dec_fwd", "dec_bwd", "enc_bwd"):
        assert bench.traffic_for(op, cfg) == j["ops"][cfg.name][op]["dram_bytes_per_launch"]


def test_traffic_is_dropped_when_the_sources_change(monkeypatch):
    monkeypatch.setattr(bench, "kernel_sources_sha", lambda: "0" * 16)
    assert bench.traffic_for("enc_bwd", synth.CONFIGS["large_bf16"]) is None


@pytest.mark.parametrize("op", ["enc_fwd", "dec_fwd", "dec_bwd", "enc_bwd"])
def test_captured_traffic_is_close_to_the_algorithmic_bytes(op):
    """ncu's DRAM bytes per launch (kernel + its reduction) against the byte model: at most 10 %
    above it (no operand is re-read from DRAM), and below it by no more than what the 129 MB L2
    can still hold dirty when the launch ends (ncu flushes L2 between launches, so that tail of
    the written tensor is not counted)."""
    with open(os.path.join(ROOT, "profiles", "dram_traffic.json")) as f:
        j = json.load(f)
    cfg = synth.CONFIGS["large_bf16"]
    got = j["ops"][cfg.name][op]["dram_bytes_per_launch"]
    alg = bench.op_bytes(cfg)[op]
    assert alg - 129e6 <= got <= 1.1 * alg, (op, got, alg)


def test_rmsnorm_byte_model():
    """The decoder + RMSNorm byte model at T = 65536, d = 4096, r = m = 32: the fused form saves
    the read-back of Y (T d 2 bytes) less its second read of B and its row sums
    (T (2r + 2 * 8 d / 256) bytes); the bench's figure of 515.6 MB."""
    T, d, r, m = 65536, 4096, 32, 32
    a = bench.rmsnorm_alg_bytes(T, d, r, m)
    saved = a["unfused_decode_then_torch_rms_norm"] - a["fused"]
    assert saved == T * 2 * d - T * (2 * r + 16 * (d // 256)) - 2 * (r * m + m * d)
    assert saved == 515635200
    assert a["decode_fwd_alone"] == T * (2 * r + 2 * d) + 2 * (r * m + m * d)
