"""The parity metric itself (CPU): bf16 errors are measured against the RMS of the output (per
token row for per-token outputs), with no per-element |o| term beyond the output's own rounding
(half a bf16 spacing)."""
import numpy as np
import pytest
import torch

from metrics import bf16_half_spacing, check, rel_err


def test_bf16_large_element_is_held_to_the_row_rms():
    o = np.ones((2, 8))
    o[0, 3] = 5.0                       # an element 5x the typical size of its row
    rms0 = np.sqrt(np.mean(o[0] ** 2))
    g = o.copy()
    g[0, 3] += 0.03 * rms0              # 3 % of the row's RMS (0.6 % of the element itself)
    h = bf16_half_spacing(g[0, 3])      # the output rounding is not charged
    assert rel_err(g, o, "bf16", rowwise=True) == pytest.approx(0.03 - h / rms0)
    with pytest.raises(AssertionError):
        check("Y", g, o, "bf16")


def test_bf16_rows_have_their_own_scale():
    o = np.vstack([np.full(4, 100.0), np.full(4, 0.01)])
    g = o.copy()
    g[1, 0] += 0.01 * 0.015             # 1.5 % of the small row's RMS
    h = bf16_half_spacing(g[1, 0])
    assert rel_err(g, o, "bf16", rowwise=True) == pytest.approx(0.015 - h / 0.01)
    check("dF", g, o, "bf16")
    # over the whole tensor (weight gradients) the small row's error is negligible
    assert rel_err(g, o, "bf16", rowwise=False) < 1e-5


def test_fp32_weight_gradients_get_no_rounding_allowance():
    """The weight gradients of a bf16 workload are fp32 outputs: their whole error counts."""
    o = np.array([[1.0, -1.0, 1.0, -1.0]])
    g = o.copy()
    g[0, 0] += 2.0 ** -10             # within half a bf16 spacing of 1.0, but a real fp32 error
    assert rel_err(g, o, "bf16", rowwise=False) == pytest.approx(2.0 ** -10)
    assert rel_err(g, o, "bf16", rowwise=True) == 0.0


def test_f32_is_relative_with_an_rms_floor():
    o = np.array([[1.0, 1e-9, -2.0, 0.5]])
    g = o.copy()
    g[0, 0] *= 1 + 5e-6
    g[0, 1] = 0.0                       # near-zero element: judged against the RMS
    assert rel_err(g, o, "f32", rowwise=False) <= 1e-5
    check("B", g, o, "f32")
    g[0, 2] *= 1 + 2e-5
    with pytest.raises(AssertionError):
        check("B", g, o, "f32")


def test_half_spacing_is_the_bf16_rounding_bound():
    rng = np.random.default_rng(0)
    x = rng.standard_normal(20000) * np.exp(rng.standard_normal(20000) * 3)
    xb = torch.from_numpy(x.astype(np.float32)).to(torch.bfloat16).double().numpy()
    # rounding fp32 -> bf16 moves a value by at most half a spacing (plus the fp32 step)
    assert np.all(np.abs(xb - x) <= bf16_half_spacing(np.maximum(np.abs(x), np.abs(xb))) * (1 + 2 ** -15))
    assert bf16_half_spacing(2.0) == 2.0 ** -7 and bf16_half_spacing(3.99) == 2.0 ** -7
    assert bf16_half_spacing(0.0) == 0.0


def test_bf16_correctly_rounded_outlier_passes_one_spacing_off_fails():
    """A row whose RMS is small next to one element (the identity-path columns of Y for a
    large-norm token): the correctly rounded value passes, one bf16 step more does not."""
    o = np.full((1, 16), 0.3)
    o[0, 0] = 2.0235155                 # ~6.5x the row's RMS
    g = o.copy()
    g[0, 0] = 2.03125                   # round_bf16(2.0235155)
    assert rel_err(g, o, "bf16", rowwise=True) == 0.0
    g[0, 0] = 2.03125 + 2.0 ** -6       # the next bf16 value
    with pytest.raises(AssertionError):
        check("Y", g, o, "bf16")


def test_carried_rounding_allowance():
    """An output computed from another rounded output (N from the stored Y) gets `allow` per
    element on top of its own half spacing, and nothing more."""
    o = np.ones((1, 100))
    o[0, ::2] = -1.0
    o[0, 0] = 4.98                                     # row RMS ~1.1
    carried = np.zeros_like(o)
    carried[0, 0] = 2.0 ** -6                          # half of Y's spacing at ~5, times rstd * gamma ~ 1
    g = o.copy()
    g[0, 0] = 5.03125                                  # the neighbouring value past both roundings
    with pytest.raises(AssertionError):
        check("N", g, o, "bf16")
    assert check("N", g, o, "bf16", allow=carried) <= 2e-2
    g[0, 1] += 0.05                                    # an element without a carried rounding
    with pytest.raises(AssertionError):
        check("N", g, o, "bf16", allow=carried)
