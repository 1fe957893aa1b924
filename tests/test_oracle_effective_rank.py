"""The effective rank of the appendix's spectral analysis (r_eff = sum sigma_i^2 / max sigma_i^2)
against what the definition fixes: orthonormal rows give the bottleneck dimension b, a rank-1
matrix gives 1, a diagonal matrix gives its closed form, and the value depends on the matrix
only through its singular values (orthogonal transforms on either side leave it unchanged).
Planted mistakes in a copy of the oracle's function must each fail some pin (no GPU)."""
import inspect
import textwrap

import numpy as np
import pytest

import oracle


def _orthonormal_rows(b, d, seed):
    q, _ = np.linalg.qr(np.random.default_rng(seed).standard_normal((d, b)))
    return q.T   # b x d, rows orthonormal


def pin_orthonormal_rows_give_the_bottleneck_dimension(reff):
    for b, d in [(32, 4096), (16, 2048), (7, 9), (1, 5)]:
        W = 3.5 * _orthonormal_rows(b, d, seed=b)
        assert reff(W) == pytest.approx(b, rel=1e-12), (b, d)


def pin_rank_one_gives_one(reff):
    rng = np.random.default_rng(1)
    for b, d in [(32, 4096), (4, 4), (1, 1)]:
        W = np.outer(rng.standard_normal(b), rng.standard_normal(d))
        assert reff(W) == pytest.approx(1.0, rel=1e-9), (b, d)


def pin_diagonal_closed_form(reff):
    s = np.array([4.0, 2.0, 1.0, 0.5, 0.0])
    W = np.zeros((5, 8))
    W[np.arange(5), np.arange(5)] = s
    assert reff(W) == pytest.approx((16 + 4 + 1 + 0.25) / 16, rel=1e-14)


def pin_only_the_singular_values_count(reff):
    rng = np.random.default_rng(2)
    W = rng.standard_normal((12, 40))
    U, _ = np.linalg.qr(rng.standard_normal((12, 12)))
    V, _ = np.linalg.qr(rng.standard_normal((40, 40)))
    r = reff(W)
    assert reff(U @ W @ V) == pytest.approx(r, rel=1e-10)
    assert reff(W.T) == pytest.approx(r, rel=1e-12)
    assert reff(-7.0 * W) == pytest.approx(r, rel=1e-12)
    # between 1 and min(rows, cols)
    assert 1.0 <= r <= 12.0


def pin_degenerate_inputs(reff):
    assert reff(np.zeros((3, 4))) == 0.0
    assert reff(np.zeros((0, 4))) == 0.0
    with pytest.raises(ValueError):
        reff(np.zeros(4))


PINS = [pin_orthonormal_rows_give_the_bottleneck_dimension, pin_rank_one_gives_one, pin_diagonal_closed_form,
        pin_only_the_singular_values_count, pin_degenerate_inputs]


@pytest.mark.parametrize("pin", PINS, ids=lambda p: p.__name__)
def test_oracle_effective_rank_pins(pin):
    pin(oracle.effective_rank)


MUTANTS = {
    "singular_values_not_squared": ("float(np.sum(sig * sig)) / top", "float(np.sum(sig)) / top"),
    "largest_not_squared": ("top = float(np.max(sig)) ** 2", "top = float(np.max(sig))"),
    "mean_not_sum": ("np.sum(sig * sig)", "np.mean(sig * sig)"),
    "smallest_singular_value": ("np.max(sig)", "np.min(sig)"),
    "zero_matrix_not_special": ("return 0.0 if top == 0.0 else float", "return float"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_planted_mistake_in_effective_rank_is_caught(name):
    find, repl = MUTANTS[name]
    src = textwrap.dedent(inspect.getsource(oracle.effective_rank))
    assert src.count(find) == 1, name
    ns = {"np": np}
    exec(compile(src.replace(find, repl), "<mutant %s>" % name, "exec"), ns)
    caught = []
    for pin in PINS:
        try:
            pin(ns["effective_rank"])
        except Exception:   # a failed assertion, or an error the mistake causes (0 / 0)
            caught.append(pin.__name__)
    assert caught, "no pin caught the planted mistake %s" % name
