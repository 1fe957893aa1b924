"""The effective rank of the appendix's spectral analysis (r_eff = sum sigma_i^2 / max sigma_i^2)
against what the definition fixes: orthonormal rows give the bottleneck dimension b, a rank-1
matrix gives 1, a diagonal matrix gives its closed form, and the value depends on the matrix
only through its singular values (orthogonal transforms on either side leave it unchanged)."""
import numpy as np
import pytest

import oracle


def _orthonormal_rows(b, d, seed):
    q, _ = np.linalg.qr(np.random.default_rng(seed).standard_normal((d, b)))
    return q.T   # b x d, rows orthonormal


@pytest.mark.parametrize("b,d", [(32, 4096), (16, 2048), (7, 9), (1, 5)])
def test_orthonormal_rows_give_the_bottleneck_dimension(b, d):
    W = 3.5 * _orthonormal_rows(b, d, seed=b)
    assert oracle.effective_rank(W) == pytest.approx(b, rel=1e-12)


@pytest.mark.parametrize("b,d", [(32, 4096), (4, 4), (1, 1)])
def test_rank_one_gives_one(b, d):
    rng = np.random.default_rng(1)
    W = np.outer(rng.standard_normal(b), rng.standard_normal(d))
    assert oracle.effective_rank(W) == pytest.approx(1.0, rel=1e-9)


def test_diagonal_closed_form():
    s = np.array([4.0, 2.0, 1.0, 0.5, 0.0])
    W = np.zeros((5, 8))
    W[np.arange(5), np.arange(5)] = s
    assert oracle.effective_rank(W) == pytest.approx((16 + 4 + 1 + 0.25) / 16, rel=1e-14)


def test_only_the_singular_values_count():
    rng = np.random.default_rng(2)
    W = rng.standard_normal((12, 40))
    U, _ = np.linalg.qr(rng.standard_normal((12, 12)))
    V, _ = np.linalg.qr(rng.standard_normal((40, 40)))
    r = oracle.effective_rank(W)
    assert oracle.effective_rank(U @ W @ V) == pytest.approx(r, rel=1e-10)
    assert oracle.effective_rank(W.T) == pytest.approx(r, rel=1e-12)
    assert oracle.effective_rank(-7.0 * W) == pytest.approx(r, rel=1e-12)
    # between 1 and min(rows, cols)
    assert 1.0 <= r <= 12.0


def test_degenerate_inputs():
    assert oracle.effective_rank(np.zeros((3, 4))) == 0.0
    assert oracle.effective_rank(np.zeros((0, 4))) == 0.0
    with pytest.raises(ValueError):
        oracle.effective_rank(np.zeros(4))
