"""Pins of the oracle's Newton-Schulz orthogonalisation (Muon's update direction) to what the
iteration fixes, by routes that share nothing with its matrix-product form: the iteration acts on
the singular values alone (an odd polynomial of X X^T times X), so it equals the SVD with the
scalar quintic map applied to each normalised singular value."""
import numpy as np
import pytest

import oracle


def _via_svd(G, steps, coeffs=oracle.NS_COEFFS, eps=1e-7):
    a, b, c = coeffs
    U, s, Vt = np.linalg.svd(np.asarray(G, np.float64), full_matrices=False)
    x = s / (np.sqrt(np.sum(s * s)) + eps)      # ||G||_F from the singular values
    for _ in range(steps):
        x = a * x + b * x ** 3 + c * x ** 5      # p(x) = a x + b x^3 + c x^5 per singular value
    return (U * x) @ Vt


@pytest.mark.parametrize("shape", [(8, 64), (64, 8), (24, 24), (16, 200)])
@pytest.mark.parametrize("steps", [0, 1, 5])
def test_matches_scalar_map_on_singular_values(shape, steps):
    rng = np.random.default_rng(1)
    G = rng.standard_normal(shape)
    assert np.allclose(oracle.newton_schulz(G, steps), _via_svd(G, steps), atol=1e-10)


def test_step_zero_is_the_frobenius_normalisation():
    G = np.arange(12.0).reshape(3, 4) - 5.0
    assert np.allclose(oracle.newton_schulz(G, 0), G / (np.sqrt(np.sum(G * G)) + 1e-7))


def test_transpose_and_orthogonal_invariance():
    rng = np.random.default_rng(2)
    G = rng.standard_normal((16, 48))
    X = oracle.newton_schulz(G, 5)
    assert np.allclose(oracle.newton_schulz(G.T, 5), X.T, atol=1e-12)
    Q, _ = np.linalg.qr(rng.standard_normal((16, 16)))
    R, _ = np.linalg.qr(rng.standard_normal((48, 48)))
    assert np.allclose(oracle.newton_schulz(Q @ G @ R, 5), Q @ X @ R, atol=1e-10)


def test_five_steps_drive_singular_values_into_a_band_around_one():
    """The quintic's design: five steps from ||X||_F = 1 push every not-too-small singular value
    into roughly [0.7, 1.2] (the iteration does not converge to exactly 1)."""
    rng = np.random.default_rng(3)
    G = rng.standard_normal((32, 512))
    s = np.linalg.svd(oracle.newton_schulz(G, 5), compute_uv=False)
    assert s.min() > 0.6 and s.max() < 1.25
    # and the singular vectors stay G's: X^T X commutes with G^T G's eigenbasis
    U, _, Vt = np.linalg.svd(G, full_matrices=False)
    X = oracle.newton_schulz(G, 5)
    D = U.T @ X @ Vt.T
    assert np.allclose(D - np.diag(np.diag(D)), 0.0, atol=1e-10)
