"""Pins of the oracle's Newton-Schulz orthogonalisation (Muon's update direction) to what the
iteration fixes, by routes that share nothing with its matrix-product form: the iteration acts on
the singular values alone (an odd polynomial of X X^T times X), so it equals the SVD with the
scalar quintic map applied to each normalised singular value. Planted mistakes in a copy of the
oracle's function must each fail some pin (no GPU)."""
import inspect
import textwrap

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


def pin_matches_scalar_map_on_singular_values(ns):
    rng = np.random.default_rng(1)
    for shape in [(8, 64), (64, 8), (24, 24), (16, 200)]:
        G = rng.standard_normal(shape)
        for steps in (0, 1, 5):
            assert np.allclose(ns(G, steps), _via_svd(G, steps), atol=1e-10), (shape, steps)


def pin_step_zero_is_the_frobenius_normalisation(ns):
    G = np.arange(12.0).reshape(3, 4) - 5.0
    assert np.allclose(ns(G, 0), G / (np.sqrt(np.sum(G * G)) + 1e-7))


def pin_transpose_and_orthogonal_invariance(ns):
    rng = np.random.default_rng(2)
    G = rng.standard_normal((16, 48))
    X = ns(G, 5)
    assert np.allclose(ns(G.T, 5), X.T, atol=1e-12)
    Q, _ = np.linalg.qr(rng.standard_normal((16, 16)))
    R, _ = np.linalg.qr(rng.standard_normal((48, 48)))
    assert np.allclose(ns(Q @ G @ R, 5), Q @ X @ R, atol=1e-10)


def pin_five_steps_drive_singular_values_into_a_band_around_one(ns):
    """The quintic's design: five steps from ||X||_F = 1 push every not-too-small singular value
    into roughly [0.7, 1.2] (the iteration does not converge to exactly 1)."""
    rng = np.random.default_rng(3)
    G = rng.standard_normal((32, 512))
    X = ns(G, 5)
    s = np.linalg.svd(X, compute_uv=False)
    assert s.min() > 0.6 and s.max() < 1.25
    # and the singular vectors stay G's: X^T X commutes with G^T G's eigenbasis
    U, _, Vt = np.linalg.svd(G, full_matrices=False)
    D = U.T @ X @ Vt.T
    assert np.allclose(D - np.diag(np.diag(D)), 0.0, atol=1e-10)


PINS = [pin_matches_scalar_map_on_singular_values, pin_step_zero_is_the_frobenius_normalisation,
        pin_transpose_and_orthogonal_invariance, pin_five_steps_drive_singular_values_into_a_band_around_one]


@pytest.mark.parametrize("pin", PINS, ids=lambda p: p.__name__)
def test_oracle_newton_schulz_pins(pin):
    pin(oracle.newton_schulz)


MUTANTS = {
    "b_and_c_swapped": ("B = b * A + c * (A @ A)", "B = c * A + b * (A @ A)"),
    "spectral_norm_not_frobenius": ("np.linalg.norm(G)", "np.linalg.norm(G, 2)"),
    "no_normalisation": ("X = G / (np.linalg.norm(G) + eps)", "X = G / (1.0 + eps)"),
    "polynomial_applied_on_the_right": ("X = a * X + B @ X", "X = a * X + X @ B"),
    "linear_coefficient_dropped": ("X = a * X + B @ X", "X = X + B @ X"),
    "gram_of_the_columns": ("A = X @ X.T", "A = X.T @ X"),
    "one_step_fewer": ("for _ in range(steps):", "for _ in range(steps - 1):"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_planted_mistake_in_newton_schulz_is_caught(name):
    find, repl = MUTANTS[name]
    src = textwrap.dedent(inspect.getsource(oracle.newton_schulz))
    assert src.count(find) == 1, name
    ns = {"np": np, "NS_COEFFS": oracle.NS_COEFFS}
    exec(compile(src.replace(find, repl), "<mutant %s>" % name, "exec"), ns)
    caught = []
    for pin in PINS:
        try:
            pin(ns["newton_schulz"])
        except Exception:   # a failed assertion, or a shape error the mistake causes
            caught.append(pin.__name__)
    assert caught, "no pin caught the planted mistake %s" % name
