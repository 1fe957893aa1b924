"""Pins of the oracle's RMSNorm (the pre-attention norm of the block the decoder starts) and of
its composition with the decoder, to values the definition fixes by hand and to invariants; and
planted mistakes in a copy of the oracle's rmsnorm, each of which some pin must catch (no GPU)."""
import inspect
import textwrap

import numpy as np
import pytest

import oracle


def pin_worked_example(rms):
    """Y = [1, 2, 2]: mean of squares 3, + eps 1 = 4, root 2; gamma = [1, 2, 0.5]."""
    N = rms(np.array([[1.0, 2.0, 2.0]]), np.array([1.0, 2.0, 0.5]), 1.0)
    assert np.array_equal(N, np.array([[0.5, 2.0, 0.5]]))


def pin_constant_row(rms):
    """A constant row c: N_j = c / sqrt(c^2 + eps) gamma_j (c = 3, eps = 7: 3/4 gamma)."""
    g = np.array([1.0, -2.0, 4.0, 0.25])
    N = rms(np.full((2, 4), 3.0), g, 7.0)
    assert np.allclose(N, np.tile(0.75 * g, (2, 1)), rtol=0, atol=1e-15)


def pin_rows_are_independent_and_unit_rms(rms):
    """Each row is normalised on its own; with eps = 0 and gamma = 1 every row has RMS 1 and the
    direction of Y; rows permute with the input."""
    rng = np.random.default_rng(5)
    Y = rng.standard_normal((6, 40)) * np.array([1e-3, 1, 10, 1e3, 0.5, 7])[:, None]
    N = rms(Y, np.ones(40), 0.0)
    assert np.allclose(np.sqrt(np.mean(N * N, axis=1)), 1.0, rtol=1e-14)
    assert np.allclose(N * np.linalg.norm(Y, axis=1)[:, None] / np.sqrt(40), Y, rtol=1e-13)
    perm = rng.permutation(6)
    assert np.array_equal(rms(Y[perm], np.ones(40), 0.0), N[perm])


def pin_scale_invariance_and_eps(rms):
    """With eps = 0, scaling a row by alpha scales N by sign(alpha); eps pulls small rows
    toward zero: a row of RMS s keeps the factor s / sqrt(s^2 + eps)."""
    rng = np.random.default_rng(6)
    Y = rng.standard_normal((3, 16))
    g = rng.standard_normal(16)
    N = rms(Y, g, 0.0)
    assert np.allclose(rms(5.0 * Y, g, 0.0), N, rtol=1e-13)
    assert np.allclose(rms(-0.25 * Y, g, 0.0), -N, rtol=1e-13)
    s = np.sqrt(np.mean(Y * Y, axis=1, keepdims=True))
    assert np.allclose(rms(Y, g, 0.3), N * s / np.sqrt(s * s + 0.3), rtol=1e-13)


PINS = [pin_worked_example, pin_constant_row, pin_rows_are_independent_and_unit_rms,
        pin_scale_invariance_and_eps]


@pytest.mark.parametrize("pin", PINS, ids=lambda p: p.__name__)
def test_oracle_rmsnorm_pins(pin):
    pin(oracle.rmsnorm)


def dpin_zero_second_layer_normalises_the_padded_identity_path(fn):
    """Wd2 = 0, merge = 1: Y = pad(B) exactly, so N's first r columns are B / sqrt(sum_j B_j^2 / d
    + eps) * gamma (the mean runs over all d columns, d - r of them zero) and the rest zero;
    merge = 0: Y = 0 and N = 0."""
    rng = np.random.default_rng(7)
    T, d, r, m = 5, 24, 4, 6
    B = rng.standard_normal((T, r))
    Wd1 = rng.standard_normal((r, m))
    g = rng.standard_normal(d)
    Y, N = fn(B, Wd1, np.zeros((m, d)), g, 0.5)
    assert np.array_equal(Y[:, :r], B) and not np.any(Y[:, r:])
    want = B / np.sqrt(np.sum(B * B, axis=1, keepdims=True) / d + 0.5) * g[:r]
    assert np.allclose(N[:, :r], want, rtol=1e-14) and not np.any(N[:, r:])
    Y0, N0 = fn(B, Wd1, np.zeros((m, d)), g, 0.5, merge=0)
    assert not np.any(Y0) and not np.any(N0)


def dpin_store_rounding_is_applied_before_the_norm(fn):
    """store = "bf16": N is the norm of the bf16 value of Y, and the Y returned is the exact one."""
    rng = np.random.default_rng(8)
    T, d, r, m = 7, 32, 8, 8
    args = (rng.standard_normal((T, r)), rng.standard_normal((r, m)), rng.standard_normal((m, d)) / 3)
    g = rng.standard_normal(d)
    Y, N = fn(*args, g, 1e-5, store="bf16")
    assert np.array_equal(Y, oracle.decode_fwd(*args, "silu", 1))
    Yb = oracle.round_to(Y, "bf16")
    assert np.array_equal(N, oracle.rmsnorm(Yb, g, 1e-5))
    assert not np.array_equal(N, oracle.rmsnorm(Y, g, 1e-5))


DPINS = [dpin_zero_second_layer_normalises_the_padded_identity_path, dpin_store_rounding_is_applied_before_the_norm]


@pytest.mark.parametrize("pin", DPINS, ids=lambda p: p.__name__)
def test_oracle_decode_fwd_rmsnorm_pins(pin):
    pin(oracle.decode_fwd_rmsnorm)


DMUTANTS = {
    "store_ignored": ("Ys = default().round_to(Y, store) if store else Y", "Ys = Y"),
    "returns_the_stored_Y": ("return Y, rmsnorm(Ys, gamma, eps)", "return Ys, rmsnorm(Ys, gamma, eps)"),
    "merge_ignored": ("default().decode_fwd(B, Wd1, Wd2, act, merge)", "default().decode_fwd(B, Wd1, Wd2, act, 1)"),
    "norm_of_the_exact_Y": ("return Y, rmsnorm(Ys, gamma, eps)", "return Y, rmsnorm(Y, gamma, eps)"),
}


@pytest.mark.parametrize("name", sorted(DMUTANTS))
def test_planted_mistake_in_decode_fwd_rmsnorm_is_caught(name):
    find, repl = DMUTANTS[name]
    src = textwrap.dedent(inspect.getsource(oracle.decode_fwd_rmsnorm))
    assert src.count(find) == 1, name
    ns = {"np": np, "default": oracle.default, "rmsnorm": oracle.rmsnorm}
    exec(compile(src.replace(find, repl), "<mutant %s>" % name, "exec"), ns)
    caught = []
    for pin in DPINS:
        try:
            pin(ns["decode_fwd_rmsnorm"])
        except (AssertionError, ValueError, IndexError):
            caught.append(pin.__name__)
    assert caught, "no pin caught the planted mistake %s" % name


MUTANTS = {
    "mean_over_tokens": ("np.mean(Y * Y, axis=1, keepdims=True)", "np.mean(Y * Y, axis=0, keepdims=True)"),
    "sum_not_mean": ("np.mean(Y * Y, axis=1, keepdims=True)", "np.sum(Y * Y, axis=1, keepdims=True)"),
    "eps_outside_root": ("np.sqrt(mean_sq + eps)", "(np.sqrt(mean_sq) + eps)"),
    "no_root": ("np.sqrt(mean_sq + eps)", "(mean_sq + eps)"),
    "gamma_by_row": ("gamma[None, :]", "gamma[:Y.shape[0], None]"),
    "mean_of_abs": ("np.mean(Y * Y, axis=1, keepdims=True)", "np.mean(np.abs(Y), axis=1, keepdims=True) ** 2"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_planted_mistake_in_rmsnorm_is_caught(name):
    find, repl = MUTANTS[name]
    src = textwrap.dedent(inspect.getsource(oracle.rmsnorm))
    assert src.count(find) == 1, name
    ns = {"np": np}
    exec(compile(src.replace(find, repl), "<mutant %s>" % name, "exec"), ns)
    caught = []
    for pin in PINS:
        try:
            pin(ns["rmsnorm"])
        except (AssertionError, ValueError, IndexError):
            caught.append(pin.__name__)
    assert caught, "no pin caught the planted mistake %s" % name


# ---- the backward --------------------------------------------------------------------------

def _fd_grads(Y, g, eps, dN, h=1e-6):
    """Central differences of sum(dN * rmsnorm(Y, g, eps)) in every element of Y and g."""
    f = lambda Y_, g_: float(np.sum(dN * oracle.rmsnorm(Y_, g_, eps)))
    dY = np.zeros_like(Y)
    for idx in np.ndindex(Y.shape):
        e = np.zeros_like(Y); e[idx] = h
        dY[idx] = (f(Y + e, g) - f(Y - e, g)) / (2 * h)
    dg = np.zeros_like(g)
    for j in range(g.size):
        e = np.zeros_like(g); e[j] = h
        dg[j] = (f(Y, g + e) - f(Y, g - e)) / (2 * h)
    return dY, dg


def bpin_finite_differences(bwd):
    rng = np.random.default_rng(11)
    Y = rng.standard_normal((3, 7)) * np.array([0.3, 1.0, 4.0])[:, None]
    g = 1 + 0.2 * rng.standard_normal(7)
    dN = rng.standard_normal((3, 7))
    dY, dg = bwd(Y, g, 0.05, dN)
    fY, fg = _fd_grads(Y, g, 0.05, dN)
    assert np.allclose(dY, fY, rtol=1e-7, atol=1e-8) and np.allclose(dg, fg, rtol=1e-7, atol=1e-8)


def bpin_scale_invariance_makes_dy_orthogonal_to_y(bwd):
    """With eps = 0, N does not change when a row is scaled, so each row's gradient is orthogonal
    to the row itself; and dgamma = sum_t dN * N / gamma."""
    rng = np.random.default_rng(12)
    Y = rng.standard_normal((4, 9))
    g = 1 + 0.1 * rng.standard_normal(9)
    dN = rng.standard_normal((4, 9))
    dY, dg = bwd(Y, g, 0.0, dN)
    assert np.allclose(np.sum(dY * Y, axis=1), 0.0, atol=1e-12)
    assert np.allclose(dg, np.sum(dN * oracle.rmsnorm(Y, g, 0.0) / g, axis=0), rtol=1e-13)


def bpin_incoming_gradient_is_added(bwd):
    rng = np.random.default_rng(13)
    Y, dN, dY0 = (rng.standard_normal((2, 5)) for _ in range(3))
    g = np.ones(5)
    a, ga = bwd(Y, g, 0.1, dN)
    b, gb = bwd(Y, g, 0.1, dN, dY0)
    assert np.allclose(b, a + dY0, rtol=0, atol=1e-15) and np.array_equal(ga, gb)


BPINS = [bpin_finite_differences, bpin_scale_invariance_makes_dy_orthogonal_to_y, bpin_incoming_gradient_is_added]


@pytest.mark.parametrize("pin", BPINS, ids=lambda p: p.__name__)
def test_oracle_rmsnorm_bwd_pins(pin):
    pin(oracle.rmsnorm_bwd)


BMUTANTS = {
    "wrong_power_of_s": ("ds * (-(s ** 3) / d) * Y", "ds * (-(s ** 2) / d) * Y"),
    "missing_1_over_d": ("ds * (-(s ** 3) / d) * Y", "ds * (-(s ** 3)) * Y"),
    "dgamma_from_Y": ("dgamma = np.sum(dN * xhat, axis=0)", "dgamma = np.sum(dN * Y, axis=0)"),
    "ds_without_gamma": ("ds = np.sum(dxhat * Y, axis=1, keepdims=True)", "ds = np.sum(dN * Y, axis=1, keepdims=True)"),
    "sign_of_second_term": ("dxhat * s + ds", "dxhat * s - ds"),
}


@pytest.mark.parametrize("name", sorted(BMUTANTS))
def test_planted_mistake_in_rmsnorm_bwd_is_caught(name):
    find, repl = BMUTANTS[name]
    src = textwrap.dedent(inspect.getsource(oracle.rmsnorm_bwd))
    assert src.count(find) == 1, name
    ns = {"np": np}
    exec(compile(src.replace(find, repl), "<mutant %s>" % name, "exec"), ns)
    caught = []
    for pin in BPINS:
        try:
            pin(ns["rmsnorm_bwd"])
        except (AssertionError, ValueError, IndexError):
            caught.append(pin.__name__)
    assert caught, "no pin caught the planted mistake %s" % name
