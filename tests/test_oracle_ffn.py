"""Pins of the oracle's encoder-after-the-down-projection (Sec. 3.2: the bottleneck follows the
feed-forward layer) to brute force and to the special cases the composition fixes; planted
mistakes in a copy of the oracle's function must each fail some pin (no GPU)."""
import inspect
import textwrap

import numpy as np
import pytest

import oracle


def _bf16(x):
    return oracle.round_to(x, "bf16")


def pin_brute_force_tiny(fde):
    rng = np.random.default_rng(5)
    T, f, d, r, m = 3, 5, 4, 2, 2
    H, W2, X = _bf16(rng.standard_normal((T, f))), _bf16(rng.standard_normal((f, d))), _bf16(rng.standard_normal((T, d)))
    We1, We2 = _bf16(rng.standard_normal((d, m))), _bf16(rng.standard_normal((m, r)))
    B, P, F = fde(H, W2, X, We1, We2, "silu")
    silu = lambda x: x / (1.0 + np.exp(-x))
    for t in range(T):
        Fr = [oracle.round_to(sum(H[t, k] * W2[k, j] for k in range(f)), "bf16") for j in range(d)]
        assert np.allclose(F[t], Fr, rtol=0, atol=0)
        Pt = [sum(Fr[j] * We1[j, i] for j in range(d)) for i in range(m)]
        assert np.allclose(P[t], Pt, rtol=1e-14)
        Bt = [X[t, n] + sum(silu(Pt[i]) * We2[i, n] for i in range(m)) for n in range(r)]
        assert np.allclose(B[t], Bt, rtol=1e-13)


def pin_zero_down_projection_leaves_the_identity_path(fde):
    rng = np.random.default_rng(6)
    H, X = _bf16(rng.standard_normal((6, 16))), _bf16(rng.standard_normal((6, 8)))
    B, P, F = fde(H, np.zeros((16, 8)), X, _bf16(rng.standard_normal((8, 4))), _bf16(rng.standard_normal((4, 2))),
                  "silu")
    assert not np.any(F) and not np.any(P)
    assert np.array_equal(B, X[:, :2])          # phi(0) = 0 for SiLU: B = X[:, :r]


def pin_identity_down_projection_is_the_plain_encoder(fde):
    rng = np.random.default_rng(7)
    H, X = _bf16(rng.standard_normal((5, 8))), _bf16(rng.standard_normal((5, 8)))
    We1, We2 = _bf16(rng.standard_normal((8, 4))), _bf16(rng.standard_normal((4, 4)))
    B, P, F = fde(H, np.eye(8), X, We1, We2, "gelu_tanh")
    B2, P2 = oracle.encode_fwd(X, H, We1, We2, "gelu_tanh")
    assert np.array_equal(F, H) and np.array_equal(B, B2) and np.array_equal(P, P2)


PINS = [pin_brute_force_tiny, pin_zero_down_projection_leaves_the_identity_path,
        pin_identity_down_projection_is_the_plain_encoder]


@pytest.mark.parametrize("pin", PINS, ids=lambda p: p.__name__)
def test_oracle_ffn_down_encode_pins(pin):
    pin(oracle.ffn_down_encode_fwd)


MUTANTS = {
    "F_not_rounded": ('default().round_to(np.asarray(H, np.float64) @ np.asarray(W2, np.float64), "bf16")',
                      "np.asarray(H, np.float64) @ np.asarray(W2, np.float64)"),
    "F_rounded_to_fp32": ('np.asarray(W2, np.float64), "bf16")', 'np.asarray(W2, np.float64), "f32")'),
    "encoder_reads_X": ("encode_fwd(X, F, We1, We2, act)", "encode_fwd(X, X, We1, We2, act)"),
    "down_projection_transposed": ("@ np.asarray(W2, np.float64)", "@ np.asarray(W2, np.float64).T"),
    "activation_fixed": ("encode_fwd(X, F, We1, We2, act)", 'encode_fwd(X, F, We1, We2, "silu")'),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_planted_mistake_in_ffn_down_encode_is_caught(name):
    find, repl = MUTANTS[name]
    src = textwrap.dedent(inspect.getsource(oracle.ffn_down_encode_fwd))
    assert src.count(find) == 1, name
    ns = {"np": np, "default": oracle.default}
    exec(compile(src.replace(find, repl), "<mutant %s>" % name, "exec"), ns)
    caught = []
    for pin in PINS:
        try:
            pin(ns["ffn_down_encode_fwd"])
        except Exception:   # a failed assertion, or a shape error the mistake causes
            caught.append(pin.__name__)
    assert caught, "no pin caught the planted mistake %s" % name
