"""Pins of the fp64 oracle to facts outside the oracle itself.

Each pin takes an oracle instance (`oracle.Oracle`) and raises AssertionError when the oracle
disagrees with what the ResBM paper or plain mathematics fixes. test_oracle_pins.py runs them
on the real oracle; test_oracle_mutants.py runs them on copies of the oracle with a planted
mistake and checks that at least one pin catches each mistake.
"""
import json
import math
import os

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
ACTS = ("silu", "gelu_tanh", "identity")


def _rand(shape, seed, scale=1.0):
    return np.random.default_rng(seed).standard_normal(shape) * scale


def _weights(d, r, m, seed):
    return dict(We1=_rand((d, m), seed + 1, 1 / math.sqrt(d)),
                We2=_rand((m, r), seed + 2, 1 / math.sqrt(m)),
                Wd1=_rand((r, m), seed + 3, 1 / math.sqrt(r)),
                Wd2=_rand((m, d), seed + 4, 1 / math.sqrt(m)))


# ---------------------------------------------------------------------------------------------
# Sec. 3.3: rectangular identity, P^id and their composition.
# ---------------------------------------------------------------------------------------------

def pin_rect_identity_is_numpy_eye(o):
    """Eq. rect_identity_definition equals numpy's rectangular eye for c<C, c>C, c=C."""
    for c, C in [(3, 5), (5, 3), (4, 4), (1, 7), (7, 1)]:
        assert np.array_equal(o.rect_identity(c, C), np.eye(c, C)), (c, C)


def pin_pid_truncate_pad_identity(o):
    """Eq. Pid bullets: c<C appends C-c zero columns, c>C drops the last c-C, c=C is I_c."""
    x = _rand((4, 6), 11)
    y = o.pid(x, 9)
    assert y.shape == (4, 9)
    assert np.array_equal(y[:, :6], x) and not np.any(y[:, 6:])
    assert np.array_equal(o.pid(x, 2), x[:, :2])
    assert np.array_equal(o.pid(x, 6), x)


def pin_composition_rank_min(o):
    """Sec. 3.3: a chain of rectangular identities multiplies to the c0 x cD rectangular
    identity restricted to rank k = min(c0..cD); it is exactly I_{c0 x cD} whenever every
    middle dimension is at least min(c0, cD) (the d -> r -> d round trip is diag(1_r, 0))."""
    chains = [(6, 9, 7, 4), (4, 6, 8), (8, 3, 8), (5, 2, 9, 5), (3, 3, 3), (16, 4, 16, 4)]
    for ch in chains:
        prod = np.eye(ch[0])
        for a, b in zip(ch[:-1], ch[1:]):
            prod = prod @ o.rect_identity(a, b)
        k = min(ch)
        expect = np.zeros((ch[0], ch[-1]))
        expect[np.arange(k), np.arange(k)] = 1.0
        assert np.array_equal(prod, expect), ch
        assert np.linalg.matrix_rank(prod) == k
        if min(ch[1:-1]) >= min(ch[0], ch[-1]):
            assert np.array_equal(prod, np.eye(ch[0], ch[-1])), ch


# ---------------------------------------------------------------------------------------------
# The nonlinearity.
# ---------------------------------------------------------------------------------------------

def pin_act_special_values(o):
    """phi(0) = 0; phi(x) - phi(-x) = x for SiLU and GELU(tanh) (both are x * (an even
    function's complement)); phi -> x for large x and -> 0 for large -x; identity is x."""
    for act in ("silu", "gelu_tanh"):
        assert o.act(act, 0.0) == 0.0
        for x in (0.3, 1.7, 4.2, 9.0):
            assert abs(o.act(act, x) - o.act(act, -x) - x) <= 1e-14 * max(1.0, x)
        assert abs(o.act(act, 40.0) - 40.0) < 1e-12
        assert abs(o.act(act, -40.0)) < 1e-12
    for x in (-3.0, 0.0, 2.5):
        assert o.act("identity", x) == x and o.dact("identity", x) == 1.0


def pin_silu_is_x_sigmoid(o):
    """SiLU(x) = x * sigmoid(x), sigmoid from scipy's expit."""
    from scipy.special import expit
    for x in np.linspace(-12, 12, 49):
        assert abs(o.act("silu", x) - x * expit(x)) <= 1e-15 * max(1.0, abs(x))


def pin_gelu_tanh_close_to_exact_gelu(o):
    """The tanh form of GELU stays within 1e-3 of x * Phi(x) (Phi from math.erf)."""
    for x in np.linspace(-8, 8, 161):
        exact = 0.5 * x * (1.0 + math.erf(x / math.sqrt(2.0)))
        assert abs(o.act("gelu_tanh", x) - exact) < 1e-3, x


def pin_dact_matches_finite_difference(o):
    h = 1e-5
    for act in ACTS:
        for x in np.linspace(-7, 7, 57):
            fd = (o.act(act, x + h) - o.act(act, x - h)) / (2 * h)
            assert abs(fd - o.dact(act, x)) <= 1e-8 * max(1.0, abs(x)), (act, x)


# ---------------------------------------------------------------------------------------------
# The identity path alone (learned contributions zeroed), Sec. 3.2-3.3.
# ---------------------------------------------------------------------------------------------

def pin_zero_weights_leave_identity_path(o):
    T, d, r, m = 5, 12, 4, 3
    X, F, dY = _rand((T, d), 21), _rand((T, d), 22), _rand((T, d), 23)
    w = _weights(d, r, m, 30)
    z_e2, z_d2 = np.zeros((m, r)), np.zeros((m, d))
    for act in ACTS:
        B, _ = o.encode_fwd(X, F, w["We1"], z_e2, act)
        assert np.array_equal(B, X[:, :r])                        # B = X . I_{d x r}
        Bw, _ = o.encode_fwd(X, F, w["We1"], w["We2"], act)
        Y = o.decode_fwd(Bw, w["Wd1"], z_d2, act, merge=1)
        assert np.array_equal(Y[:, :r], Bw) and not np.any(Y[:, r:])  # Y = B . I_{r x d}
        assert not np.any(o.decode_fwd(Bw, w["Wd1"], z_d2, act, merge=0))
        dB, dWd1, _ = o.decode_bwd(dY, Bw, w["Wd1"], z_d2, act, merge=1)
        assert np.array_equal(dB, dY[:, :r]) and not np.any(dWd1)
        dF, dX, _, dWe2 = o.encode_bwd(dB, F, w["We1"], z_e2, act)
        assert not np.any(dF)
        assert np.array_equal(dX[:, :r], dB) and not np.any(dX[:, r:])
    # c = C: with no compression and zero learned weights the block is the vanilla residual
    Xs = _rand((T, 6), 24)
    ws = _weights(6, 6, 2, 40)
    B, _ = o.encode_fwd(Xs, Xs, ws["We1"], np.zeros((2, 6)), "silu")
    assert np.array_equal(o.decode_fwd(B, ws["Wd1"], np.zeros((2, 6)), "silu", 1), Xs)


# ---------------------------------------------------------------------------------------------
# The textbook special case: phi = identity makes encoder and decoder two plain matmuls.
# ---------------------------------------------------------------------------------------------

def pin_identity_act_is_two_matmuls(o):
    T, d, r, m = 6, 10, 3, 4
    X, F, dY = _rand((T, d), 51), _rand((T, d), 52), _rand((T, d), 53)
    w = _weights(d, r, m, 60)
    We1, We2, Wd1, Wd2 = w["We1"], w["We2"], w["Wd1"], w["Wd2"]
    tol = dict(rtol=1e-12, atol=1e-12)
    B, P = o.encode_fwd(X, F, We1, We2, "identity")
    np.testing.assert_allclose(P, np.matmul(F, We1), **tol)
    np.testing.assert_allclose(B, X[:, :r] + np.matmul(np.matmul(F, We1), We2), **tol)
    for merge in (0, 1):
        Y = o.decode_fwd(B, Wd1, Wd2, "identity", merge)
        pad = np.hstack([B, np.zeros((T, d - r))]) * merge
        np.testing.assert_allclose(Y, pad + B @ Wd1 @ Wd2, **tol)
        dB, dWd1, dWd2 = o.decode_bwd(dY, B, Wd1, Wd2, "identity", merge)
        np.testing.assert_allclose(dB, merge * dY[:, :r] + dY @ Wd2.T @ Wd1.T, **tol)
        np.testing.assert_allclose(dWd2, (B @ Wd1).T @ dY, **tol)
        np.testing.assert_allclose(dWd1, B.T @ (dY @ Wd2.T), **tol)
    dBup = _rand((T, r), 54)
    dF, dX, dWe1, dWe2 = o.encode_bwd(dBup, F, We1, We2, "identity")
    np.testing.assert_allclose(dF, dBup @ We2.T @ We1.T, **tol)
    np.testing.assert_allclose(dWe1, F.T @ (dBup @ We2.T), **tol)
    np.testing.assert_allclose(dWe2, (F @ We1).T @ dBup, **tol)
    np.testing.assert_allclose(dX, np.hstack([dBup, np.zeros((T, d - r))]), **tol)


# ---------------------------------------------------------------------------------------------
# Brute force: central finite differences of the scalar sum(dY * Y) through both sides.
# ---------------------------------------------------------------------------------------------

def _fd_check(o, T, d, r, m, act, merge, seed):
    X, F, dY = _rand((T, d), seed), _rand((T, d), seed + 1), _rand((T, d), seed + 2)
    w = _weights(d, r, m, seed + 10)
    params = dict(X=X, F=F, **w)

    def loss(p):
        B, _ = o.encode_fwd(p["X"], p["F"], p["We1"], p["We2"], act)
        return float(np.sum(dY * o.decode_fwd(B, p["Wd1"], p["Wd2"], act, merge)))

    B, _ = o.encode_fwd(X, F, w["We1"], w["We2"], act)
    dB, dWd1, dWd2 = o.decode_bwd(dY, B, w["Wd1"], w["Wd2"], act, merge)
    dF, dX, dWe1, dWe2 = o.encode_bwd(dB, F, w["We1"], w["We2"], act)
    grads = dict(X=dX, F=dF, We1=dWe1, We2=dWe2, Wd1=dWd1, Wd2=dWd2)
    for name, g in grads.items():
        assert g.shape == params[name].shape, name
        scale = max(1.0, float(np.max(np.abs(g))))
        for idx in np.ndindex(*g.shape):
            p = {k: v.copy() for k, v in params.items()}
            x0 = p[name][idx]
            h = 1e-6 * max(1.0, abs(x0))
            p[name][idx] = x0 + h
            lp = loss(p)
            p[name][idx] = x0 - h
            lm = loss(p)
            fd = (lp - lm) / (2 * h)
            assert abs(fd - g[idx]) <= 1e-7 * scale, (act, merge, name, idx, fd, g[idx])


def pin_gradients_match_finite_differences(o):
    # distinct T, d, r, m so that a transposed operand cannot go unnoticed
    for act in ACTS:
        for merge in (1, 0):
            _fd_check(o, T=3, d=7, r=2, m=3, act=act, merge=merge, seed=100)
    _fd_check(o, T=2, d=5, r=4, m=2, act="silu", merge=1, seed=200)   # r > m
    _fd_check(o, T=2, d=3, r=3, m=2, act="silu", merge=1, seed=300)   # r = d (c = C)


def pin_weight_grads_sum_over_tokens(o):
    """The weight gradients are sums over tokens: the gradient of a batch is the sum of the
    gradients of its two halves; the per-token outputs of a row do not depend on the others."""
    T, d, r, m = 8, 9, 2, 3
    X, F, dY = _rand((T, d), 71), _rand((T, d), 72), _rand((T, d), 73)
    w = _weights(d, r, m, 80)
    B, _ = o.encode_fwd(X, F, w["We1"], w["We2"], "silu")
    full = o.decode_bwd(dY, B, w["Wd1"], w["Wd2"], "silu", 1)
    lo = o.decode_bwd(dY[:3], B[:3], w["Wd1"], w["Wd2"], "silu", 1)
    hi = o.decode_bwd(dY[3:], B[3:], w["Wd1"], w["Wd2"], "silu", 1)
    np.testing.assert_array_equal(full[0], np.vstack([lo[0], hi[0]]))
    for k in (1, 2):
        np.testing.assert_allclose(full[k], lo[k] + hi[k], rtol=1e-12, atol=1e-12)
    efull = o.encode_bwd(full[0], F, w["We1"], w["We2"], "silu")
    elo = o.encode_bwd(full[0][:5], F[:5], w["We1"], w["We2"], "silu")
    ehi = o.encode_bwd(full[0][5:], F[5:], w["We1"], w["We2"], "silu")
    for k in (0, 1):
        np.testing.assert_array_equal(efull[k], np.vstack([elo[k], ehi[k]]))
    for k in (2, 3):
        np.testing.assert_allclose(efull[k], elo[k] + ehi[k], rtol=1e-12, atol=1e-12)
    Bsub, _ = o.encode_fwd(X[[6, 1]], F[[6, 1]], w["We1"], w["We2"], "silu")
    np.testing.assert_array_equal(Bsub, B[[6, 1]])


# ---------------------------------------------------------------------------------------------
# One linear layer per side (the single-matrix special case of the encoder / decoder).
# ---------------------------------------------------------------------------------------------

def pin_linear_is_plain_matrix_products(o):
    """One linear layer per side against numpy's matmul, the textbook form of every output."""
    T, d, r = 5, 9, 3
    X, F, dY = _rand((T, d), 401), _rand((T, d), 402), _rand((T, d), 403)
    We, Wd = _rand((d, r), 404, 0.3), _rand((r, d), 405, 0.3)
    tol = dict(rtol=1e-12, atol=1e-12)
    B = o.linear_encode_fwd(X, F, We)
    np.testing.assert_allclose(B, X[:, :r] + F @ We, **tol)
    for merge in (0, 1):
        pad = np.hstack([B, np.zeros((T, d - r))]) * merge
        np.testing.assert_allclose(o.linear_decode_fwd(B, Wd, merge), pad + B @ Wd, **tol)
        dB, dWd = o.linear_decode_bwd(dY, B, Wd, merge)
        np.testing.assert_allclose(dB, merge * dY[:, :r] + dY @ Wd.T, **tol)
        np.testing.assert_allclose(dWd, B.T @ dY, **tol)
    dBup = _rand((T, r), 406)
    dF, dX, dWe = o.linear_encode_bwd(dBup, F, We)
    np.testing.assert_allclose(dF, dBup @ We.T, **tol)
    np.testing.assert_allclose(dWe, F.T @ dBup, **tol)
    np.testing.assert_allclose(dX, np.hstack([dBup, np.zeros((T, d - r))]), **tol)


def pin_linear_is_two_layer_form_with_identity_second_layers(o):
    """The two independent code paths agree: one linear layer per side equals the two-layer
    form with phi = identity and identity matrices as the second layers (We2 = Wd1 = I_r)."""
    T, d, r = 6, 8, 3
    X, F, dY = _rand((T, d), 411), _rand((T, d), 412), _rand((T, d), 413)
    We, Wd = _rand((d, r), 414, 0.3), _rand((r, d), 415, 0.3)
    I = np.eye(r)
    a = o.linear_boundary_step(X, F, dY, We, Wd, merge=1)
    b = o.boundary_step(X, F, dY, We, I, I, Wd, act="identity", merge=1)
    for k in ("B", "Y", "dB", "dF", "dX", "dWe1", "dWd2"):
        np.testing.assert_allclose(a[k], b[k], rtol=1e-12, atol=1e-12, err_msg=k)


def pin_linear_gradients_match_finite_differences(o):
    T, d, r = 3, 7, 2
    X, F, dY = _rand((T, d), 421), _rand((T, d), 422), _rand((T, d), 423)
    params = dict(X=X, F=F, We=_rand((d, r), 424, 0.3), Wd=_rand((r, d), 425, 0.3))
    for merge in (1, 0):
        def loss(p):
            B = o.linear_encode_fwd(p["X"], p["F"], p["We"])
            return float(np.sum(dY * o.linear_decode_fwd(B, p["Wd"], merge)))

        B = o.linear_encode_fwd(X, F, params["We"])
        dB, dWd = o.linear_decode_bwd(dY, B, params["Wd"], merge)
        dF, dX, dWe = o.linear_encode_bwd(dB, F, params["We"])
        grads = dict(X=dX, F=dF, We=dWe, Wd=dWd)
        for name, g in grads.items():
            scale = max(1.0, float(np.max(np.abs(g))))
            for idx in np.ndindex(*g.shape):
                p = {k: v.copy() for k, v in params.items()}
                x0 = p[name][idx]
                h = 1e-6 * max(1.0, abs(x0))
                p[name][idx] = x0 + h
                lp = loss(p)
                p[name][idx] = x0 - h
                lm = loss(p)
                assert abs((lp - lm) / (2 * h) - g[idx]) <= 1e-7 * scale, (merge, name, idx)


def pin_linear_zero_weights_leave_identity_path(o):
    T, d, r = 4, 6, 2
    X, F, dY = _rand((T, d), 431), _rand((T, d), 432), _rand((T, d), 433)
    z = o.linear_boundary_step(X, F, dY, np.zeros((d, r)), np.zeros((r, d)), merge=1)
    np.testing.assert_array_equal(z["B"], X[:, :r])
    np.testing.assert_array_equal(z["Y"], np.hstack([X[:, :r], np.zeros((T, d - r))]))
    np.testing.assert_array_equal(z["dB"], dY[:, :r])
    np.testing.assert_array_equal(z["dF"], np.zeros((T, d)))


# ---------------------------------------------------------------------------------------------
# Transfer rounding of B and dB (they cross the boundary in bf16, Appendix A.3).
# ---------------------------------------------------------------------------------------------

def pin_transfer_rounding_nearest_even(o):
    """bf16 keeps 8 significant bits: between 1 and 2 the spacing is 2^-7. Ties go to the even
    neighbour, values past a tie go up even when fp32 could not hold them, and rounding to
    fp32 keeps 24 bits."""
    r = lambda v: float(o.round_to(np.array([v]), "bf16")[0])  # noqa: E731
    assert r(1.0 + 2 ** -8) == 1.0                       # tie -> even (1.0)
    assert r(1.0 + 3 * 2 ** -8) == 1.0 + 2 ** -6         # tie -> even (1 + 2^-6)
    assert r(-(1.0 + 3 * 2 ** -8)) == -(1.0 + 2 ** -6)
    assert r(1.0 + 2 ** -8 + 2 ** -40) == 1.0 + 2 ** -7  # just above the tie: up
    assert r(1.0 + 2 ** -8 - 2 ** -40) == 1.0            # just below: down
    assert r(3.0 * 2 ** 70) == 3.0 * 2 ** 70 and r(0.0) == 0.0
    assert r(255.5) == 256.0 and r(254.5) == 254.0       # 8 bits: 254 and 256 are neighbours
    f = lambda v: float(o.round_to(np.array([v]), "f32")[0])  # noqa: E731
    assert f(1.0 + 2 ** -24) == 1.0 and f(1.0 + 3 * 2 ** -24) == 1.0 + 2 ** -22
    assert f(1.0 + 2 ** -23) == 1.0 + 2 ** -23


def pin_transfer_rounding_matches_torch_on_fp32_values(o):
    import torch
    x = (np.random.default_rng(7).standard_normal(20000) * 30).astype(np.float32)
    want = torch.from_numpy(x).to(torch.bfloat16).double().numpy()
    np.testing.assert_array_equal(o.round_to(x.astype(np.float64), "bf16"), want)
    y = np.random.default_rng(8).standard_normal(20000) * 1e3
    np.testing.assert_array_equal(o.round_to(y, "f32"), y.astype(np.float32).astype(np.float64))


def pin_step_hands_over_rounded_tensors(o):
    """With bf16 transfer, the decoder sees the bf16 value of B and the encoder backward the
    bf16 value of dB: the step equals the single ops chained on the rounded tensors."""
    T, d, r, m = 5, 16, 4, 3
    X, F, dY = _rand((T, d), 111), _rand((T, d), 112), _rand((T, d), 113)
    w = _weights(d, r, m, 114)
    s = o.boundary_step(X, F, dY, w["We1"], w["We2"], w["Wd1"], w["Wd2"], transfer="bf16")
    B, _ = o.encode_fwd(X, F, w["We1"], w["We2"])
    Bq = o.round_to(B, "bf16")
    assert np.array_equal(s["B"], Bq) and not np.array_equal(Bq, B)
    np.testing.assert_array_equal(s["Y"], o.decode_fwd(Bq, w["Wd1"], w["Wd2"]))
    dB, _, _ = o.decode_bwd(dY, Bq, w["Wd1"], w["Wd2"])
    np.testing.assert_array_equal(s["dB"], o.round_to(dB, "bf16"))
    np.testing.assert_array_equal(s["dF"], o.encode_bwd(o.round_to(dB, "bf16"), F, w["We1"], w["We2"])[0])



def pin_linear_step_hands_over_rounded_tensors(o):
    """The one-linear-layer step with bf16 transfer: the decoder sees the bf16 value of B and the
    encoder backward the bf16 value of dB, as in the two-layer step."""
    T, d, r = 5, 16, 4
    X, F, dY = _rand((T, d), 121), _rand((T, d), 122), _rand((T, d), 123)
    We, Wd = _rand((d, r), 124, 0.25), _rand((r, d), 125, 0.5)
    s = o.linear_boundary_step(X, F, dY, We, Wd, transfer="bf16")
    Bq = o.round_to(o.linear_encode_fwd(X, F, We), "bf16")
    assert np.array_equal(s["B"], Bq)
    np.testing.assert_array_equal(s["Y"], o.linear_decode_fwd(Bq, Wd))
    dB, _ = o.linear_decode_bwd(dY, Bq, Wd)
    dBq = o.round_to(dB, "bf16")
    assert np.array_equal(s["dB"], dBq) and not np.array_equal(dBq, dB)
    np.testing.assert_array_equal(s["dF"], o.linear_encode_bwd(dBq, F, We)[0])

# ---------------------------------------------------------------------------------------------
# Appendix A.3 / Sec. 4.1: what crosses the boundary.
# ---------------------------------------------------------------------------------------------

def pin_boundary_bytes(o):
    with open(os.path.join(GOLDEN, "appendix_a3_bytes.json")) as f:
        g = json.load(f)["facts"]
    T = g["microbatch"] * g["tokens_per_boundary_message"]
    d, r, m, e = g["hidden_dim"], g["bottleneck_dim_128x"], g["bottleneck_dim_128x"], g["bytes_per_element_bf16"]
    assert d // r == g["compression_rate"]
    X = _rand((T, d), 91)
    w = _weights(d, r, m, 92)
    B, _ = o.encode_fwd(X, X, w["We1"], w["We2"], "silu")
    assert X.size * e == g["uncompressed_boundary_bytes"]
    assert B.shape == (T, r) and B.size * e == g["compressed_boundary_bytes"]
    dB, _, _ = o.decode_bwd(X, B, w["Wd1"], w["Wd2"], "silu", 1)   # the gradient sent back
    assert dB.shape == (T, r)
    per_step = g["stage_boundaries"] * g["directions"]
    assert per_step * X.size * e == g["uncompressed_step_bytes"]
    assert per_step * (B.size + dB.size) // 2 * e == g["compressed_step_bytes"]


def pin_encoder_saves_the_preactivation(o):
    """The saved P is F . We1 before phi (Sec. 3.2's encoder; the backward needs phi'(P)), by
    brute-force loops on a tiny case with nonlinear phi, where P and phi(P) differ."""
    T, d, r, m = 3, 5, 2, 4
    X, F = _rand((T, d), 71), _rand((T, d), 72)
    w = _weights(d, r, m, 73)
    for act in ("silu", "gelu_tanh"):
        _, P = o.encode_fwd(X, F, w["We1"], w["We2"], act)
        for t in range(T):
            for i in range(m):
                want = sum(F[t, j] * w["We1"][j, i] for j in range(d))
                assert abs(P[t, i] - want) <= 1e-13 * (1.0 + abs(want)), (act, t, i)


PINS = [v for k, v in sorted(globals().items()) if k.startswith("pin_")]
