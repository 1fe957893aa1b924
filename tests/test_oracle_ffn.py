"""Pins of the oracle's encoder-after-the-down-projection (Sec. 3.2: the bottleneck follows the
feed-forward layer) to brute force and to the special cases the composition fixes."""
import numpy as np

import oracle


def _bf16(x):
    return oracle.round_to(x, "bf16")


def test_brute_force_tiny():
    rng = np.random.default_rng(5)
    T, f, d, r, m = 3, 5, 4, 2, 2
    H, W2, X = _bf16(rng.standard_normal((T, f))), _bf16(rng.standard_normal((f, d))), _bf16(rng.standard_normal((T, d)))
    We1, We2 = _bf16(rng.standard_normal((d, m))), _bf16(rng.standard_normal((m, r)))
    B, P, F = oracle.ffn_down_encode_fwd(H, W2, X, We1, We2, "silu")
    silu = lambda x: x / (1.0 + np.exp(-x))
    for t in range(T):
        Fr = [oracle.round_to(sum(H[t, k] * W2[k, j] for k in range(f)), "bf16") for j in range(d)]
        assert np.allclose(F[t], Fr, rtol=0, atol=0)
        Pt = [sum(Fr[j] * We1[j, i] for j in range(d)) for i in range(m)]
        assert np.allclose(P[t], Pt, rtol=1e-14)
        Bt = [X[t, n] + sum(silu(Pt[i]) * We2[i, n] for i in range(m)) for n in range(r)]
        assert np.allclose(B[t], Bt, rtol=1e-13)


def test_zero_down_projection_leaves_the_identity_path():
    rng = np.random.default_rng(6)
    H, X = _bf16(rng.standard_normal((6, 16))), _bf16(rng.standard_normal((6, 8)))
    B, P, F = oracle.ffn_down_encode_fwd(H, np.zeros((16, 8)), X, _bf16(rng.standard_normal((8, 4))),
                                         _bf16(rng.standard_normal((4, 2))), "silu")
    assert not np.any(F) and not np.any(P)
    assert np.array_equal(B, X[:, :2])          # phi(0) = 0 for SiLU: B = X[:, :r]


def test_identity_down_projection_is_the_plain_encoder():
    rng = np.random.default_rng(7)
    H, X = _bf16(rng.standard_normal((5, 8))), _bf16(rng.standard_normal((5, 8)))
    We1, We2 = _bf16(rng.standard_normal((8, 4))), _bf16(rng.standard_normal((4, 4)))
    B, P, F = oracle.ffn_down_encode_fwd(H, np.eye(8), X, We1, We2, "gelu_tanh")
    B2, P2 = oracle.encode_fwd(X, H, We1, We2, "gelu_tanh")
    assert np.array_equal(F, H) and np.array_equal(B, B2) and np.array_equal(P, P2)
