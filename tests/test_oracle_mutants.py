"""Planted mistakes in a copy of the oracle must each fail at least one pin (no GPU).

Every mutant is a one-line textual change to a temporary copy of oracle/resbm_oracle.c (the
committed oracle is never touched); each keeps all memory accesses in bounds.
"""
import os
import tempfile

import pytest

import oracle
from oracle import build as obuild
from oracle_pins import PINS

MUTANTS = {
    "dropped_send_skip": ("B[i] = S[i] + E[i];", "B[i] = E[i];"),
    "wrong_sign_receive_merge": ("Y[i] = merge ? R[i] + D[i] : D[i];",
                                 "Y[i] = merge ? R[i] - D[i] : D[i];"),
    "silu_derivative_sign": ("return s + x * s * (1.0 - s);", "return s + x * s * (1.0 + s);"),
    "dact_at_wrong_tensor": ("dQ[i] = dG[i] * oracle_dact(act, Q[i]);",
                             "dQ[i] = dG[i] * oracle_dact(act, G[i]);"),
    "missing_dact_in_encoder": ("dP[i] = dA[i] * oracle_dact(act, P[i]);", "dP[i] = dA[i];"),
    "dropped_skip_gradient": ("        if (merge) {\n            rc = pid_backward",
                              "        if (0) {\n            rc = pid_backward"),
    "identity_on_antidiagonal": ("I[i * C + j] = (i == j) ? 1.0 : 0.0;",
                                 "I[i * C + j] = (i == C - 1 - j) ? 1.0 : 0.0;"),
    "gelu_constant": ("kGeluC = 0.044715;", "kGeluC = 0.44715;"),
    "dropped_first_token_in_reduction": (
        "        for (int64_t k = 0; k < K; ++k) {\n            const double a = A[k * M + i];",
        "        for (int64_t k = 1; k < K; ++k) {\n            const double a = A[k * M + i];"),
    "transposed_operand_in_nt_product": ("acc += A[i * K + k] * B[j * K + k];",
                                         "acc += A[i * K + k] * B[k * N + j];"),
    "encoder_reads_decoder_order": ("mm_nn(T, r, m, A, We2, E);", "mm_nn(T, r, m, P, We2, E);"),
    "rounding_ties_away_from_zero": ("double r = nearbyint(scaled);", "double r = round(scaled);"),
    "rounding_keeps_one_bit_less": ("double scaled = ldexp(f, bits);",
                                    "double scaled = ldexp(f, bits - 1);"),
    "linear_decoder_bwd_transposed": ("mm_nt(T, r, d, dY, Wd, dB);              /* dB  = dY . Wd^T         */",
                                      "mm_nn(T, r, d, dY, Wd, dB);              /* dB  = dY . Wd^T         */"),
    "linear_encoder_bwd_drops_dX": ("return dX ? pid_backward(T, d, r, dB, dX) : 0;", "return 0;"),
    "gelu_derivative_drops_factor_3": ("double du = kSqrt2OverPi * (1.0 + 3.0 * kGeluC * x * x);",
                                       "double du = kSqrt2OverPi * (1.0 + kGeluC * x * x);"),
    "gelu_derivative_tanh_sign": ("0.5 * x * (1.0 - th * th) * du", "0.5 * x * (1.0 + th * th) * du"),
    "identity_derivative_zero": ("    return 1.0;\n}", "    return 0.0;\n}"),
    "linear_decoder_drops_padded_skip": ("Y[i] = merge ? Pad[i] + L[i] : L[i];", "Y[i] = L[i];"),
    "encoder_saves_activation_for_P": ("if (P_out) memcpy(P_out, P,", "if (P_out) memcpy(P_out, A,"),
    "decoder_gradient_from_Q_for_G": ("mm_tn(m, d, T, G, dY, dWd2);", "mm_tn(m, d, T, Q, dY, dWd2);"),
    "encoder_gradient_from_P_for_A": ("mm_tn(m, r, T, A, dB, dWe2);", "mm_tn(m, r, T, P, dB, dWe2);"),
    "decoder_skips_activation": ("apply_act(act, T * m, Q, G);\n        mm_nn(T, d, m, G, Wd2, D);",
                                 "apply_act(act, T * m, Q, G);\n        mm_nn(T, d, m, Q, Wd2, D);"),
    "rounding_ties_down": ("double r = nearbyint(scaled);", "double r = floor(scaled);"),
    "rounding_skips_small_magnitudes": ("if (x == 0.0 || !isfinite(x)) return x;",
                                        "if (x == 0.0 || !isfinite(x) || fabs(x) < 1.0) return x;"),
    "nn_product_drops_last_k": ("        for (int64_t k = 0; k < K; ++k) {\n            const double a = A[i * K + k];",
                                "        for (int64_t k = 0; k < K - 1; ++k) {\n            const double a = A[i * K + k];"),
    "identity_backward_not_transposed": ("mm_nt(L, c, C, dy, I, dx);", "mm_nn(L, c, C, dy, I, dx);"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_planted_mistake_is_caught(name):
    find, repl = MUTANTS[name]
    src = open(obuild.SRC).read()
    assert src.count(find) == 1, "mutation anchor not unique: %s" % name
    with tempfile.TemporaryDirectory() as tmp:
        path = os.path.join(tmp, "mutant.c")
        with open(path, "w") as f:
            f.write(src.replace(find, repl))
        lib = obuild.build(src=path, out=os.path.join(tmp, "libmutant.so"))
        o = oracle.Oracle(lib)
        caught = []
        for pin in PINS:
            try:
                pin(o)
            except AssertionError:
                caught.append(pin.__name__)
        assert caught, "no pin caught the planted mistake %s" % name


# Planted mistakes in the Python side of the oracle (the methods that chain the C functions and
# round what crosses the boundary): a copy of one method, changed, on a subclass.
PY_MUTANTS = {
    "step_B_not_rounded": ("boundary_step", "B = self.round_to(B, transfer)", "B = B"),
    "step_dB_not_rounded": ("boundary_step", "dB = self.round_to(dB, transfer)", "dB = dB"),
    "step_decoder_reads_unrounded_B": ("boundary_step", "B = self.round_to(B, transfer)\n",
                                       "Bq = self.round_to(B, transfer)\n"),
    "step_forward_merge_flipped": ("boundary_step", "Y = self.decode_fwd(B, Wd1, Wd2, act, merge)",
                                   "Y = self.decode_fwd(B, Wd1, Wd2, act, 1 - merge)"),
    "step_backward_merge_flipped": ("boundary_step", "dB, dWd1, dWd2 = self.decode_bwd(dY, B, Wd1, Wd2, act, merge)",
                                    "dB, dWd1, dWd2 = self.decode_bwd(dY, B, Wd1, Wd2, act, 1 - merge)"),
    "linear_step_B_not_rounded": ("linear_boundary_step", "B = self.round_to(B, transfer)", "B = B"),
    "linear_step_dB_not_rounded": ("linear_boundary_step", "dB = self.round_to(dB, transfer)", "dB = dB"),
    "linear_step_merge_flipped": ("linear_boundary_step", "Y = self.linear_decode_fwd(B, Wd, merge)",
                                  "Y = self.linear_decode_fwd(B, Wd, 1 - merge)"),
}


@pytest.mark.parametrize("name", sorted(PY_MUTANTS))
def test_planted_mistake_in_python_oracle_is_caught(name):
    import inspect
    import textwrap
    method, find, repl = PY_MUTANTS[name]
    src = textwrap.dedent(inspect.getsource(getattr(oracle.Oracle, method)))
    assert src.count(find) == 1, "mutation anchor not unique: %s" % name
    ns = dict(vars(oracle))
    exec(compile(src.replace(find, repl), "<mutant %s>" % name, "exec"), ns)
    o = type("MutantOracle", (oracle.Oracle,), {method: ns[method]})()
    caught = []
    for pin in PINS:
        try:
            pin(o)
        except AssertionError:
            caught.append(pin.__name__)
    assert caught, "no pin caught the planted mistake %s" % name


def test_transfer_width_mistake_is_caught():
    """fp32 transfer rounding to 23 significant bits instead of 24."""
    o = type("MutantOracle", (oracle.Oracle,), {"_BITS": {"bf16": 8, "f32": 23}})()
    caught = []
    for pin in PINS:
        try:
            pin(o)
        except AssertionError:
            caught.append(pin.__name__)
    assert caught

