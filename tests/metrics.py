"""Error metrics of the GPU-vs-oracle parity tests.

fp32 I/O:  max over elements of |g - o| / max(|o|, rms(o))                         <= 1e-5
bf16 I/O:  per-token outputs (B, Y, dB, dF, dX; bf16 tensors):
             max over elements of max(0, |g - o| - h(g, o)) / rms(o[row])           <= 2e-2
           weight gradients (fp32 tensors, sums over all tokens):
             max over elements of |g - o| / rms(o)                                  <= 2e-2
           where row is the element's token row and h(g, o) = half the bf16 spacing at
           max(|g|, |o|). Only a bf16 output gets h: the weight gradients are fp32 and are not
           rounded to bf16.
The bf16 bound is the error of the computation normalised by the output's RMS. A bf16 output
cannot be closer to the exact (fp64) value than its own final rounding, half a bf16 spacing,
2^-9 of the element's magnitude: h excludes exactly that and nothing else. (It is not a
tolerance proportional to |o|: an element several times its row's RMS is held to the same
absolute bound 2e-2 * rms(row) on the error before its rounding as every other element. Without
h, a correctly rounded element more than ~10x its row's RMS fails by construction: in Y the
first r columns carry the token-scaled identity path, the other d - r columns only D(B), so
such rows occur.) The RMS is taken per token row because the synthetic residual stream spreads
token norms log-normally (a factor exp(0.5 n), n ~ N(0,1)).
An output computed from another rounded output (N = RMSNorm(Y) * gamma reads the stored bf16 Y)
passes `allow`: per element, the earlier rounding carried into it (half Y's spacing times
|rstd * gamma|), excluded on top of its own h.
"""
import numpy as np

TOL = {"f32": 1e-5, "bf16": 2e-2}
ROWWISE = {"B", "Y", "dB", "dF", "dX", "F", "N", "dY_out"}


def bf16_half_spacing(x):
    """Half the distance between consecutive bf16 values (8 significant bits) at |x|: 2^(e - 8)
    for |x| in [2^e, 2^(e+1)); 0 at 0."""
    a = np.abs(np.asarray(x, np.float64))
    out = np.zeros_like(a)
    nz = a > 0
    out[nz] = np.exp2(np.floor(np.log2(a[nz])) - 8.0)
    return out


def _errors(g, o, dtype, rowwise, allow=None):
    g = np.asarray(g, np.float64)
    o = np.asarray(o, np.float64)
    assert g.shape == o.shape, (g.shape, o.shape)
    diff = np.abs(g - o)
    if allow is not None:
        diff = np.maximum(diff - np.asarray(allow, np.float64), 0.0)
    if dtype == "bf16":
        if rowwise:   # a bf16 output: its own rounding is not charged
            diff = np.maximum(diff - bf16_half_spacing(np.maximum(np.abs(g), np.abs(o))), 0.0)
        if rowwise and o.ndim == 2:
            den = np.sqrt(np.mean(o * o, axis=1, keepdims=True))
        else:
            den = np.sqrt(np.mean(o * o))
        den = np.broadcast_to(den, o.shape)
    else:
        den = np.maximum(np.abs(o), np.sqrt(np.mean(o * o)))
    with np.errstate(invalid="ignore", divide="ignore"):
        return np.where(den > 0, diff / np.where(den > 0, den, 1), diff)


def rel_err(g, o, dtype, rowwise, allow=None):
    if np.asarray(o).size == 0:
        return 0.0
    return float(np.max(_errors(g, o, dtype, rowwise, allow)))


def worst(g, o, dtype, rowwise, allow=None):
    """(error, index) of the worst element under rel_err's metric (for failure messages)."""
    r = _errors(g, o, dtype, rowwise, allow)
    i = np.unravel_index(int(np.argmax(r)), r.shape)
    return float(r[i]), tuple(int(x) for x in i)


def check(name, g, o, dtype, tol=None, allow=None):
    rowwise = name in ROWWISE
    e = rel_err(g, o, dtype, rowwise, allow)
    t = TOL[dtype] if tol is None else tol
    if e > t:
        _, i = worst(g, o, dtype, rowwise, allow)
        o = np.asarray(o, np.float64)
        den = (np.sqrt(np.mean(o[i[0]] ** 2)) if rowwise and o.ndim == 2 else np.sqrt(np.mean(o ** 2)))
        raise AssertionError("%s: error %.3e > %.1e at %s (got %r, want %r, rms %.4g)"
                             % (name, e, t, i, float(np.asarray(g)[i]), float(o[i]), den))
    return e
