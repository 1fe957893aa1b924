"""Error metrics of the GPU-vs-oracle parity tests.

fp32 I/O:  max over elements of |g - o| / max(|o|, rms(o))            <= 1e-5
bf16 I/O:  max over elements of |g - o| / max(|o|, rms(o[row]))       <= 2e-2
           where row is the element's token row for the per-token outputs (B, Y, dB, dF, dX)
           and the whole tensor for the weight gradients (sums over all tokens).
The rms floor keeps near-zero elements from dominating; for bf16 the floor is taken per token
because the synthetic residual stream spreads token norms log-normally, and a once-rounded
bf16 output of a large-norm token is off by up to 2^-8 of its own size.
"""
import numpy as np

TOL = {"f32": 1e-5, "bf16": 2e-2}
ROWWISE = {"B", "Y", "dB", "dF", "dX"}


def rel_err(g, o, dtype, rowwise):
    g = np.asarray(g, np.float64)
    o = np.asarray(o, np.float64)
    assert g.shape == o.shape, (g.shape, o.shape)
    if o.size == 0:
        return 0.0
    diff = np.abs(g - o)
    if dtype == "bf16" and rowwise and o.ndim == 2:
        floor = np.sqrt(np.mean(o * o, axis=1, keepdims=True))
    else:
        floor = np.sqrt(np.mean(o * o))
    den = np.maximum(np.abs(o), floor)
    with np.errstate(invalid="ignore", divide="ignore"):
        r = np.where(den > 0, diff / np.where(den > 0, den, 1), diff)
    return float(np.max(r))


def check(name, g, o, dtype, tol=None):
    e = rel_err(g, o, dtype, name in ROWWISE)
    t = TOL[dtype] if tol is None else tol
    assert e <= t, "%s: relative error %.3e > %.1e" % (name, e, t)
    return e
