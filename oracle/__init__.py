"""fp64 CPU oracle of the ResBM boundary bottleneck -- TEST INFRASTRUCTURE.

Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline / reference leg import this
package. The product path never does; it shares no code with it.

Each function converts its inputs to C-contiguous float64 (exact for bf16 and fp32 values),
calls the plain C implementation in resbm_oracle.c and returns float64 numpy arrays.
Citations (sections and equations of the ResBM paper):
  pid / rect_identity ........ Sec. 3.3, Eq. rect_identity_definition and Eq. Pid_definition
  encode_fwd / decode_fwd .... Sec. 3.2 (two linear layers with a nonlinearity; placement
                               across the boundary; identity path) and
                               Eq. generalized_transformer_equation
  decode_bwd / encode_bwd .... the chain rule of the two forward functions
  effective_rank ............. the appendix's spectral analysis of the bottleneck output
                               projections: r_eff = sum_i sigma_i^2 / max_i sigma_i^2
  ffn_down_encode_fwd ........ Sec. 3.2's bottleneck after the feed-forward layer: the encoder on
                               the FFN's output z = H . W2 (stored in bf16 by the FFN)
  rmsnorm_bwd ................ the chain rule of rmsnorm (for the upstream dN), plus an incoming
                               dY added to the input gradient
  rmsnorm / decode_fwd_rmsnorm  the pre-attention RMSNorm of the block the decoder starts (Sec. 3.2
                               places the decoder at the start of block l+1; Sec. 4.1's model is a
                               pre-norm transformer with RMSNorm): N = Y / sqrt(mean_j Y_j^2 + eps)
                               * gamma over each row, on the decoder's output as stored
  newton_schulz .............. Muon's orthogonalisation of the gradient momentum (Sec. 3.4.2
                               trains the bottleneck weights with Muon): X_0 = G / ||G||_F, then
                               X <- a X + b (X X^T) X + c (X X^T)^2 X on the wide orientation,
                               with the coefficients published with Muon (the paper cites Muon and
                               does not restate them)
"""
import ctypes
import os

import numpy as np

from . import build as _build

ACT_SILU, ACT_GELU_TANH, ACT_IDENTITY = 0, 1, 2
ACTS = {"silu": ACT_SILU, "gelu_tanh": ACT_GELU_TANH, "identity": ACT_IDENTITY}

_lib = None
_dp = ctypes.POINTER(ctypes.c_double)
_i64 = ctypes.c_int64


def _load(path=None):
    lib = ctypes.CDLL(path or _build.build())
    lib.oracle_max_threads.restype = ctypes.c_int
    lib.oracle_set_threads.argtypes = [ctypes.c_int]
    lib.oracle_act.restype = ctypes.c_double
    lib.oracle_act.argtypes = [ctypes.c_int, ctypes.c_double]
    lib.oracle_dact.restype = ctypes.c_double
    lib.oracle_dact.argtypes = [ctypes.c_int, ctypes.c_double]
    lib.oracle_rect_identity.argtypes = [_i64, _i64, _dp]
    lib.oracle_round_array.argtypes = [ctypes.c_int, _i64, _dp]
    lib.oracle_pid.restype = ctypes.c_int
    lib.oracle_pid.argtypes = [_i64, _i64, _i64, _dp, _dp]
    lib.oracle_encode_fwd.restype = ctypes.c_int
    lib.oracle_encode_fwd.argtypes = [_i64] * 4 + [ctypes.c_int] + [_dp] * 6
    lib.oracle_decode_fwd.restype = ctypes.c_int
    lib.oracle_decode_fwd.argtypes = [_i64] * 4 + [ctypes.c_int] * 2 + [_dp] * 4
    lib.oracle_decode_bwd.restype = ctypes.c_int
    lib.oracle_decode_bwd.argtypes = [_i64] * 4 + [ctypes.c_int] * 2 + [_dp] * 7
    lib.oracle_encode_bwd.restype = ctypes.c_int
    lib.oracle_encode_bwd.argtypes = [_i64] * 4 + [ctypes.c_int] + [_dp] * 8
    lib.oracle_linear_encode_fwd.restype = ctypes.c_int
    lib.oracle_linear_encode_fwd.argtypes = [_i64] * 3 + [_dp] * 4
    lib.oracle_linear_decode_fwd.restype = ctypes.c_int
    lib.oracle_linear_decode_fwd.argtypes = [_i64] * 3 + [ctypes.c_int] + [_dp] * 3
    lib.oracle_linear_decode_bwd.restype = ctypes.c_int
    lib.oracle_linear_decode_bwd.argtypes = [_i64] * 3 + [ctypes.c_int] + [_dp] * 5
    lib.oracle_linear_encode_bwd.restype = ctypes.c_int
    lib.oracle_linear_encode_bwd.argtypes = [_i64] * 3 + [_dp] * 6
    return lib


def lib():
    global _lib
    if _lib is None:
        _lib = _load()
    return _lib


class Oracle:
    """The oracle bound to one compiled library (the default one, or a test variant)."""

    def __init__(self, path=None):
        self._l = _load(path) if path else lib()

    # -- helpers ---------------------------------------------------------------------------
    @staticmethod
    def _in(a, shape):
        a = np.ascontiguousarray(np.asarray(a, dtype=np.float64))
        if a.shape != tuple(shape):
            raise ValueError("expected shape %s, got %s" % (tuple(shape), a.shape))
        return a

    @staticmethod
    def _p(a):
        return None if a is None else a.ctypes.data_as(_dp)

    @staticmethod
    def _act(act):
        return ACTS[act] if isinstance(act, str) else int(act)

    def max_threads(self):
        return int(self._l.oracle_max_threads())

    def set_threads(self, n):
        """OpenMP threads of later calls (the results do not depend on it)."""
        self._l.oracle_set_threads(int(n))

    # -- transfer rounding (Appendix A.3: the boundary tensors travel in bf16) ----------------
    _BITS = {"bf16": 8, "f32": 24}

    def round_to(self, x, dtype):
        """x rounded to the transfer dtype ("bf16" or "f32"), nearest-even, from fp64."""
        y = np.array(x, dtype=np.float64, copy=True, order="C")
        self._l.oracle_round_array(self._BITS[dtype], y.size, self._p(y))
        return y

    # -- Sec. 3.3 ---------------------------------------------------------------------------
    def act(self, act, x):
        return self._l.oracle_act(self._act(act), float(x))

    def dact(self, act, x):
        return self._l.oracle_dact(self._act(act), float(x))

    def rect_identity(self, c, C):
        out = np.empty((c, C), np.float64)
        self._l.oracle_rect_identity(c, C, self._p(out))
        return out

    def pid(self, x, C):
        x = np.ascontiguousarray(np.asarray(x, dtype=np.float64))
        L, c = x.shape
        y = np.empty((L, C), np.float64)
        if self._l.oracle_pid(L, c, C, self._p(x), self._p(y)) != 0:
            raise MemoryError("oracle_pid")
        return y

    # -- Sec. 3.2 forward -------------------------------------------------------------------
    def encode_fwd(self, X, F, We1, We2, act="silu"):
        """Returns (B, P): B = X . I_{d x r} + phi(F . We1) . We2, P = F . We1."""
        F = np.asarray(F)
        T, d = F.shape
        m, r = np.asarray(We2).shape
        X = self._in(X, (T, d)); F = self._in(F, (T, d))
        We1 = self._in(We1, (d, m)); We2 = self._in(We2, (m, r))
        B = np.empty((T, r)); P = np.empty((T, m))
        rc = self._l.oracle_encode_fwd(T, d, r, m, self._act(act), self._p(X), self._p(F),
                                       self._p(We1), self._p(We2), self._p(B), self._p(P))
        if rc != 0:
            raise MemoryError("oracle_encode_fwd")
        return B, P

    def decode_fwd(self, B, Wd1, Wd2, act="silu", merge=1):
        """Returns Y = [merge] B . I_{r x d} + phi(B . Wd1) . Wd2."""
        B = np.asarray(B)
        T, r = B.shape
        m, d = np.asarray(Wd2).shape
        B = self._in(B, (T, r)); Wd1 = self._in(Wd1, (r, m)); Wd2 = self._in(Wd2, (m, d))
        Y = np.empty((T, d))
        rc = self._l.oracle_decode_fwd(T, d, r, m, self._act(act), int(merge), self._p(B),
                                       self._p(Wd1), self._p(Wd2), self._p(Y))
        if rc != 0:
            raise MemoryError("oracle_decode_fwd")
        return Y

    # -- chain rule -------------------------------------------------------------------------
    def decode_bwd(self, dY, B, Wd1, Wd2, act="silu", merge=1):
        """Returns (dB, dWd1, dWd2) for the upstream gradient dY of decode_fwd's Y."""
        B = np.asarray(B)
        T, r = B.shape
        m, d = np.asarray(Wd2).shape
        dY = self._in(dY, (T, d)); B = self._in(B, (T, r))
        Wd1 = self._in(Wd1, (r, m)); Wd2 = self._in(Wd2, (m, d))
        dB = np.empty((T, r)); dWd1 = np.empty((r, m)); dWd2 = np.empty((m, d))
        rc = self._l.oracle_decode_bwd(T, d, r, m, self._act(act), int(merge), self._p(dY),
                                       self._p(B), self._p(Wd1), self._p(Wd2), self._p(dB),
                                       self._p(dWd1), self._p(dWd2))
        if rc != 0:
            raise MemoryError("oracle_decode_bwd")
        return dB, dWd1, dWd2

    def encode_bwd(self, dB, F, We1, We2, act="silu", want_dX=True):
        """Returns (dF, dX, dWe1, dWe2) for the upstream gradient dB of encode_fwd's B.

        dX is the full T x d gradient of X (dB in the first r columns, zeros after) or None.
        """
        F = np.asarray(F)
        T, d = F.shape
        m, r = np.asarray(We2).shape
        dB = self._in(dB, (T, r)); F = self._in(F, (T, d))
        We1 = self._in(We1, (d, m)); We2 = self._in(We2, (m, r))
        dF = np.empty((T, d)); dX = np.empty((T, d)) if want_dX else None
        dWe1 = np.empty((d, m)); dWe2 = np.empty((m, r))
        rc = self._l.oracle_encode_bwd(T, d, r, m, self._act(act), self._p(dB), self._p(F),
                                       self._p(We1), self._p(We2), self._p(dF), self._p(dX),
                                       self._p(dWe1), self._p(dWe2))
        if rc != 0:
            raise MemoryError("oracle_encode_bwd")
        return dF, dX, dWe1, dWe2

    # -- one linear layer per side (no nonlinearity) ------------------------------------------
    def linear_encode_fwd(self, X, F, We):
        """Returns B = X . I_{d x r} + F . We (We: d x r)."""
        F = np.asarray(F)
        T, d = F.shape
        r = np.asarray(We).shape[1]
        X = self._in(X, (T, d)); F = self._in(F, (T, d)); We = self._in(We, (d, r))
        B = np.empty((T, r))
        if self._l.oracle_linear_encode_fwd(T, d, r, self._p(X), self._p(F), self._p(We), self._p(B)) != 0:
            raise MemoryError("oracle_linear_encode_fwd")
        return B

    def linear_decode_fwd(self, B, Wd, merge=1):
        """Returns Y = [merge] B . I_{r x d} + B . Wd (Wd: r x d)."""
        B = np.asarray(B)
        T, r = B.shape
        d = np.asarray(Wd).shape[1]
        B = self._in(B, (T, r)); Wd = self._in(Wd, (r, d))
        Y = np.empty((T, d))
        if self._l.oracle_linear_decode_fwd(T, d, r, int(merge), self._p(B), self._p(Wd), self._p(Y)) != 0:
            raise MemoryError("oracle_linear_decode_fwd")
        return Y

    def linear_decode_bwd(self, dY, B, Wd, merge=1):
        """Returns (dB, dWd) for the upstream gradient dY of linear_decode_fwd's Y."""
        B = np.asarray(B)
        T, r = B.shape
        d = np.asarray(Wd).shape[1]
        dY = self._in(dY, (T, d)); B = self._in(B, (T, r)); Wd = self._in(Wd, (r, d))
        dB = np.empty((T, r)); dWd = np.empty((r, d))
        if self._l.oracle_linear_decode_bwd(T, d, r, int(merge), self._p(dY), self._p(B), self._p(Wd),
                                            self._p(dB), self._p(dWd)) != 0:
            raise MemoryError("oracle_linear_decode_bwd")
        return dB, dWd

    def linear_encode_bwd(self, dB, F, We, want_dX=True):
        """Returns (dF, dX, dWe) for the upstream gradient dB of linear_encode_fwd's B."""
        F = np.asarray(F)
        T, d = F.shape
        r = np.asarray(We).shape[1]
        dB = self._in(dB, (T, r)); F = self._in(F, (T, d)); We = self._in(We, (d, r))
        dF = np.empty((T, d)); dX = np.empty((T, d)) if want_dX else None; dWe = np.empty((d, r))
        if self._l.oracle_linear_encode_bwd(T, d, r, self._p(dB), self._p(F), self._p(We), self._p(dF),
                                            self._p(dX), self._p(dWe)) != 0:
            raise MemoryError("oracle_linear_encode_bwd")
        return dF, dX, dWe

    def linear_boundary_step(self, X, F, dY, We, Wd, merge=1, transfer=None):
        """The one-linear-layer boundary forward + backward, chained like boundary_step."""
        B = self.linear_encode_fwd(X, F, We)
        if transfer:
            B = self.round_to(B, transfer)
        Y = self.linear_decode_fwd(B, Wd, merge)
        dB, dWd = self.linear_decode_bwd(dY, B, Wd, merge)
        if transfer:
            dB = self.round_to(dB, transfer)
        dF, dX, dWe = self.linear_encode_bwd(dB, F, We)
        return dict(B=B, Y=Y, dB=dB, dF=dF, dX=dX, dWe1=dWe, dWd2=dWd)

    def boundary_step(self, X, F, dY, We1, We2, Wd1, Wd2, act="silu", merge=1, transfer=None):
        """One boundary forward + backward: the four functions above chained. B is handed to
        the decoder and dB back to the encoder; with transfer = "bf16" / "f32" they are first
        rounded to that dtype, as they are when sent across the boundary (Appendix A.3). The
        returned B and dB are the values that crossed."""
        B, P = self.encode_fwd(X, F, We1, We2, act)
        if transfer:
            B = self.round_to(B, transfer)
        Y = self.decode_fwd(B, Wd1, Wd2, act, merge)
        dB, dWd1, dWd2 = self.decode_bwd(dY, B, Wd1, Wd2, act, merge)
        if transfer:
            dB = self.round_to(dB, transfer)
        dF, dX, dWe1, dWe2 = self.encode_bwd(dB, F, We1, We2, act)
        return dict(B=B, P=P, Y=Y, dB=dB, dF=dF, dX=dX, dWe1=dWe1, dWe2=dWe2,
                    dWd1=dWd1, dWd2=dWd2)


def effective_rank(W):
    """r_eff of a matrix as the appendix's spectral analysis defines it: the sum of its squared
    singular values over the largest squared singular value (1 when one singular value
    dominates, the smaller dimension when all are equal; 0 for the zero matrix). Singular
    values from numpy's SVD in float64."""
    W = np.asarray(W, dtype=np.float64)
    if W.ndim != 2:
        raise ValueError("effective_rank takes a matrix")
    if W.size == 0:
        return 0.0
    sig = np.linalg.svd(W, compute_uv=False)
    top = float(np.max(sig)) ** 2
    return 0.0 if top == 0.0 else float(np.sum(sig * sig)) / top


_default = None


def default():
    global _default
    if _default is None:
        _default = Oracle()
    return _default


def __getattr__(name):
    # module-level shortcuts: oracle.encode_fwd(...) etc.
    if name in ("act", "dact", "rect_identity", "pid", "encode_fwd", "decode_fwd", "round_to",
                "decode_bwd", "encode_bwd", "boundary_step", "max_threads", "set_threads", "linear_encode_fwd",
                "linear_decode_fwd", "linear_decode_bwd", "linear_encode_bwd",
                "linear_boundary_step"):
        return getattr(default(), name)
    raise AttributeError(name)


NS_COEFFS = (3.4445, -4.7750, 2.0315)   # Muon's quintic Newton-Schulz coefficients (a, b, c)


def newton_schulz(G, steps=5, coeffs=NS_COEFFS, eps=1e-7):
    """Muon's Newton-Schulz orthogonalisation in float64, step by step as the iteration is
    stated: X_0 = G / (||G||_F + eps); for a matrix with more rows than columns the iteration runs
    on its transpose; each step A = X X^T, B = b A + c A A, X <- a X + B X. numpy's matmul is the
    library step for every product."""
    G = np.asarray(G, dtype=np.float64)
    if G.ndim != 2:
        raise ValueError("newton_schulz takes a matrix")
    a, b, c = coeffs
    X = G / (np.linalg.norm(G) + eps)
    tall = X.shape[0] > X.shape[1]
    if tall:
        X = X.T
    for _ in range(steps):
        A = X @ X.T
        B = b * A + c * (A @ A)
        X = a * X + B @ X
    return X.T if tall else X


def ffn_down_encode_fwd(H, W2, X, We1, We2, act="silu"):
    """The encoder applied after the feed-forward layer (Sec. 3.2: the bottleneck follows the FFN;
    its input z is the FFN's output): F = H . W2 (numpy's matmul, float64) rounded to bf16 as the
    FFN's output tensor, then (B, P) = encode_fwd(X, F, We1, We2). Returns (B, P, F)."""
    F = default().round_to(np.asarray(H, np.float64) @ np.asarray(W2, np.float64), "bf16")
    B, P = default().encode_fwd(X, F, We1, We2, act)
    return B, P, F


def rmsnorm(Y, gamma, eps):
    """RMSNorm of every row of Y in float64: the row's root mean square over its d columns,
    with eps added under the square root, divides the row, and gamma (d) scales each column:
    N[t, j] = Y[t, j] / sqrt(mean_j Y[t, j]^2 + eps) * gamma[j]."""
    Y = np.asarray(Y, dtype=np.float64)
    gamma = np.asarray(gamma, dtype=np.float64)
    if Y.ndim != 2 or gamma.shape != (Y.shape[1],):
        raise ValueError("rmsnorm takes a T x d matrix and d weights")
    mean_sq = np.mean(Y * Y, axis=1, keepdims=True)
    return Y / np.sqrt(mean_sq + eps) * gamma[None, :]


def decode_fwd_rmsnorm(B, Wd1, Wd2, gamma, eps, act="silu", merge=1, store=None):
    """The decoder forward and the next block's pre-attention RMSNorm: Y = decode_fwd(B, Wd1, Wd2),
    then N = rmsnorm(Y as stored, gamma, eps). store = "bf16" / "f32" rounds Y to that dtype first
    (the residual stream is a tensor of that dtype, and the norm reads it); None keeps it exact.
    Returns (Y, N) with Y unrounded."""
    Y = default().decode_fwd(B, Wd1, Wd2, act, merge)
    Ys = default().round_to(Y, store) if store else Y
    return Y, rmsnorm(Ys, gamma, eps)


def rmsnorm_bwd(Y, gamma, eps, dN, dY=None):
    """Gradients of N = rmsnorm(Y, gamma, eps) for the upstream dN, in float64, by the chain rule
    of its three steps (s = 1 / sqrt(mean_j Y_j^2 + eps), xhat = Y s, N = xhat gamma):
      dxhat = dN gamma
      ds    = sum_j dxhat_j Y_j                    (per row)
      dY_j  = dxhat_j s + ds * (-s^3 / d) Y_j       (d s / d Y_j = -s^3 Y_j / d)
      dgamma = sum over rows of dN xhat.
    An incoming dY (the residual stream's own gradient) is added to the input gradient.
    Returns (dY_total, dgamma)."""
    Y = np.asarray(Y, dtype=np.float64)
    gamma = np.asarray(gamma, dtype=np.float64)
    dN = np.asarray(dN, dtype=np.float64)
    d = Y.shape[1]
    s = 1.0 / np.sqrt(np.mean(Y * Y, axis=1, keepdims=True) + eps)
    xhat = Y * s
    dxhat = dN * gamma[None, :]
    ds = np.sum(dxhat * Y, axis=1, keepdims=True)
    dY_norm = dxhat * s + ds * (-(s ** 3) / d) * Y
    dgamma = np.sum(dN * xhat, axis=0)
    if dY is not None:
        dY_norm = dY_norm + np.asarray(dY, dtype=np.float64)
    return dY_norm, dgamma
