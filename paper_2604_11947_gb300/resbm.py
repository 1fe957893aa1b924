"""Python binding of the C ABI in include/resbm.h (libresbm.so).

Argument marshalling only: every function here has the C function's name, takes torch tensors
(device memory owned by the caller) or None, passes their data pointers and the current CUDA
stream, and raises ResbmError when the C call returns a status other than RESBM_OK. No compute
happens in Python, and there is no fallback: if libresbm.so cannot be loaded, every call raises.
"""
from __future__ import annotations

import ctypes
import os

import torch

from . import build as _build

RESBM_OK, RESBM_ERR_INVALID_ARG, RESBM_ERR_UNSUPPORTED, RESBM_ERR_WORKSPACE, RESBM_ERR_CUDA = range(5)
RESBM_F32, RESBM_BF16 = 0, 1
RESBM_ACT_SILU, RESBM_ACT_GELU_TANH, RESBM_ACT_IDENTITY = 0, 1, 2
(RESBM_OP_ENCODE_FWD, RESBM_OP_DECODE_FWD, RESBM_OP_DECODE_BWD, RESBM_OP_ENCODE_BWD,
 RESBM_OP_BOUNDARY_STEP, RESBM_OP_BOUNDARY_STEP_HOST, RESBM_OP_EFFECTIVE_RANK, RESBM_OP_NEWTON_SCHULZ,
 RESBM_OP_DECODE_FWD_RMSNORM, RESBM_OP_RMSNORM_BWD) = range(10)
(RESBM_HBM_READ_V4, RESBM_HBM_WRITE_V4, RESBM_HBM_COPY_V4, RESBM_HBM_READ_TMA_2D, RESBM_HBM_READ_TMA_2D_PAIR,
 RESBM_HBM_READ_TMA_3D, RESBM_HBM_READ_BULK, RESBM_HBM_WRITE_TMA_2D, RESBM_HBM_WRITE_BULK,
 RESBM_HBM_READ_TMA_2D_TILES, RESBM_HBM_WRITE_TMA_2D_TILES) = range(11)
HBM_FORMS = {"read_v4": RESBM_HBM_READ_V4, "write_v4": RESBM_HBM_WRITE_V4, "copy_v4": RESBM_HBM_COPY_V4,
             "read_tma_2d": RESBM_HBM_READ_TMA_2D, "read_tma_2d_pair": RESBM_HBM_READ_TMA_2D_PAIR,
             "read_tma_3d": RESBM_HBM_READ_TMA_3D, "read_bulk": RESBM_HBM_READ_BULK,
             "write_tma_2d": RESBM_HBM_WRITE_TMA_2D, "write_bulk": RESBM_HBM_WRITE_BULK,
             "read_tma_2d_tiles": RESBM_HBM_READ_TMA_2D_TILES, "write_tma_2d_tiles": RESBM_HBM_WRITE_TMA_2D_TILES}
RESBM_FLAG_GENERIC = 1
RESBM_FLAG_LINEAR = 2
RESBM_FLAG_GEMM = 4
RESBM_STATIC_SCRATCH_BYTES = 32 << 20

ACTS = {"silu": RESBM_ACT_SILU, "gelu_tanh": RESBM_ACT_GELU_TANH, "identity": RESBM_ACT_IDENTITY}
DTYPES = {"f32": RESBM_F32, "bf16": RESBM_BF16}
TORCH_DTYPES = {RESBM_F32: torch.float32, RESBM_BF16: torch.bfloat16}

EXPORTS = ("resbm_version", "resbm_status_string", "resbm_last_cuda_error", "resbm_kernel_launches",
           "resbm_device_error",
           "resbm_workspace_bytes", "resbm_encode_fwd", "resbm_decode_fwd", "resbm_decode_bwd",
           "resbm_encode_bwd", "resbm_boundary_step", "resbm_boundary_step_host",
           "resbm_decode_bwd_noalloc", "resbm_selftest_wait_timeout", "resbm_matrix_workspace_bytes",
           "resbm_newton_schulz", "resbm_effective_rank", "resbm_ffn_down_encode_workspace_bytes",
           "resbm_ffn_down_encode_fwd", "resbm_decode_fwd_rmsnorm", "resbm_rmsnorm_bwd",
           "resbm_measure_hbm_form")


class resbm_desc(ctypes.Structure):
    _fields_ = [("T", ctypes.c_int64), ("d", ctypes.c_int64), ("r", ctypes.c_int64),
                ("m", ctypes.c_int64), ("dtype", ctypes.c_int32), ("act", ctypes.c_int32),
                ("merge_identity", ctypes.c_int32), ("flags", ctypes.c_uint32)]


class resbm_step_args(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in
                ("X", "F", "dY", "We1", "We2", "Wd1", "Wd2", "B", "P", "Y", "dB", "dF", "dX",
                 "dWe1", "dWe2", "dWd1", "dWd2", "wait_before_inputs", "inputs_done")]


class ResbmError(RuntimeError):
    def __init__(self, fn, status, cuda_error=0):
        self.status, self.cuda_error = status, cuda_error
        msg = "%s failed: %s" % (fn, status_string(status))
        if status == RESBM_ERR_CUDA:
            msg += " (cudaError %d)" % cuda_error
        super().__init__(msg)


_lib = None


def library_path() -> str:
    return _build.LIB


def load(path: str | None = None) -> ctypes.CDLL:
    """Load libresbm.so (built in-tree by build.build()); raise if it is missing."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = path or _build.LIB
    if not os.path.exists(p):
        raise RuntimeError("libresbm.so not found at %s: run paper_2604_11947_gb300.build.build() "
                           "(there is no CPU fallback)" % p)
    lib = ctypes.CDLL(p)
    vp, sz, i32 = ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int
    D = ctypes.POINTER(resbm_desc)
    lib.resbm_version.restype = ctypes.c_char_p
    lib.resbm_status_string.restype = ctypes.c_char_p
    lib.resbm_status_string.argtypes = [i32]
    lib.resbm_last_cuda_error.restype = i32
    lib.resbm_kernel_launches.restype = ctypes.c_uint64
    lib.resbm_device_error.restype = i32
    lib.resbm_device_error.argtypes = [ctypes.POINTER(ctypes.c_uint), i32]
    lib.resbm_workspace_bytes.restype = i32
    lib.resbm_workspace_bytes.argtypes = [D, i32, ctypes.POINTER(sz)]
    lib.resbm_encode_fwd.restype = i32
    lib.resbm_encode_fwd.argtypes = [D] + [vp] * 6 + [vp, sz, vp]
    lib.resbm_decode_fwd.restype = i32
    lib.resbm_decode_fwd.argtypes = [D] + [vp] * 4 + [vp, sz, vp]
    lib.resbm_rmsnorm_bwd.restype = i32
    lib.resbm_rmsnorm_bwd.argtypes = [D, vp, vp, ctypes.c_float] + [vp] * 4 + [vp, sz, vp]
    lib.resbm_decode_fwd_rmsnorm.restype = i32
    lib.resbm_decode_fwd_rmsnorm.argtypes = [D] + [vp] * 4 + [ctypes.c_float] + [vp] * 2 + [vp, sz, vp]
    lib.resbm_decode_bwd.restype = i32
    lib.resbm_decode_bwd.argtypes = [D] + [vp] * 7 + [vp, sz, vp]
    lib.resbm_encode_bwd.restype = i32
    lib.resbm_encode_bwd.argtypes = [D] + [vp] * 9 + [vp, sz, vp]
    lib.resbm_boundary_step.restype = i32
    lib.resbm_selftest_wait_timeout.restype = i32
    lib.resbm_selftest_wait_timeout.argtypes = [vp]
    lib.resbm_decode_bwd_noalloc.restype = i32
    lib.resbm_decode_bwd_noalloc.argtypes = [D] + [vp] * 7 + [vp]
    lib.resbm_boundary_step.argtypes = [D, ctypes.POINTER(resbm_step_args), vp, sz, vp]
    lib.resbm_boundary_step_host.restype = i32
    lib.resbm_boundary_step_host.argtypes = [D, ctypes.POINTER(resbm_step_args), vp, sz, vp]
    i64 = ctypes.c_int64
    lib.resbm_matrix_workspace_bytes.restype = i32
    lib.resbm_matrix_workspace_bytes.argtypes = [i32, i64, i64, ctypes.POINTER(sz)]
    lib.resbm_newton_schulz.restype = i32
    lib.resbm_newton_schulz.argtypes = [i64, i64, vp, ctypes.c_int32, ctypes.c_int32, vp, vp, sz, vp]
    lib.resbm_effective_rank.restype = i32
    lib.resbm_effective_rank.argtypes = [i64, i64, vp, vp, vp, sz, vp]
    lib.resbm_ffn_down_encode_workspace_bytes.restype = i32
    lib.resbm_ffn_down_encode_workspace_bytes.argtypes = [D, i64, ctypes.POINTER(sz)]
    lib.resbm_ffn_down_encode_fwd.restype = i32
    lib.resbm_ffn_down_encode_fwd.argtypes = [D, i64] + [vp] * 8 + [vp, sz, vp]
    lib.resbm_measure_hbm_form.restype = i32
    lib.resbm_measure_hbm_form.argtypes = [i32, vp, vp, i64, vp]
    if path is None:
        _lib = lib
    return lib


def status_string(status: int) -> str:
    return load().resbm_status_string(int(status)).decode()


def resbm_version() -> str:
    return load().resbm_version().decode()


def resbm_kernel_launches() -> int:
    return int(load().resbm_kernel_launches())


def resbm_device_error(clear=False) -> int:
    """The tensor-core kernels' error word (synchronizes with the device)."""
    out = ctypes.c_uint(0)
    _check("resbm_device_error", load().resbm_device_error(ctypes.byref(out), int(bool(clear))))
    return int(out.value)


def resbm_selftest_wait_timeout(stream=None):
    """Enqueue the failure-path self-test kernel (a wait that gives up after ~2 s)."""
    _check("resbm_selftest_wait_timeout", load().resbm_selftest_wait_timeout(_stream(stream)))


def resbm_measure_hbm_form(form, a, b, stream=None):
    """One launch of an HBM access-form probe (resbm_hbm_form; a name of HBM_FORMS or its value)
    over a's bytes: a read, b written; both device tensors of the same byte size."""
    f = HBM_FORMS[form] if isinstance(form, str) else int(form)
    n = _nbytes(a)
    if _nbytes(b) != n:
        raise ValueError("a and b must have the same byte size")
    _check("resbm_measure_hbm_form", load().resbm_measure_hbm_form(f, _p(a), _p(b), n, _stream(stream)))


def make_desc(T, d, r, m, dtype="bf16", act="silu", merge_identity=1, flags=0) -> resbm_desc:
    dt = DTYPES[dtype] if isinstance(dtype, str) else int(dtype)
    a = ACTS[act] if isinstance(act, str) else int(act)
    return resbm_desc(int(T), int(d), int(r), int(m), dt, a, int(merge_identity), int(flags))


def desc_from_config(cfg, flags=0) -> resbm_desc:
    return make_desc(cfg.T, cfg.d, cfg.r, cfg.m, cfg.dtype, cfg.act, cfg.merge, flags)


def resbm_workspace_bytes(desc: resbm_desc, op: int) -> int:
    out = ctypes.c_size_t(0)
    st = load().resbm_workspace_bytes(ctypes.byref(desc), int(op), ctypes.byref(out))
    if st != RESBM_OK:
        raise ResbmError("resbm_workspace_bytes", st)
    return int(out.value)


def workspace(desc: resbm_desc, op: int, device="cuda") -> torch.Tensor:
    """A torch-owned scratch buffer of the size the C ABI asks for (allocated by torch)."""
    n = resbm_workspace_bytes(desc, op)
    return torch.empty(max(n, 1), dtype=torch.uint8, device=device)


def _p(t):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _nbytes(t):
    return 0 if t is None else t.numel() * t.element_size()


def _stream(stream):
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    return stream if isinstance(stream, int) else stream.cuda_stream


def _check(fn, st):
    if st != RESBM_OK:
        raise ResbmError(fn, st, load().resbm_last_cuda_error() if st == RESBM_ERR_CUDA else 0)


def resbm_encode_fwd(desc, X, F, We1, We2, B, P_save, ws, stream=None):
    st = load().resbm_encode_fwd(ctypes.byref(desc), _p(X), _p(F), _p(We1), _p(We2), _p(B),
                                 _p(P_save), _p(ws), _nbytes(ws), _stream(stream))
    _check("resbm_encode_fwd", st)


def resbm_decode_fwd(desc, B, Wd1, Wd2, Y, ws, stream=None):
    st = load().resbm_decode_fwd(ctypes.byref(desc), _p(B), _p(Wd1), _p(Wd2), _p(Y), _p(ws),
                                 _nbytes(ws), _stream(stream))
    _check("resbm_decode_fwd", st)


def resbm_decode_fwd_rmsnorm(desc, B, Wd1, Wd2, gamma, eps, Y, N, ws, stream=None):
    st = load().resbm_decode_fwd_rmsnorm(ctypes.byref(desc), _p(B), _p(Wd1), _p(Wd2), _p(gamma), float(eps),
                                         _p(Y), _p(N), _p(ws), _nbytes(ws), _stream(stream))
    _check("resbm_decode_fwd_rmsnorm", st)


def resbm_rmsnorm_bwd(desc, Y, gamma, eps, dN, dY, dY_out, dgamma, ws, stream=None):
    st = load().resbm_rmsnorm_bwd(ctypes.byref(desc), _p(Y), _p(gamma), float(eps), _p(dN), _p(dY), _p(dY_out),
                                  _p(dgamma), _p(ws), _nbytes(ws), _stream(stream))
    _check("resbm_rmsnorm_bwd", st)


def resbm_decode_bwd(desc, dY, B, Wd1, Wd2, dB, dWd1, dWd2, ws, stream=None):
    st = load().resbm_decode_bwd(ctypes.byref(desc), _p(dY), _p(B), _p(Wd1), _p(Wd2), _p(dB),
                                 _p(dWd1), _p(dWd2), _p(ws), _nbytes(ws), _stream(stream))
    _check("resbm_decode_bwd", st)


def resbm_decode_bwd_noalloc(desc, dY, B, Wd1, Wd2, dB, dWd1, dWd2, stream=None):
    """resbm_decode_bwd with the library's fixed device scratch instead of a workspace."""
    st = load().resbm_decode_bwd_noalloc(ctypes.byref(desc), _p(dY), _p(B), _p(Wd1), _p(Wd2),
                                         _p(dB), _p(dWd1), _p(dWd2), _stream(stream))
    _check("resbm_decode_bwd_noalloc", st)


def resbm_encode_bwd(desc, dB, F, P_save, We1, We2, dF, dX, dWe1, dWe2, ws, stream=None):
    st = load().resbm_encode_bwd(ctypes.byref(desc), _p(dB), _p(F), _p(P_save), _p(We1),
                                 _p(We2), _p(dF), _p(dX), _p(dWe1), _p(dWe2), _p(ws),
                                 _nbytes(ws), _stream(stream))
    _check("resbm_encode_bwd", st)


def resbm_boundary_step(desc, ws, stream=None, **tensors):
    """tensors: X, F, dY, We1, We2, Wd1, Wd2 (inputs); B, P, Y, dB, dF, dX, dWe1, dWe2, dWd1,
    dWd2 (outputs; P and dX may be omitted)."""
    args = resbm_step_args(**{k: _p(v) for k, v in tensors.items()})
    st = load().resbm_boundary_step(ctypes.byref(desc), ctypes.byref(args), _p(ws), _nbytes(ws),
                                    _stream(stream))
    _check("resbm_boundary_step", st)


def _event(ev):
    """The cudaEvent_t handle of a torch.cuda.Event (recorded once already, so that it exists)."""
    if ev is None:
        return None
    h = ev.cuda_event if hasattr(ev, "cuda_event") else int(ev)
    if not h:
        raise ValueError("the event has no CUDA handle yet: record it once first")
    return h


def resbm_boundary_step_host(desc, ws, stream=None, wait_before_inputs=None, inputs_done=None, **tensors):
    """resbm_boundary_step with host tensors (CPU torch tensors, pinned for asynchronous
    copies); ws is the device workspace of RESBM_OP_BOUNDARY_STEP_HOST. wait_before_inputs /
    inputs_done: torch.cuda.Event objects chaining consecutive calls' host-to-device copies."""
    args = resbm_step_args(**{k: _p(v) for k, v in tensors.items()},
                           wait_before_inputs=_event(wait_before_inputs), inputs_done=_event(inputs_done))
    st = load().resbm_boundary_step_host(ctypes.byref(desc), ctypes.byref(args), _p(ws), _nbytes(ws),
                                         _stream(stream))
    _check("resbm_boundary_step_host", st)


# ---- convenience: output buffers of one boundary step (allocated by torch) -------------------
def step_outputs(desc: resbm_desc, device="cuda", with_dX=True) -> dict:
    T, d, r, m = desc.T, desc.d, desc.r, desc.m
    io = TORCH_DTYPES[desc.dtype]
    f32 = torch.float32
    out = dict(B=torch.empty(T, r, dtype=io, device=device),
               P=torch.empty(T, m, dtype=f32, device=device),
               Y=torch.empty(T, d, dtype=io, device=device),
               dB=torch.empty(T, r, dtype=io, device=device),
               dF=torch.empty(T, d, dtype=io, device=device),
               dWe1=torch.empty(d, m, dtype=f32, device=device),
               dWe2=torch.empty(m, r, dtype=f32, device=device),
               dWd1=torch.empty(r, m, dtype=f32, device=device),
               dWd2=torch.empty(m, d, dtype=f32, device=device))
    if with_dX:
        out["dX"] = torch.zeros(T, d, dtype=io, device=device)
    return out


# ---- utilities on the bottleneck weights ------------------------------------------------------
def resbm_matrix_workspace_bytes(op: int, rows: int, cols: int) -> int:
    out = ctypes.c_size_t(0)
    _check("resbm_matrix_workspace_bytes", load().resbm_matrix_workspace_bytes(int(op), int(rows), int(cols),
                                                                               ctypes.byref(out)))
    return int(out.value)


def matrix_workspace(op: int, rows: int, cols: int, device="cuda") -> torch.Tensor:
    return torch.empty(max(resbm_matrix_workspace_bytes(op, rows, cols), 1), dtype=torch.uint8, device=device)


def resbm_newton_schulz(G, steps, X, ws, stream=None):
    """X (bf16, G's shape) = Muon's Newton-Schulz orthogonalisation of G (fp32 or bf16)."""
    rows, cols = G.shape
    g_dtype = RESBM_F32 if G.dtype == torch.float32 else RESBM_BF16
    _check("resbm_newton_schulz", load().resbm_newton_schulz(rows, cols, _p(G), g_dtype, int(steps), _p(X), _p(ws),
                                                             _nbytes(ws), _stream(stream)))


def resbm_effective_rank(W, out, ws, stream=None):
    """out (device float64, 4): sigma_max^2, ||W||_F^2, r_eff, power iterations taken."""
    rows, cols = W.shape
    _check("resbm_effective_rank", load().resbm_effective_rank(rows, cols, _p(W), _p(out), _p(ws), _nbytes(ws),
                                                               _stream(stream)))


# ---- the encoder fused into the FFN down-projection ------------------------------------------
def resbm_ffn_down_encode_workspace_bytes(desc: resbm_desc, f: int) -> int:
    out = ctypes.c_size_t(0)
    _check("resbm_ffn_down_encode_workspace_bytes",
           load().resbm_ffn_down_encode_workspace_bytes(ctypes.byref(desc), int(f), ctypes.byref(out)))
    return int(out.value)


def ffn_down_encode_workspace(desc: resbm_desc, f: int, device="cuda") -> torch.Tensor:
    return torch.empty(max(resbm_ffn_down_encode_workspace_bytes(desc, f), 1), dtype=torch.uint8, device=device)


def resbm_ffn_down_encode_fwd(desc, H, W2, X, We1, We2, B, P_save, F_out, ws, stream=None):
    """B (and P_save, F_out if given) from the FFN hidden state H (T x f) and the down-projection
    W2 (f x d): the encoder applied to F = H . W2 without storing F unless F_out is given."""
    f = H.shape[1]
    st = load().resbm_ffn_down_encode_fwd(ctypes.byref(desc), int(f), _p(H), _p(W2), _p(X), _p(We1), _p(We2),
                                          _p(B), _p(P_save), _p(F_out), _p(ws), _nbytes(ws), _stream(stream))
    _check("resbm_ffn_down_encode_fwd", st)
