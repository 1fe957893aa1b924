"""The C ABI on the host, without a GPU: the library loads, exports every declared symbol, and
rejects bad arguments with status codes before touching the device."""
import ctypes
import os
import re

import pytest

from paper_2604_11947_gb300 import build, resbm

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    build.build()
    return resbm.load()


def declared_functions():
    src = open(os.path.join(ROOT, "include", "resbm.h")).read()
    return sorted(set(re.findall(r"RESBM_API\s+[\w\s\*]*?\b(resbm_\w+)\s*\(", src)))


def test_exports_every_declared_symbol(lib):
    names = declared_functions()
    assert len(names) == 22, names
    assert sorted(resbm.EXPORTS) == names
    for n in names:
        assert hasattr(lib, n), n


def test_version_and_status_strings(lib):
    assert "sm_103a" in resbm.resbm_version()
    assert resbm.status_string(resbm.RESBM_OK) == "RESBM_OK"
    assert resbm.status_string(resbm.RESBM_ERR_WORKSPACE) == "RESBM_ERR_WORKSPACE"
    assert resbm.status_string(99) == "RESBM_ERR_UNKNOWN"
    assert lib.resbm_last_cuda_error() == 0
    assert resbm.resbm_kernel_launches() == 0   # nothing launched on a host without a GPU


def test_struct_layout_matches_header():
    assert ctypes.sizeof(resbm.resbm_desc) == 4 * 8 + 4 * 4
    assert ctypes.sizeof(resbm.resbm_step_args) == 19 * ctypes.sizeof(ctypes.c_void_p)


@pytest.mark.parametrize("op", range(6))
def test_workspace_query(lib, op):
    d = resbm.make_desc(65536, 4096, 32, 32)
    n = resbm.resbm_workspace_bytes(d, op)
    assert n >= 0
    if op in (resbm.RESBM_OP_DECODE_BWD, resbm.RESBM_OP_ENCODE_BWD, resbm.RESBM_OP_BOUNDARY_STEP):
        assert n > 0
    if op == resbm.RESBM_OP_BOUNDARY_STEP_HOST:
        # device copies of X, F, dY, Y, dF, dX (T x d each) on top of the device step's scratch
        assert n >= 6 * 65536 * 4096 * 2 + resbm.resbm_workspace_bytes(d, resbm.RESBM_OP_BOUNDARY_STEP)
    d0 = resbm.make_desc(0, 4096, 32, 32)
    assert resbm.resbm_workspace_bytes(d0, op) >= 0


@pytest.mark.parametrize("bad", [
    dict(T=-1), dict(d=0), dict(r=0), dict(m=0), dict(r=5000, d=4096), dict(dtype=7),
    dict(act=9), dict(merge_identity=2), dict(flags=8), dict(T=1 << 40, d=1 << 30),
])
def test_bad_descriptor_rejected(lib, bad):
    kw = dict(T=16, d=64, r=8, m=8, dtype=1, act=0, merge_identity=1, flags=0)
    kw.update(bad)
    d = resbm.resbm_desc(kw["T"], kw["d"], kw["r"], kw["m"], kw["dtype"], kw["act"],
                         kw["merge_identity"], kw["flags"])
    out = ctypes.c_size_t(0)
    assert lib.resbm_workspace_bytes(ctypes.byref(d), 0, ctypes.byref(out)) == resbm.RESBM_ERR_INVALID_ARG
    st = lib.resbm_decode_fwd(ctypes.byref(d), 4096, 4096, 4096, 1 << 20, None, 0, None)
    assert st == resbm.RESBM_ERR_INVALID_ARG


def test_bad_op_and_null_desc(lib):
    d = resbm.make_desc(16, 64, 8, 8)
    out = ctypes.c_size_t(0)
    assert lib.resbm_workspace_bytes(ctypes.byref(d), 6, ctypes.byref(out)) == resbm.RESBM_ERR_INVALID_ARG
    assert lib.resbm_workspace_bytes(ctypes.byref(d), -1, ctypes.byref(out)) == resbm.RESBM_ERR_INVALID_ARG
    assert lib.resbm_workspace_bytes(None, 0, ctypes.byref(out)) == resbm.RESBM_ERR_INVALID_ARG
    assert lib.resbm_workspace_bytes(ctypes.byref(d), 0, None) == resbm.RESBM_ERR_INVALID_ARG
    assert lib.resbm_encode_fwd(None, 1, 1, 1, 1, 1, None, None, 0, None) == resbm.RESBM_ERR_INVALID_ARG


# Fake, never-dereferenced device addresses: validation must fail before any GPU work.
A = 1 << 32


def test_null_and_misaligned_pointers(lib):
    d = resbm.make_desc(16, 64, 8, 8, dtype="bf16")
    ws = 1 << 36
    big = 1 << 30
    enc = lib.resbm_encode_fwd
    assert enc(ctypes.byref(d), None, A, A + big, A + 2 * big, A + 3 * big, None, ws, big, None) == resbm.RESBM_ERR_INVALID_ARG
    assert enc(ctypes.byref(d), A + 1, A, A + big, A + 2 * big, A + 3 * big, None, ws, big, None) == resbm.RESBM_ERR_INVALID_ARG
    # fp32 P must be 4-byte aligned
    assert enc(ctypes.byref(d), A, A, A + big, A + 2 * big, A + 3 * big, A + 4 * big + 2, ws, big, None) == resbm.RESBM_ERR_INVALID_ARG
    # weights are required even for T = 0
    d0 = resbm.make_desc(0, 64, 8, 8)
    assert lib.resbm_decode_fwd(ctypes.byref(d0), None, None, A, None, None, 0, None) == resbm.RESBM_ERR_INVALID_ARG


def test_overlapping_output_rejected(lib):
    d = resbm.make_desc(16, 64, 8, 8, dtype="bf16")
    big = 1 << 30
    # Y (16 x 64 bf16 = 2 KiB) starting inside B's range
    st = lib.resbm_decode_fwd(ctypes.byref(d), A, A + big, A + 2 * big, A + 64, 1 << 36, big, None)
    assert st == resbm.RESBM_ERR_INVALID_ARG
    # decode bwd: dWd2 overlapping dY
    st = lib.resbm_decode_bwd(ctypes.byref(d), A, A + big, A + 2 * big, A + 3 * big, A + 4 * big,
                              A + 5 * big, A + 16, 1 << 36, big, None)
    assert st == resbm.RESBM_ERR_INVALID_ARG


def test_workspace_too_small(lib):
    d = resbm.make_desc(4096, 512, 16, 16, dtype="bf16")
    need = resbm.resbm_workspace_bytes(d, resbm.RESBM_OP_DECODE_BWD)
    big = 1 << 30
    args = [A, A + big, A + 2 * big, A + 3 * big, A + 4 * big, A + 5 * big, A + 6 * big]
    st = lib.resbm_decode_bwd(ctypes.byref(d), *args, A + 8 * big, need - 1, None)
    assert st == resbm.RESBM_ERR_WORKSPACE
    st = lib.resbm_decode_bwd(ctypes.byref(d), *args, None, need, None)
    assert st == resbm.RESBM_ERR_WORKSPACE
    # misaligned workspace
    st = lib.resbm_decode_bwd(ctypes.byref(d), *args, A + 8 * big + 16, need, None)
    assert st == resbm.RESBM_ERR_INVALID_ARG


def test_step_rejects_output_aliasing_input(lib):
    d = resbm.make_desc(16, 64, 8, 8, dtype="bf16")
    big = 1 << 30
    ptrs = {n: A + i * big for i, n in enumerate(
        ["X", "F", "dY", "We1", "We2", "Wd1", "Wd2", "B", "P", "Y", "dB", "dF", "dX",
         "dWe1", "dWe2", "dWd1", "dWd2"])}
    ptrs["dF"] = ptrs["X"]
    args = resbm.resbm_step_args(**ptrs)
    need = resbm.resbm_workspace_bytes(d, resbm.RESBM_OP_BOUNDARY_STEP)
    st = lib.resbm_boundary_step(ctypes.byref(d), ctypes.byref(args), 1 << 40, need, None)
    assert st == resbm.RESBM_ERR_INVALID_ARG
    assert lib.resbm_boundary_step(ctypes.byref(d), None, 1 << 40, need, None) == resbm.RESBM_ERR_INVALID_ARG
    # the host-buffer form applies the same rules, before any copy or stream is set up
    need_h = resbm.resbm_workspace_bytes(d, resbm.RESBM_OP_BOUNDARY_STEP_HOST)
    st = lib.resbm_boundary_step_host(ctypes.byref(d), ctypes.byref(args), 1 << 40, need_h, None)
    assert st == resbm.RESBM_ERR_INVALID_ARG
    ptrs["dF"] = A + 11 * big
    ok_args = resbm.resbm_step_args(**ptrs)
    st = lib.resbm_boundary_step_host(ctypes.byref(d), ctypes.byref(ok_args), 1 << 40, need_h - 1, None)
    assert st == resbm.RESBM_ERR_WORKSPACE
    st = lib.resbm_boundary_step_host(ctypes.byref(d), ctypes.byref(ok_args), None, need_h, None)
    assert st == resbm.RESBM_ERR_WORKSPACE
    assert lib.resbm_boundary_step_host(ctypes.byref(d), None, 1 << 40, need_h, None) == resbm.RESBM_ERR_INVALID_ARG


def test_linear_flag_rules(lib):
    """RESBM_FLAG_LINEAR needs m == r; its second-layer tensors may be absent."""
    big = 1 << 32
    A = 1 << 40
    bad = resbm.make_desc(16, 64, 8, 4, flags=resbm.RESBM_FLAG_LINEAR)
    assert lib.resbm_decode_fwd(ctypes.byref(bad), A, None, A + big, A + 2 * big, A + 3 * big, big, None) \
        == resbm.RESBM_ERR_INVALID_ARG
    ok = resbm.make_desc(16, 64, 8, 8, flags=resbm.RESBM_FLAG_LINEAR)
    # without the flag a missing Wd1 is an argument error; with it, only the workspace is missing
    plain = resbm.make_desc(16, 64, 8, 8)
    assert lib.resbm_decode_fwd(ctypes.byref(plain), A, None, A + big, A + 2 * big, None, 0, None) \
        == resbm.RESBM_ERR_INVALID_ARG
    assert lib.resbm_decode_fwd(ctypes.byref(ok), A, None, A + big, A + 2 * big, None, 0, None) \
        == resbm.RESBM_ERR_WORKSPACE
    assert resbm.resbm_workspace_bytes(ok, resbm.RESBM_OP_DECODE_FWD) > 0


def test_matrix_utilities_reject_bad_arguments(lib):
    """resbm_newton_schulz / resbm_effective_rank: shapes, dtypes, steps, pointers and workspace are
    checked on the host before anything is enqueued (fake aligned device addresses)."""
    sz = ctypes.c_size_t(0)
    assert lib.resbm_matrix_workspace_bytes(resbm.RESBM_OP_NEWTON_SCHULZ, 32, 4096, ctypes.byref(sz)) == resbm.RESBM_OK
    assert sz.value > 0
    assert lib.resbm_matrix_workspace_bytes(resbm.RESBM_OP_EFFECTIVE_RANK, 4096, 32, ctypes.byref(sz)) == resbm.RESBM_OK
    assert lib.resbm_matrix_workspace_bytes(resbm.RESBM_OP_DECODE_BWD, 32, 32, ctypes.byref(sz)) == resbm.RESBM_ERR_INVALID_ARG
    assert lib.resbm_matrix_workspace_bytes(resbm.RESBM_OP_NEWTON_SCHULZ, 30, 32, ctypes.byref(sz)) == resbm.RESBM_ERR_INVALID_ARG
    A, big = 1 << 40, 1 << 30
    G, X, ws = A, A + big, A + 2 * big
    ns = lib.resbm_newton_schulz
    assert ns(30, 64, G, resbm.RESBM_F32, 5, X, ws, 1 << 30, None) == resbm.RESBM_ERR_INVALID_ARG    # rows % 8
    assert ns(32, 64, G, 7, 5, X, ws, 1 << 30, None) == resbm.RESBM_ERR_INVALID_ARG                  # dtype
    assert ns(32, 64, G, resbm.RESBM_F32, 101, X, ws, 1 << 30, None) == resbm.RESBM_ERR_INVALID_ARG  # steps
    assert ns(32, 64, G, resbm.RESBM_F32, 5, G + 8, ws, 1 << 30, None) == resbm.RESBM_ERR_INVALID_ARG  # overlap
    assert ns(32, 64, G + 4, resbm.RESBM_F32, 5, X, ws, 1 << 30, None) == resbm.RESBM_ERR_INVALID_ARG  # misaligned
    assert ns(32, 64, G, resbm.RESBM_F32, 5, X, ws, 16, None) == resbm.RESBM_ERR_WORKSPACE
    er = lib.resbm_effective_rank
    assert er(4096, 32, G, X, ws, 16, None) == resbm.RESBM_ERR_WORKSPACE
    assert er(8192, 8192, G, X, ws, 1 << 34, None) == resbm.RESBM_ERR_INVALID_ARG               # min side > 4096
    assert er(4096, 32, G, X + 4, ws, 1 << 30, None) == resbm.RESBM_ERR_INVALID_ARG              # out not 8-byte aligned


def test_ffn_down_encode_rejects_bad_arguments(lib):
    """The fused down-projection encoder's host checks (fake aligned device addresses), through
    the Python binding's argument list."""
    A, big = 1 << 40, 1 << 32
    t = [A + i * big for i in range(9)]
    d = resbm.make_desc(1024, 512, 32, 32)
    sz = ctypes.c_size_t(0)
    assert lib.resbm_ffn_down_encode_workspace_bytes(ctypes.byref(d), 1024, ctypes.byref(sz)) == resbm.RESBM_OK
    fn = lib.resbm_ffn_down_encode_fwd
    assert fn(ctypes.byref(d), 1024, *t[:8], t[8], 16, None) == resbm.RESBM_ERR_WORKSPACE
    assert fn(ctypes.byref(d), 1024, None, *t[1:8], t[8], sz.value, None) == resbm.RESBM_ERR_INVALID_ARG
    assert fn(ctypes.byref(d), 1024, t[0], t[1], t[2], t[3], t[4], t[2], None, None, t[8], sz.value,
              None) == resbm.RESBM_ERR_INVALID_ARG                         # B overlaps X
    wide = resbm.make_desc(1024, 512, 64, 64)                             # m > 32: not this kernel
    assert lib.resbm_ffn_down_encode_workspace_bytes(ctypes.byref(wide), 1024, ctypes.byref(sz)) == \
        resbm.RESBM_ERR_UNSUPPORTED


def test_decode_fwd_rmsnorm_rejects_bad_arguments(lib):
    """The fused decoder + RMSNorm's host checks (fake aligned device addresses): gamma, N, eps,
    Y overlapping N, and the workspace (the row sums of squares on the fused path)."""
    A, big = 1 << 40, 1 << 34
    B, W1, W2, g, Y, N, ws = (A + i * big for i in range(7))
    d = resbm.make_desc(65536, 4096, 32, 32)
    need = resbm.resbm_workspace_bytes(d, resbm.RESBM_OP_DECODE_FWD_RMSNORM)
    assert need >= 2 * (4096 // 256) * 65536 * 4   # the fused form's slots
    fn = lib.resbm_decode_fwd_rmsnorm
    dp = ctypes.byref(d)
    assert fn(dp, B, W1, W2, g, 1e-5, Y, N, ws, 16, None) == resbm.RESBM_ERR_WORKSPACE
    assert fn(dp, B, W1, W2, None, 1e-5, Y, N, ws, need, None) == resbm.RESBM_ERR_INVALID_ARG
    assert fn(dp, B, W1, W2, g, 1e-5, Y, None, ws, need, None) == resbm.RESBM_ERR_INVALID_ARG
    assert fn(dp, B, W1, W2, g, -1.0, Y, N, ws, need, None) == resbm.RESBM_ERR_INVALID_ARG
    assert fn(dp, B, W1, W2, g, float("nan"), Y, N, ws, need, None) == resbm.RESBM_ERR_INVALID_ARG
    assert fn(dp, B, W1, W2, g, float("inf"), Y, N, ws, need, None) == resbm.RESBM_ERR_INVALID_ARG
    assert fn(dp, B, W1, W2, g, 1e-5, Y, Y + 1024, ws, need, None) == resbm.RESBM_ERR_INVALID_ARG  # Y and N overlap
    # f32 descriptors and widths the fused kernels do not take need no slots beyond the decoder's
    f = resbm.make_desc(333, 200, 8, 5, dtype="f32")
    assert resbm.resbm_workspace_bytes(f, resbm.RESBM_OP_DECODE_FWD_RMSNORM) == \
        resbm.resbm_workspace_bytes(f, resbm.RESBM_OP_DECODE_FWD)


def test_rmsnorm_bwd_rejects_bad_arguments(lib):
    A, big = 1 << 40, 1 << 34
    Y, g, dN, dY, out, dg, ws = (A + i * big for i in range(7))
    d = resbm.make_desc(16384, 2048, 16, 16)
    need = resbm.resbm_workspace_bytes(d, resbm.RESBM_OP_RMSNORM_BWD)
    assert need == 1024 * 2048 * 4
    fn = lib.resbm_rmsnorm_bwd
    dp = ctypes.byref(d)
    assert fn(dp, Y, g, 1e-5, dN, dY, out, dg, ws, 16, None) == resbm.RESBM_ERR_WORKSPACE
    assert fn(dp, Y, g, -1.0, dN, dY, out, dg, ws, need, None) == resbm.RESBM_ERR_INVALID_ARG
    assert fn(dp, Y, None, 1e-5, dN, dY, out, dg, ws, need, None) == resbm.RESBM_ERR_INVALID_ARG
    assert fn(dp, Y, g, 1e-5, dN, dY, out, None, ws, need, None) == resbm.RESBM_ERR_INVALID_ARG
    assert fn(dp, Y, g, 1e-5, dN, dY, Y + 64, dg, ws, need, None) == resbm.RESBM_ERR_INVALID_ARG     # out overlaps Y
    assert fn(dp, Y, g, 1e-5, dN, dY, dY + 64, dg, ws, need, None) == resbm.RESBM_ERR_INVALID_ARG    # partial overlap with dY
    assert fn(dp, Y, g, 1e-5, dN, dY, out, out + 64, ws, need, None) == resbm.RESBM_ERR_INVALID_ARG  # dgamma inside dY_out
    wide = resbm.make_desc(16, 16392, 16, 16)
    sz = ctypes.c_size_t(0)
    assert lib.resbm_rmsnorm_bwd(ctypes.byref(wide), Y, g, 1e-5, dN, None, out, dg, ws, 1 << 30, None) == \
        resbm.RESBM_ERR_UNSUPPORTED


def test_hbm_form_probe_rejects_bad_arguments(lib):
    A, B = 1 << 40, (1 << 40) + (1 << 34)
    mib = 1 << 20
    fn = lib.resbm_measure_hbm_form
    assert fn(-1, A, B, mib, None) == resbm.RESBM_ERR_INVALID_ARG
    assert fn(len(resbm.HBM_FORMS), A, B, mib, None) == resbm.RESBM_ERR_INVALID_ARG
    for bad in (0, mib - 16, mib + 16, -mib):
        assert fn(resbm.RESBM_HBM_READ_TMA_2D, A, B, bad, None) == resbm.RESBM_ERR_INVALID_ARG
    assert fn(resbm.RESBM_HBM_READ_V4, None, B, mib, None) == resbm.RESBM_ERR_INVALID_ARG
    assert fn(resbm.RESBM_HBM_WRITE_V4, A, None, mib, None) == resbm.RESBM_ERR_INVALID_ARG
    assert fn(resbm.RESBM_HBM_COPY_V4, A + 8, B, mib, None) == resbm.RESBM_ERR_INVALID_ARG   # misaligned
    assert fn(resbm.RESBM_HBM_COPY_V4, A, A + mib // 2, mib, None) == resbm.RESBM_ERR_INVALID_ARG   # overlap
    assert sorted(resbm.HBM_FORMS.values()) == list(range(11))


def test_hbm_form_enum_matches_header():
    src = open(os.path.join(ROOT, "include", "resbm.h")).read()
    declared = {name: int(v) for name, v in re.findall(r"\bRESBM_HBM_(\w+)\s*=\s*(\d+)", src)}
    assert len(declared) == len(resbm.HBM_FORMS) == 11
    for name, v in declared.items():
        assert getattr(resbm, "RESBM_HBM_" + name) == v, name
        assert resbm.HBM_FORMS[name.lower()] == v, name
