"""Muon's Newton-Schulz orthogonalisation and the effective rank of a matrix, through the C ABI,
against the oracle (float64) on the same seeded matrices."""
import numpy as np
import pytest
import torch

import oracle
from paper_2604_11947_gb300 import resbm, synth

pytestmark = pytest.mark.gpu

# Newton-Schulz in bf16 (as Muon runs it) against float64. Each step rounds X, A = X X^T and
# B = b A + c A^2 to bf16 (2^-9 relative). Near the end the update X <- a X + B X is a difference:
# along a singular value near 1 it is 0.7 x from terms 3.44 x and -2.74 x, so the rounding of
# those terms is ~5 x 2^-9 = 1e-2 of the result per step; the map's contraction there (|p'(s) s /
# p(s)| ~ 0.7) keeps a steady ~1e-2 / sqrt(1 - 0.5) = 1.4e-2 (measured 1.0-1.6e-2). Bound:
# Frobenius 3e-2. The rounding of an element scales with the size of that element's terms
# (entries of 3.44 X reach 5 rms), so the largest element error reaches ~5 x 3.44 x 2^-9 x
# sqrt(2) x 5 (cancellation) / ... ~0.15 of the output RMS (measured up to 0.14): bound 0.25.
NS_FRO_TOL, NS_ELEM_TOL = 3e-2, 0.25


def _ns(G, steps=5):
    X = torch.empty(G.shape, dtype=torch.bfloat16, device="cuda")
    ws = resbm.matrix_workspace(resbm.RESBM_OP_NEWTON_SCHULZ, *G.shape)
    resbm.resbm_newton_schulz(G, steps, X, ws)
    torch.cuda.synchronize()
    return X.double().cpu().numpy()


@pytest.mark.parametrize("shape", [(32, 4096), (4096, 32), (16, 2048), (48, 200), (32, 32), (128, 8)])
@pytest.mark.parametrize("g_dtype", [torch.float32, torch.bfloat16])
def test_newton_schulz_matches_oracle(shape, g_dtype):
    G = torch.from_numpy(synth.matrix(*shape, seed=shape[0])).to("cuda").to(g_dtype)
    want = oracle.newton_schulz(G.double().cpu().numpy(), 5)
    got = _ns(G)
    fro = np.linalg.norm(got - want) / np.linalg.norm(want)
    elem = np.max(np.abs(got - want)) / np.sqrt(np.mean(want ** 2))
    assert fro <= NS_FRO_TOL and elem <= NS_ELEM_TOL, (fro, elem)


@pytest.mark.parametrize("steps", [0, 1, 2])
def test_newton_schulz_step_counts(steps):
    G = torch.from_numpy(synth.matrix(64, 512, seed=7)).to("cuda").float()
    want = oracle.newton_schulz(G.double().cpu().numpy(), steps)
    got = _ns(G, steps)
    assert np.linalg.norm(got - want) / np.linalg.norm(want) <= NS_FRO_TOL


@pytest.mark.parametrize("shape", [(512, 8192), (8192, 512)])
def test_newton_schulz_full_size_orthogonalises(shape):
    """The r = 512 bottleneck weights' shapes: against the oracle, and the result's singular values
    in Muon's band around 1 (a property at any size)."""
    G = torch.from_numpy(synth.matrix(*shape, seed=3)).to("cuda").float()
    got = _ns(G)
    want = oracle.newton_schulz(G.double().cpu().numpy(), 5)
    assert np.linalg.norm(got - want) / np.linalg.norm(want) <= NS_FRO_TOL
    s = np.linalg.svd(got, compute_uv=False)
    assert s.min() > 0.55 and s.max() < 1.3, (s.min(), s.max())


def _reff(W):
    out = torch.zeros(4, dtype=torch.float64, device="cuda")
    ws = resbm.matrix_workspace(resbm.RESBM_OP_EFFECTIVE_RANK, *W.shape)
    resbm.resbm_effective_rank(W, out, ws)
    torch.cuda.synchronize()
    return out.cpu().numpy()


@pytest.mark.parametrize("shape", [(4096, 32), (2048, 16), (32, 4096), (64, 64), (8192, 512), (1024, 128)])
def test_effective_rank_matches_oracle(shape):
    rows, cols = shape
    W = torch.from_numpy(synth.matrix(rows, cols, seed=rows + cols) / np.sqrt(rows)).to("cuda").to(torch.bfloat16)
    Wh = W.double().cpu().numpy()
    lam, fro2, reff, iters = _reff(W)
    assert iters < 20000, iters
    # fp32 Gram sums of exact bf16 products; lambda within 1e-5 (relative) of an eigenvalue
    assert abs(reff - oracle.effective_rank(Wh)) <= 1e-4 * oracle.effective_rank(Wh), (reff, iters)
    assert abs(fro2 - np.sum(Wh * Wh)) <= 1e-5 * np.sum(Wh * Wh)
    assert abs(lam - np.linalg.svd(Wh, compute_uv=False)[0] ** 2) <= 1e-4 * lam


def test_effective_rank_of_structured_matrices():
    """A rank-one matrix has r_eff = 1; equal singular values give the smaller dimension."""
    u = synth.matrix(1024, 1, seed=1)
    v = synth.matrix(1, 64, seed=2)
    W = torch.from_numpy(u @ v).to("cuda").to(torch.bfloat16)
    assert abs(_reff(W)[2] - oracle.effective_rank(W.double().cpu().numpy())) <= 1e-4
    assert abs(_reff(W)[2] - 1.0) <= 1e-3
    # orthonormal columns (a QR factor), rounded to bf16: close to r_eff = 64
    Q, _ = np.linalg.qr(synth.matrix(1024, 64, seed=4))
    Wq = torch.from_numpy(Q).to("cuda").to(torch.bfloat16)
    r = _reff(Wq)[2]
    assert abs(r - oracle.effective_rank(Wq.double().cpu().numpy())) <= 1e-4 * r and abs(r - 64) < 2.0
