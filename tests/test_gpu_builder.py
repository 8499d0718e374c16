"""GPU parity of the offline transform builder (Sec. 3.1-3.3) against the oracle.

* Top-1 token indices, the copied rows and column maxima are exact (max of
  absolute values is exact in fp32 for bf16 / fp32 inputs).
* The power-iteration direction agrees with the oracle's eigensolver: with
  eigenvalue ratio r = lam2 / lam1, iters steps leave an angle of order
  r^iters, plus fp32 rounding; the tests use well-separated spectra (a planted
  outlier direction) and check 1 - |v . v_ref| against that.
* Reflection and fusion are fp32 chains: a dot product of D terms, one
  multiply-add per element and log2(g) butterfly stages. Each output is within
  (D + log2 g + 8) u times the sum of the magnitudes its chain adds.
"""

import math

import numpy as np
import pytest
import torch

import oracle as O
from paper_2606_07116_gb300 import build as B
from paper_2606_07116_gb300 import offq as Q
from parity import U32

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    B.build()
    Q.load_library()


def _calibration(S, L, D, seed, mag=(60.0, 120.0)):
    rng = np.random.default_rng(seed)
    v = rng.standard_normal(D)
    v /= np.linalg.norm(v)
    x = rng.standard_normal((S, L, D))
    spikes = rng.integers(0, L, size=S)
    x[np.arange(S), spikes] += rng.uniform(*mag, size=S)[:, None] * v
    return x, v, spikes


@pytest.mark.parametrize("dt", [torch.bfloat16, torch.float32])
def test_top1_tokens_exact(dt):
    S, L, D = 24, 96, 512
    x, _, spikes = _calibration(S, L, D, seed=80)
    xt = torch.from_numpy(x).to(dt)
    idx, rows = Q.top1_tokens(xt.cuda())
    torch.cuda.synchronize()
    ref_idx, ref_rows = O.top1_tokens(xt.to(torch.float64).numpy())
    np.testing.assert_array_equal(idx.cpu().numpy(), ref_idx)
    np.testing.assert_array_equal(idx.cpu().numpy(), spikes)
    np.testing.assert_array_equal(rows.cpu().numpy().astype(np.float64), ref_rows)


def test_top1_direction_matches_eigensolver():
    S, L, D = 64, 32, 1024
    x, v_true, _ = _calibration(S, L, D, seed=81)
    _, X = O.top1_tokens(x)
    X32 = X.astype(np.float32)
    v_ref, lam1, lam2 = O.top1_pca(X32.astype(np.float64))
    iters = 60
    v, proj = Q.top1_direction(torch.from_numpy(X32).cuda(), iters=iters)
    torch.cuda.synchronize()
    vg = v.cpu().numpy().astype(np.float64)
    ratio = lam2 / lam1
    bound = 4 * ratio ** iters + 1e3 * U32 * math.sqrt(D)
    assert abs(np.linalg.norm(vg) - 1) < 1e-5
    assert 1 - vg @ v_ref <= bound, (1 - vg @ v_ref, bound)
    np.testing.assert_allclose(proj.cpu().numpy(), X32.astype(np.float64) @ vg,
                               atol=(D + 8) * U32 * np.abs(X32).sum(axis=1).max())


def _check_rows(out, ref, A, w_max, extra_terms=0):
    D = A.shape[1]
    tol = (D + extra_terms + 8) * U32 * (np.abs(A).sum(axis=1, keepdims=True) * (1 + 2 * w_max) + 1e-30)
    err = np.abs(out - ref)
    assert np.all(err <= tol), f"worst {np.max(err / tol):.3g}x the bound"


def test_reflect_rows_and_column_absmax():
    rng = np.random.default_rng(82)
    R, D = 40, 2048
    A = rng.standard_normal((R, D)).astype(np.float32)
    v = rng.standard_normal(D).astype(np.float32)
    out = Q.reflect_rows(torch.from_numpy(A).cuda(), torch.from_numpy(v).cuda())
    mag = Q.column_absmax(out)
    torch.cuda.synchronize()
    U = O.householder_to_first(v.astype(np.float64))
    ref = A.astype(np.float64) @ U
    _check_rows(out.cpu().numpy().astype(np.float64), ref, A.astype(np.float64), 2.0)
    np.testing.assert_array_equal(mag.cpu().numpy(), np.max(np.abs(out.cpu().numpy()), axis=0))


@pytest.mark.parametrize("D,g", [(1024, 1024), (4096, 128), (512, 2)])
def test_fuse_rotation_parity(D, g):
    rng = np.random.default_rng(83)
    N = 33
    W = (rng.standard_normal((N, D)) * 0.02).astype(np.float32)
    v = rng.standard_normal(D).astype(np.float32)
    perm = O.sorted_grouping(rng.standard_normal(D), D // g)
    out = Q.fuse_rotation(torch.from_numpy(W).cuda(), torch.from_numpy(v).cuda(),
                          torch.from_numpy(perm.astype(np.int32)), g)
    torch.cuda.synchronize()
    M = O.offset_basis(v.astype(np.float64), perm, g)
    ref = O.fuse_rotation(W.astype(np.float64), M)
    _check_rows(out.cpu().numpy().astype(np.float64), ref, W.astype(np.float64), 2.0, int(math.log2(g)) + 1)


def test_builder_end_to_end_preserves_layer_and_offsets_outlier():
    """GPU builder on calibration data: the fused weights reproduce W x for
    activations rotated by the same M, and the planted direction leaves as one
    group's offset."""
    S, L, D, G = 48, 32, 1024, 8
    g = D // G
    x, v_true, _ = _calibration(S, L, D, seed=84)
    xt = torch.from_numpy(x).to(torch.bfloat16).cuda()
    _, rows = Q.top1_tokens(xt)
    v, _ = Q.top1_direction(rows, iters=60)
    mag = Q.column_absmax(Q.reflect_rows(rows, v))
    perm = Q.sorted_grouping(mag, G)
    W = np.random.default_rng(85).standard_normal((16, D)).astype(np.float32) * 0.02
    Wf = Q.fuse_rotation(torch.from_numpy(W).cuda(), v, perm, g)
    torch.cuda.synchronize()
    M = O.offset_basis(v.cpu().numpy().astype(np.float64), perm.numpy(), g)
    Xs = rows.cpu().numpy().astype(np.float64)
    Xr = Xs @ M
    np.testing.assert_allclose(Xr @ Wf.cpu().numpy().astype(np.float64).T, Xs @ W.astype(np.float64).T,
                               rtol=1e-4, atol=1e-4 * np.abs(Xs @ W.T).max())
    # The calibration estimate of the planted direction: with S tokens of D
    # unit-variance channels and spikes a >= 60, the angle is about
    # sqrt(D / S) / a (~0.08 here), so 1 - cos stays below 1e-2.
    assert abs(abs(v.cpu().numpy() @ v_true) - 1) < 1e-2
    offs = np.abs(Xr.reshape(S, G, g).mean(axis=2)).mean(axis=0)
    assert offs.max() > 5 * np.sort(offs)[-2]
