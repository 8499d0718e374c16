"""GPU parity of the MXFP4 path (offsets as zero-points, Sec. 3.4 extension)
against the oracle (quantize_act_mx, prepare_weight_mx, mx_linear).

* Codes are decided in fp32 on the residual the kernel rotates in fp32, and in
  float64 by the oracle: a block exponent may differ only where the block's
  largest magnitude lies within the rotation's error bound of a power of two (and
  then the whole row's shifts may move with it); a code may differ by one
  magnitude step only where r / 2^X lies within that bound of one of the
  rounding decision points 0.25, 0.75, 1.25, 1.75, 2.5, 3.5, 5; at most 1e-4 of
  the codes.
* The weights' operand block sums are exact (multiples of 1/2).
* GEMM outputs, from the GPU's own codes: products of E4M3 values are exact, the
  fp32 accumulation of K of them errs by at most 2 K u times the sum of their
  magnitudes, the epilogue chain by (G + 4) u times its terms, plus half an ulp
  of a 16-bit output."""

import math

import numpy as np
import pytest
import torch

import oracle as O
import workloads as W
from paper_2606_07116_gb300 import build as B
from paper_2606_07116_gb300 import offq as Q
from parity import U32, check_offsets, rotation_abs_error

pytestmark = pytest.mark.gpu

DECISIONS = np.array([0.25, 0.75, 1.25, 1.75, 2.5, 3.5, 5.0])
OUT_DT = {"f32": torch.float32, "bf16": torch.bfloat16, "f16": torch.float16}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    B.build()
    Q.load_library()


def _decode(codes, shifts, scale, R, K):
    code = O.unpack_mx_codes(O.untile_codes(codes.cpu().numpy(), R, K))
    sh = O.untile_mx_shifts(shifts.cpu().numpy(), R, K)
    xlo = np.round(np.log2(scale.cpu().numpy().astype(np.float64))).astype(np.int64)
    return code, sh, sh + xlo[:, None]


def check_mx(code, X, ref, x, g, rotate, what="mx"):
    """GPU codes / exponents against the oracle's quantize_mx_rows result on the same rows."""
    T, K = code.shape
    r = ref["residual"]
    err = rotation_abs_error(x, g, rotate)[:, None] / (math.sqrt(g) if rotate else 1.0) + 4 * U32 * np.abs(r).max()
    amax = np.abs(r.reshape(T, K // 32, 32)).max(axis=2)
    with np.errstate(divide="ignore"):
        near_pow2 = np.abs(amax - np.exp2(np.round(np.log2(np.maximum(amax, 1e-300))))) <= 2 * err
    xd = X != ref["X"]
    rows_moved = near_pow2.any(axis=1)
    assert np.all(near_pow2[xd] | rows_moved.repeat(K // 32).reshape(T, -1)[xd]), f"{what}: exponent off a power of two"
    same = np.repeat(~xd, 32, axis=1)
    m = np.abs(r) / np.repeat(np.ldexp(1.0, ref["X"]), 32, axis=1)
    tol = np.repeat(err / np.ldexp(1.0, ref["X"]), 32, axis=1)
    near = (np.abs(m[..., None] - DECISIONS) <= tol[..., None] + 1e-6).any(axis=-1)
    d = np.abs(O.e2m1_value(code)) != np.abs(O.e2m1_value(ref["code"]))
    bad = same & d & ~near
    assert not bad.any(), f"{what}: {bad.sum()} codes differ away from a decision point"
    sign_bad = same & (np.sign(O.e2m1_value(code)) * np.sign(O.e2m1_value(ref["code"])) < 0)
    assert not sign_bad.any(), f"{what}: sign differs"
    assert (same & d).sum() <= max(1, 1e-4 * code.size), f"{what}: {(same & d).sum()} codes differ"


def _quant(x_np, g, rotate, dt="bf16"):
    xt = torch.from_numpy(x_np).to(OUT_DT[dt] if dt != "f32" else torch.float32)
    codes, shifts, scale, off = Q.quantize_act_mx(xt.cuda(), g, rotate=rotate, offset=True)
    torch.cuda.synchronize()
    assert Q.offq_get_device_status() == Q.OFFQ_OK
    return xt.to(torch.float64).numpy(), codes, shifts, scale, off


@pytest.mark.parametrize("dt", ["bf16", "f32", "f16"])
@pytest.mark.parametrize("T,K,g,rotate", [(37, 512, 512, True), (16, 4096, 1024, True), (45, 4096, 4096, False),
                                          (9, 11008, 256, True), (5, 384, 128, False)])
def test_mx_quantizer_parity(dt, T, K, g, rotate):
    x = W.activations(T, K, seed=T + K, n_out=3, mult=90.0)
    xe, codes, shifts, scale, off = _quant(x, g, rotate, dt)
    ref = O.quantize_act_mx(xe, g, rotate=rotate, offset=True)
    code, sh, X = _decode(codes, shifts, scale, T, K)
    check_mx(code, X, ref, xe, g, rotate)
    check_offsets(off.cpu().numpy(), ref["offset"], xe, g, rotate)
    assert np.all((sh >= 0) & (sh <= O.MX_SPAN))


@pytest.mark.parametrize("T,K,g,rotate,dt", [
    (700, 28672, 1024, True, "bf16"),     # Llama-2-70B down-proj width: one row of 28 warps per CTA
    (1200, 8192, 8192, False, "bf16"),    # one offset block over the 8 warps of a row
    (2000, 4096, 2048, False, "f16"),     # offset blocks of two warps
    (1500, 2048, 1024, True, "f32"),      # two rows per CTA, fp32 rows
    (5003, 1024, 1024, False, "bf16"),    # four rows of one warp per CTA, a ragged last group
])
def test_mx_quantizer_persistent_form(T, K, g, rotate, dt):
    """Prefill-sized inputs take the persistent warp-per-1024-channel MX kernel: sampled rows
    (first and last included) against the oracle."""
    x = W.activations(T, K, seed=T + K + g, n_out=4, mult=100.0)
    xe, codes, shifts, scale, off = _quant(x, g, rotate, dt)
    rows = np.unique(np.concatenate([W.unit_index_sample(T, 96, seed=13), [0, 1, T - 2, T - 1]]))
    ref = O.quantize_act_mx(xe[rows], g, rotate=rotate, offset=True)
    code, sh, X = _decode(codes, shifts, scale, T, K)
    check_mx(code[rows], X[rows], ref, xe[rows], g, rotate)
    check_offsets(off.cpu().numpy()[rows], ref["offset"], xe[rows], g, rotate)
    assert np.all((sh >= 0) & (sh <= O.MX_SPAN))


def test_mx_weight_prep_and_block_sums():
    N, K, g = 300, 1024, 256
    w = W.weights(N, K, seed=91)
    wc, ws, wsc, wsum = Q.prepare_weight_mx(torch.from_numpy(w).cuda(), g, rotate=True)
    torch.cuda.synchronize()
    ref = O.prepare_weight_mx(w.astype(np.float64), g, rotate=True)
    code, sh, X = _decode(wc, ws, wsc, N, K)
    check_mx(code, X, ref, w.astype(np.float64), g, True)
    opv = O.e2m1_value(code) * np.repeat(np.ldexp(1.0, sh), 32, axis=1)
    np.testing.assert_array_equal(wsum.cpu().numpy(), opv.reshape(N, K // g, g).sum(axis=2).T.astype(np.float32))
    # Padding rows of the last 32-row group are zero codes and shifts.
    tail = O.untile_codes(wc.cpu().numpy(), Q.padded_rows(N), K)[N:]
    assert not tail.any()
    assert not O.untile_mx_shifts(ws.cpu().numpy(), Q.padded_rows(N), K)[N:].any()


def _check_mx_layer(T, K, N, g, out_dt, rotate, seed=0, rows=None, dist="normal", n_out=3, mult=90.0):
    x = W.activations(T, K, seed=seed, dist=dist, n_out=n_out, mult=mult)
    gen = torch.Generator(device="cuda").manual_seed(seed + 1)
    w = torch.randn((N, K), generator=gen, device="cuda") * 0.02
    ac, ash, asc, aoff = Q.quantize_act_mx(torch.from_numpy(x).to(torch.bfloat16).cuda(), g, rotate=rotate)
    wc, wsh, wsc, wsum = Q.prepare_weight_mx(w, g, rotate=rotate)
    out = torch.full((T, N), float("nan"), dtype=OUT_DT[out_dt], device="cuda")
    Q.offq_mx_linear(ac, ash, asc, aoff, T, N, K, g, wc, wsh, wsc, wsum, out, N)
    torch.cuda.synchronize()
    assert Q.offq_get_device_status() == Q.OFFQ_OK
    sel = np.arange(T) if rows is None else rows
    y = out.index_select(0, torch.from_numpy(sel).cuda()).float().cpu().numpy().astype(np.float64)
    acode, ash_np, _ = _decode(ac, ash, asc, T, K)
    wcode, wsh_np, _ = _decode(wc, wsh, wsc, N, K)
    A = (O.e2m1_value(acode) * np.repeat(np.ldexp(1.0, ash_np), 32, axis=1))[sel]
    Wv = O.e2m1_value(wcode) * np.repeat(np.ldexp(1.0, wsh_np), 32, axis=1)
    sa = asc.cpu().numpy().astype(np.float64)[sel]
    sw = wsc.cpu().numpy().astype(np.float64)
    o = aoff.cpu().numpy().astype(np.float64)[sel]
    R = wsum.cpu().numpy().astype(np.float64)
    acc = A @ Wv.T
    absacc = np.abs(A) @ np.abs(Wv).T
    corr = o @ R
    y_ref = sw[None, :] * (sa[:, None] * acc + corr)
    G = K // g
    tol = sw[None, :] * (sa[:, None] * 2 * K * U32 * absacc + (G + 4) * U32 * (np.abs(sa[:, None] * acc)
                                                                              + np.abs(o) @ np.abs(R)))
    if out_dt == "bf16":
        tol = tol + 2.0 ** -8 * np.abs(y_ref)
    elif out_dt == "f16":
        tol = tol + 2.0 ** -11 * np.abs(y_ref) + 2.0 ** -25
    err = np.abs(y - y_ref)
    assert np.all(err <= tol + 1e-30), f"{(err > tol).sum()} outputs out of bound; worst {np.max(err / (tol + 1e-30)):.3g}x"
    return y, x[sel], w


@pytest.mark.parametrize("T,K,N,g,out_dt,rotate", [
    (16, 512, 512, 512, "f32", True),      # the toy layer's shape
    (300, 1024, 640, 256, "bf16", True),   # two m-pairs, ragged N, 4 offset blocks
    (64, 4096, 1000, 4096, "f16", False),  # one block of 4096, ragged N
    (130, 11008, 264, 256, "bf16", True),  # 43 offset blocks
    (5, 384, 200, 128, "f32", False),      # three k-tiles, a few tokens
])
def test_mx_gemm_layers(T, K, N, g, out_dt, rotate):
    y, x, w = _check_mx_layer(T, K, N, g, out_dt, rotate, seed=T + N)
    if rotate and T >= 16:
        ref = O.linear_reference(x, w.cpu().numpy())
        assert np.linalg.norm(y - ref) < 0.3 * np.linalg.norm(ref)


def test_mx_gemm_llama2_7b_gate_sampled():
    """The bench's gate projection (2048 x 4096 -> 11008) on sampled rows."""
    rows = np.unique(np.concatenate([W.unit_index_sample(2048, 48, seed=92), [0, 2047]]))
    _check_mx_layer(2048, 4096, 11008, 4096, "bf16", False, seed=93, rows=rows, n_out=4, mult=100.0)
