"""Comparison helpers for the GPU-vs-oracle parity tests.

Tolerances follow from the arithmetic of the kernels (fp32, unit roundoff
u = 2^-24), never from observed differences:

* Codes. The kernel decides each code in fp32 and the oracle in float64, so a
  code may differ only where the oracle's r/s lies within the fp32 error of a
  rounding tie; mismatches must be +-1, within TIE_WINDOW code units of a
  half-integer, and at most 1e-4 of all codes (the stated bound).
* Scales and offsets. The kernel's transform is a radix-2 tree of L = log2(g)
  fp32 additions per output, so each rotated value carries an absolute error of
  at most L u sum|x| over its block; the scale inherits that relative to max|r|.
  The tensor-core form of g = 1024 (bf16 rows) sums the first 128 terms of each
  output (the H_128 factor) in the MMA's fp32 accumulator: its products are
  exact, and allowing each of the 128 additions two ulps (truncation), plus the
  removal of x[0] and the 3 register stages, the bound is TC_FACTOR u sum|x|
  over the block.
  There a code may also differ within that bound (in code units) of a tie.
  Without the rotation the offset is an fp32 block sum whose summation depth
  is at most g/8 + 16.
* GEMM outputs. Integer accumulators are exact, and so is the removal of the
  activation codes' +8 from them (an integer below 2^24). The epilogue is then
  a chain of G+2 fp32 multiply-adds over s_a acc and the offset terms o_b R_b,
  whose error is bounded by (G + 4) u times the sum of their magnitudes; a
  bf16 / fp16 result adds half an ulp of its own format (relative 2^-8 / 2^-11).
"""

from __future__ import annotations

import math

import numpy as np

U32 = 2.0 ** -24
TC_FACTOR = 2 * 128 + 8 + 1 + 3 + 4
TIE_WINDOW = 1e-3
MAX_MISMATCH_FRACTION = 1e-4


def check_codes(q_gpu: np.ndarray, q_ref: np.ndarray, r_ref: np.ndarray, s_ref: np.ndarray, what: str = "codes",
                window=None):
    """q_* int codes [rows, K]; r_ref residual [rows, K]; s_ref scale [rows] (oracle, float64).
    window: per-row tie window in code units (at least TIE_WINDOW) where the kernel's bound is wider."""
    q_gpu = np.asarray(q_gpu, dtype=np.int64)
    q_ref = np.asarray(q_ref, dtype=np.int64)
    assert q_gpu.shape == q_ref.shape, (q_gpu.shape, q_ref.shape)
    diff = q_gpu - q_ref
    mism = diff != 0
    n = int(mism.sum())
    if n == 0:
        return 0
    assert np.all(np.abs(diff) <= 1), f"{what}: a code differs by more than 1"
    s = np.broadcast_to(np.asarray(s_ref, np.float64).reshape(-1, *([1] * (q_ref.ndim - 1))), q_ref.shape)
    with np.errstate(divide="ignore", invalid="ignore"):
        z = np.where(s > 0, np.asarray(r_ref, np.float64) / s, 0.0)
    zm = np.abs(z[mism])
    dist = np.abs(zm - np.floor(zm) - 0.5)
    win = TIE_WINDOW
    if window is not None:
        w = np.broadcast_to(np.asarray(window, np.float64).reshape(-1, *([1] * (q_ref.ndim - 1))), q_ref.shape)
        win = np.maximum(TIE_WINDOW, w[mism])
    assert np.all(dist < win), f"{what}: mismatch away from a rounding tie (min dist {dist.max():.3g})"
    frac = n / q_ref.size
    assert frac <= MAX_MISMATCH_FRACTION, f"{what}: {n} codes differ ({frac:.2e} > {MAX_MISMATCH_FRACTION})"
    return n


def rotation_abs_error(x: np.ndarray, g: int, rotate: bool, tc: bool = False) -> np.ndarray:
    """Per-row bound on the absolute fp32 error of an unnormalised rotated value
    (tc: the tensor-core form of g = 1024)."""
    x = np.abs(np.asarray(x, np.float64))
    T, K = x.shape
    blk = x.reshape(T, K // g, g).sum(axis=2).max(axis=1)
    L = int(math.log2(g)) if rotate else 0
    return (TC_FACTOR if tc else L + 2) * U32 * blk


def code_window(s_ref, x, g, tc: bool = False):
    """Per-row tie window in code units: r / s moves by at most the residual's bound
    over s plus the scale's relative error times 7."""
    s_ref = np.asarray(s_ref, np.float64)
    err = rotation_abs_error(x, g, True, tc) / math.sqrt(g)
    with np.errstate(divide="ignore", invalid="ignore"):
        return np.where(s_ref > 0, 2.0 * err / s_ref, 0.0) + 1e-6


def tensor_core_form(x, g: int, rotate: bool, ldx=None) -> bool:
    """Whether offq_quantize_act takes the tensor-core form of g = 1024 for the torch
    tensor x: bf16 rows of 1024 G channels (G <= 64) with the rotation, a row pitch of a
    multiple of 8 elements, and at least as many tiles of 64 // G rows as SMs."""
    import torch
    T, K = x.shape
    ld = K if ldx is None else ldx
    if x.dtype != torch.bfloat16 or g != 1024 or not rotate or K % 1024 or K // 1024 > 64 or ld % 8:
        return False
    P = 64 // (K // 1024)
    return -(-T // P) >= torch.cuda.get_device_properties(0).multi_processor_count


def check_scales(s_gpu, s_ref, x, g, rotate, what="scale", tc=False):
    s_gpu = np.asarray(s_gpu, np.float64)
    s_ref = np.asarray(s_ref, np.float64)
    norm = math.sqrt(g) if rotate else 1.0
    err_u = rotation_abs_error(x, g, rotate, tc)      # on the unnormalised residual
    tol = err_u / (7.0 * norm) + 4 * U32 * np.abs(s_ref)
    bad = np.abs(s_gpu - s_ref) > tol
    assert not np.any(bad), f"{what}: {bad.sum()} rows out of tolerance; worst " \
                            f"{np.max(np.abs(s_gpu - s_ref) / np.maximum(tol, 1e-300)):.3g}x"


def check_offsets(o_gpu, o_ref, x, g, rotate, what="offset"):
    o_gpu = np.asarray(o_gpu, np.float64)
    o_ref = np.asarray(o_ref, np.float64)
    x = np.abs(np.asarray(x, np.float64))
    T, K = x.shape
    if rotate:
        tol = 4 * U32 * np.abs(o_ref)   # x[0] * fl(1/sqrt(g)): two roundings
    else:
        # A block sum in fp32 by balanced trees: every kernel adds the g values of a
        # block along paths of log2(g) additions (the 1/g is exact); one extra level
        # of slack.
        depth = int(math.log2(g)) + 1
        tol = depth * U32 * x.reshape(T, K // g, g).sum(axis=2) / g + 2 * U32 * np.abs(o_ref)
    bad = np.abs(o_gpu - o_ref) > tol
    assert not np.any(bad), f"{what}: {bad.sum()} offsets out of tolerance"


def epilogue_terms(acc, s_a, o, s_w, R):
    """Magnitudes the fp32 epilogue adds up (float64), for its error bound:
    s_w (|s_a acc| + sum_b |o_b| |R_b|), acc the integer dot product of the codes."""
    s_a = np.asarray(s_a, np.float64)
    s_w = np.abs(np.asarray(s_w, np.float64))
    o = np.abs(np.asarray(o, np.float64))
    return s_w[None, :] * (np.abs(s_a[:, None] * np.asarray(acc, np.float64)) + o @ np.abs(R))


def check_outputs(y_gpu, y_ref, terms, G, out_dtype: str, what="y"):
    y_gpu = np.asarray(y_gpu, np.float64)
    y_ref = np.asarray(y_ref, np.float64)
    tol = (G + 4) * U32 * terms + 1e-30
    if out_dtype == "bf16":
        tol = tol + 2.0 ** -8 * np.abs(y_ref)
    elif out_dtype == "f16":
        tol = tol + 2.0 ** -11 * np.abs(y_ref) + 2.0 ** -25
    err = np.abs(y_gpu - y_ref)
    bad = err > tol
    assert not np.any(bad), f"{what}: {bad.sum()} of {bad.size} outputs out of tolerance; worst " \
                            f"{np.max(err / tol):.3g}x the bound"
    return float(np.max(err / np.maximum(np.abs(y_ref), 1e-2 * np.sqrt(np.mean(y_ref ** 2)) + 1e-30)))


def max_rel_err_floored(y_gpu, y_ref):
    """max |y - y_ref| / max(|y_ref|, 1e-2 rms(y_ref)) (elementwise relative error with a floor)."""
    y_gpu = np.asarray(y_gpu, np.float64)
    y_ref = np.asarray(y_ref, np.float64)
    floor = 1e-2 * np.sqrt(np.mean(y_ref ** 2)) + 1e-30
    return float(np.max(np.abs(y_gpu - y_ref) / np.maximum(np.abs(y_ref), floor)))


def act_q(codes, T: int, K: int) -> np.ndarray:
    """Integer codes [T, K] from a tiled activation-code buffer (decoded by the oracle)."""
    import oracle as O
    arr = codes.cpu().numpy() if hasattr(codes, "cpu") else np.asarray(codes)
    return O.unpack_act_codes(O.untile_codes(arr, T, K))


def weight_q(codes, N: int, K: int) -> np.ndarray:
    """Integer codes [N, K] from a tiled weight-code buffer (decoded by the oracle)."""
    import oracle as O
    arr = codes.cpu().numpy() if hasattr(codes, "cpu") else np.asarray(codes)
    return O.unpack_weight_codes(O.untile_codes(arr, N, K))


def check_group_quant(q_gpu, s_gpu, z_gpu, ref, x, g, rotate, group=128, what="group"):
    """Per-group asymmetric quantizer (GPU, fp32 decisions) against the oracle.

    q_gpu [T, K] codes in [0, 15]; s_gpu, z_gpu [T, K/group]; ref the oracle's
    quantize_act_group result on the same input.
    * Scales: the group range comes from rotated values each off by at most
      the rotation bound, so s differs by at most 2/15 of it (over sqrt(g))
      plus a few roundings.
    * Zero-points: equal, except +-1 where the oracle's min/s lies within
      TIE_WINDOW of a half-integer.
    * Codes, compared as q - z (what dequantizes): equal, except +-1 where
      y/s lies within TIE_WINDOW of a half-integer, or at the grid's ends of a
      group whose zero-point took the other side of a tie; at most
      MAX_MISMATCH_FRACTION of all codes.
    """
    q_gpu = np.asarray(q_gpu, np.int64)
    s_gpu = np.asarray(s_gpu, np.float64)
    z_gpu = np.asarray(z_gpu, np.float64)
    s_ref, z_ref, q_ref, y = ref["scale"], ref["zero"], ref["q"], ref["y"]
    T, K = q_ref.shape
    Gq = K // group
    norm = math.sqrt(g) if rotate else 1.0
    err_u = rotation_abs_error(x, g, rotate)[:, None]
    tol_s = 2.0 * err_u / (15.0 * norm) + 4 * U32 * np.abs(s_ref)
    bad = np.abs(s_gpu - s_ref) > tol_s
    assert not np.any(bad), f"{what}: {bad.sum()} scales out of tolerance"
    yg = y.reshape(T, Gq, group)
    with np.errstate(divide="ignore", invalid="ignore"):
        t_min = np.where(s_ref > 0, yg.min(axis=2) / s_ref, 0.0)
        ratio = np.where(np.repeat(s_ref, group, axis=1) > 0, y / np.repeat(s_ref, group, axis=1), 0.0)
    near = lambda v: np.abs(np.abs(v) - np.floor(np.abs(v)) - 0.5) < TIE_WINDOW
    zd = z_gpu != z_ref
    assert np.all(np.abs(z_gpu - z_ref)[zd] <= 1) and np.all(near(t_min[zd])), f"{what}: zero-point off a tie"
    d = (q_gpu - np.repeat(z_gpu, group, axis=1).astype(np.int64)) - (q_ref - np.repeat(z_ref, group, axis=1).astype(np.int64))
    mism = d != 0
    if mism.any():
        assert np.all(np.abs(d[mism]) <= 1), f"{what}: a code differs by more than 1"
        at_end = (q_gpu == 0) | (q_gpu == 15) | (q_ref == 0) | (q_ref == 15)
        allowed = near(ratio) | (np.repeat(zd, group, axis=1) & at_end)
        assert np.all(allowed[mism]), f"{what}: code mismatch away from a rounding tie"
        assert mism.sum() <= max(1, MAX_MISMATCH_FRACTION * mism.size), f"{what}: {mism.sum()} codes differ"
    return int(mism.sum())


def group_terms(P, s, z, R, s_w):
    """Magnitudes the per-group fp32 chain adds up: s_w sum_j |s_j| (|P_j| + |z_j R_j|)."""
    acc = np.zeros(P.shape[1:])
    for j in range(P.shape[0]):
        acc += np.abs(s[:, j, None]) * (np.abs(P[j]) + np.abs(z[:, j, None] * R[j][None, :]))
    return np.abs(np.asarray(s_w, np.float64))[None, :] * acc
