"""Plain CPU oracle for the OffQ W4A4 linear path (test infrastructure).

This is test infrastructure, not the product. Only ``tests/``,
``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py`` may import
it. It shares no code with the CUDA path: it builds the Hadamard matrix
explicitly, rotates with a dense float64 matmul, takes offsets as plain block
means, and computes the integer GEMM exactly.

Every function follows the paper (OffQ, arxiv 2606.07116) and cites the passage
it implements. Where the paper is silent, it uses these readings:

* Rounding of Eq. 1's round operator: round half to even (``numpy.rint``).
* Residual quantizer: symmetric signed 4-bit with one scale per token,
  s = max|R| / 7, codes clamped to [-7, 7] (the sign-magnitude 4-bit range),
  s = 0 and all codes 0 for an all-zero residual row.
* Offset of block b: the mean of the rotated block. For the Sylvester Hadamard
  it equals the block's first channel divided by sqrt(g) (Sec. 3.2, Eq. 4-5).
* Online rotation: the Sylvester Hadamard in natural order (first row all ones,
  Sec. 3.2), applied block-diagonally with block size g (group-wise offsetting,
  Sec. 3.2 "Group-Wise Offsetting"), normalised by 1/sqrt(g).
* Weights: per-output-channel symmetric round-to-nearest (Sec. 4 settings; GPTQ
  needs calibration data), after the same block rotation so that
  W x = (W H)(H x) for the orthonormal, symmetric block Hadamard H.
* Offset correction table: R[b, n] = sum_{k in b} Qw[n, k], the quantized
  weights' integer block row sums, so the epilogue
  y = s_a s_w acc + s_w sum_b o_b R[b, n] reproduces W_hat @ X_hat exactly
  (Sec. 3.2, Eq. 5: the offset is a constant added to every channel of a
  block, so it leaves through the weight row sums).
* Packing of activation codes: Eq. 1's unsigned form with zero-point 8 (nibble
  q + 8), two per byte, even channel low. Weight codes: sign-magnitude nibbles
  interleaved per 8 channels (layout in :func:`pack_weight_codes`).
* The per-group asymmetric activation path (the paper's evaluated setting)
  has its own readings, listed with :func:`quantize_groups_asym`.

Decisions that turn floating point into integers (the codes) are taken here in
float64.
"""

from __future__ import annotations

import functools
import math
from typing import Dict, Optional

import numpy as np

QMAX = 7  # largest code magnitude of the symmetric 4-bit grid (Eq. 1 with b = 4, z absent)


# ---------------------------------------------------------------------------
# Hadamard matrix and the online rotation  (Sec. 3.2, Eq. 4)
# ---------------------------------------------------------------------------

@functools.lru_cache(maxsize=4)
def _sylvester_cached(g: int) -> np.ndarray:
    h = np.ones((1, 1), dtype=np.int64)
    while h.shape[0] < g:
        h = np.block([[h, h], [h, -h]])
    h.setflags(write=False)
    return h


@functools.lru_cache(maxsize=4)
def _hadamard_f64(g: int) -> np.ndarray:
    h = _sylvester_cached(g).astype(np.float64)
    h.setflags(write=False)
    return h


def sylvester_hadamard(g: int) -> np.ndarray:
    """Sylvester Hadamard H_g (int64, entries +-1), H_1 = [1], H_2m = [[H, H], [H, -H]].

    The paper needs an orthogonal matrix with +-1 entries whose first row is all
    ones (Sec. 3.2, "Offsetting Technique"); the Sylvester recursion gives one
    for every power of two.
    """
    if g < 1 or (g & (g - 1)) != 0:
        raise ValueError("g must be a power of two")
    return _sylvester_cached(g).copy()


def rotate_blocks(x: np.ndarray, g: int) -> np.ndarray:
    """Y = X @ blockdiag(H_g, ..., H_g) / sqrt(g) for token rows X [T, K] (Eq. 4, group-wise).

    Written as a dense float64 matmul per block of g channels: the definition,
    not a butterfly.
    """
    x = np.asarray(x, dtype=np.float64)
    T, K = x.shape
    if K % g != 0:
        raise ValueError("g must divide K")
    H = _hadamard_f64(g)  # the Sylvester matrix of sylvester_hadamard, as float64
    y = np.empty_like(x)
    for b in range(K // g):
        sl = slice(b * g, (b + 1) * g)
        y[:, sl] = x[:, sl] @ H / math.sqrt(g)
    return y


def block_offsets(y: np.ndarray, g: int) -> np.ndarray:
    """o[t, b] = mean of Y[t, b*g:(b+1)*g]: the constant each block carries (Sec. 3.2, Eq. 5).

    Each block sum is the correctly rounded sum (``math.fsum``), so the mean is
    exact whenever it is representable.
    """
    y = np.asarray(y, dtype=np.float64)
    T, K = y.shape
    blocks = y.reshape(T * (K // g), g)
    sums = np.fromiter((math.fsum(row) for row in blocks), dtype=np.float64, count=blocks.shape[0])
    return (sums / g).reshape(T, K // g)


def subtract_offsets(y: np.ndarray, o: np.ndarray, g: int) -> np.ndarray:
    """Residual R = Y - o broadcast over each block (the part left after offsetting, Eq. 5)."""
    T, K = y.shape
    return (y.reshape(T, K // g, g) - o[:, :, None]).reshape(T, K)


# ---------------------------------------------------------------------------
# Uniform quantizer  (Sec. 3, Eq. 1)
# ---------------------------------------------------------------------------

def quantize_rows(r: np.ndarray):
    """Symmetric per-row 4-bit quantization of Eq. 1 (no zero-point).

    s[t] = max_k |r[t, k]| / 7;  q = clamp(round_half_even(r / s), -7, 7);
    a row of zeros gets s = 0 and q = 0. Returns (q int64, s float64).
    """
    r = np.asarray(r, dtype=np.float64)
    amax = np.max(np.abs(r), axis=1) if r.shape[1] > 0 else np.zeros(r.shape[0])
    s = amax / QMAX
    q = np.zeros(r.shape, dtype=np.int64)
    nz = s > 0
    q[nz] = np.clip(np.rint(r[nz] / s[nz, None]), -QMAX, QMAX).astype(np.int64)
    return q, s


def pack_act_codes(q: np.ndarray) -> np.ndarray:
    """Activation codes [.., K] -> bytes [.., K/2] in Eq. 1's unsigned form.

    Eq. 1 stores x_q = round(x / s) + z in [0, 2^b - 1]; with b = 4 and the
    zero-point z = 8 a symmetric code q in [-7, 7] becomes the nibble q + 8.
    Two nibbles per byte, the even channel in the low nibble.
    """
    q = np.asarray(q, dtype=np.int64)
    if q.shape[-1] % 2:
        raise ValueError("K must be even")
    if np.any(np.abs(q) > QMAX):
        raise ValueError("code out of range")
    u = (q + 8).astype(np.uint8)
    return (u[..., 0::2] | (u[..., 1::2] << 4)).astype(np.uint8)


def unpack_act_codes(packed: np.ndarray) -> np.ndarray:
    """Inverse of :func:`pack_act_codes`."""
    p = np.asarray(packed, dtype=np.uint8).astype(np.int64)
    out = np.empty(p.shape[:-1] + (2 * p.shape[-1],), dtype=np.int64)
    out[..., 0::2] = (p & 0xF) - 8
    out[..., 1::2] = (p >> 4) - 8
    return out


def pack_weight_codes(q: np.ndarray) -> np.ndarray:
    """Weight codes [.., K] -> bytes [.., K/2], sign-magnitude, interleaved by 8.

    Each group of 8 channels c0..c7 occupies 4 bytes B0..B3 with
    Bj bits 0-2 = |q(c_2j)|, bit 7 = sign(q(c_2j)), bits 4-6 = |q(c_2j+1)|,
    bit 3 = sign(q(c_(2j-1) mod 8)); sign = 1 for a negative code.
    """
    q = np.asarray(q, dtype=np.int64)
    if q.shape[-1] % 8:
        raise ValueError("K must be a multiple of 8")
    if np.any(np.abs(q) > QMAX):
        raise ValueError("code out of range")
    lead = q.shape[:-1]
    g8 = q.reshape(lead + (q.shape[-1] // 8, 8))
    mag = np.abs(g8)
    neg = (g8 < 0).astype(np.int64)
    out = np.zeros(lead + (q.shape[-1] // 8, 4), dtype=np.int64)
    for j in range(4):
        out[..., j] = (mag[..., 2 * j] | (neg[..., 2 * j] << 7) | (mag[..., 2 * j + 1] << 4)
                       | (neg[..., (2 * j - 1) % 8] << 3))
    return out.reshape(lead + (q.shape[-1] // 2,)).astype(np.uint8)


def unpack_weight_codes(packed: np.ndarray) -> np.ndarray:
    """Inverse of :func:`pack_weight_codes`."""
    p = np.asarray(packed, dtype=np.uint8).astype(np.int64)
    lead = p.shape[:-1]
    b = p.reshape(lead + (p.shape[-1] // 4, 4))
    q = np.zeros(lead + (p.shape[-1] // 4, 8), dtype=np.int64)
    for j in range(4):
        q[..., 2 * j] = np.where((b[..., j] >> 7) & 1, -1, 1) * (b[..., j] & 7)
        q[..., 2 * j + 1] = ((b[..., j] >> 4) & 7) * np.where((b[..., (j + 1) % 4] >> 3) & 1, -1, 1)
    return q.reshape(lead + (2 * p.shape[-1],))


TILE_ROWS = 32   # rows per tile of the GEMM operand layout
TILE_CODES = 32  # codes (16 bytes) per row of a tile


def tile_codes(packed: np.ndarray) -> np.ndarray:
    """Row-major packed codes [R, K/2] -> the tiled byte order of the GEMM operands.

    Rows are padded with zero bytes to a multiple of 32. The result is the
    array [ceil(R/32), K/32, 32, 16] flattened: tile (rb, c) of 512 bytes holds
    the 16-byte chunk c (codes 32c .. 32c+31) of rows 32 rb .. 32 rb + 31, one
    row after the other. Byte (r, j) of the row-major input lands at
    ((r // 32) * (K // 32) + j // 16) * 512 + (r % 32) * 16 + j % 16.
    """
    p = np.asarray(packed, dtype=np.uint8)
    R, KB = p.shape
    if KB % 16:
        raise ValueError("K must be a multiple of 32")
    Rp = -(-R // TILE_ROWS) * TILE_ROWS
    q = np.zeros((Rp, KB), dtype=np.uint8)
    q[:R] = p
    return q.reshape(Rp // TILE_ROWS, TILE_ROWS, KB // 16, 16).transpose(0, 2, 1, 3).reshape(-1).copy()


def untile_codes(tiled: np.ndarray, R: int, K: int) -> np.ndarray:
    """Inverse of :func:`tile_codes`: the first R rows as row-major [R, K/2]."""
    t = np.asarray(tiled, dtype=np.uint8).reshape(-1)
    Rp = -(-R // TILE_ROWS) * TILE_ROWS
    KB = K // 2
    return t[:Rp * KB].reshape(Rp // TILE_ROWS, KB // 16, TILE_ROWS, 16).transpose(0, 2, 1, 3).reshape(Rp, KB)[:R].copy()


# ---------------------------------------------------------------------------
# Online activation path  (Sec. 3.2 offsetting + Sec. 3 Eq. 1)
# ---------------------------------------------------------------------------

def quantize_act(x: np.ndarray, g: int, rotate: bool = True, offset: bool = True) -> Dict[str, np.ndarray]:
    """Rotate -> offset -> quantize -> pack one batch of token rows X [T, K].

    Steps, in the paper's order:
      1. Y = X H / sqrt(g) block-wise when ``rotate`` (Eq. 4); else Y = X.
      2. o[t, b] = mean of block b of Y when ``offset`` (Eq. 5); else o = 0.
      3. R = Y - o.
      4. s[t] = max|R[t]| / 7, q = clamp(rne(R / s), -7, 7) (Eq. 1, symmetric).
      5. Two codes per byte.

    The product X H and its block means are formed before the 1/sqrt(g)
    normalisation. For bf16/fp32 inputs of moderate range that keeps them exact
    in float64, so a block holding only its leading (outlier) channel leaves a
    residual of exactly zero, as the paper states (Eq. 5). R / s equals
    7 R_u / max|R_u| for the unnormalised residual R_u = sqrt(g) R, so the codes
    are taken from R_u directly.
    """
    x = np.asarray(x, dtype=np.float64)
    T, K = x.shape
    if K % g != 0:
        raise ValueError("g must divide K")
    G = K // g
    if rotate:
        H = _hadamard_f64(g)  # the Sylvester matrix of sylvester_hadamard, as float64
        yu = np.empty_like(x)
        for b in range(G):
            sl = slice(b * g, (b + 1) * g)
            yu[:, sl] = x[:, sl] @ H
        norm = math.sqrt(g)
    else:
        yu = x.copy()
        norm = 1.0
    ou = block_offsets(yu, g) if offset else np.zeros((T, G))
    ru = subtract_offsets(yu, ou, g)
    q, su = quantize_rows(ru)
    return {"y": yu / norm, "offset": ou / norm, "residual": ru / norm, "q": q,
            "scale": su / norm, "codes": pack_act_codes(q)}


def dequantize_act(q: np.ndarray, s: np.ndarray, o: np.ndarray, g: int) -> np.ndarray:
    """X_hat[t, k] = s[t] * q[t, k] + o[t, k // g]: what the 4-bit activation stands for."""
    T, K = q.shape
    xh = q.astype(np.float64) * s[:, None]
    return (xh.reshape(T, K // g, g) + o[:, :, None]).reshape(T, K)


# ---------------------------------------------------------------------------
# Weights (offline)  (Sec. 3.3 Step 2 fusion of the rotation, Sec. 4 settings)
# ---------------------------------------------------------------------------

def prepare_weight(w: np.ndarray, g: int, rotate: bool = True) -> Dict[str, np.ndarray]:
    """Per-output-channel symmetric 4-bit weights for y = W x with W [N, K].

    W_eff = W blockdiag(H_g) / sqrt(g) when the input takes the online rotation
    (Sec. 3.3 Step 2 (4): the inverse rotation is fused into the weight, and the
    block Hadamard is symmetric and orthonormal); s_w[n] = max|W_eff[n]| / 7;
    Qw = clamp(rne(W_eff / s_w), -7, 7); R[b, n] = sum_{k in block b} Qw[n, k] (integers).
    """
    w = np.asarray(w, dtype=np.float64)
    N, K = w.shape
    # Same rotate-then-quantize steps as the activations, with no offset.
    res = quantize_act(w, g, rotate=rotate, offset=False)
    w_eff, qw, sw = res["y"], res["q"], res["scale"]
    G = K // g
    rowsum = qw.reshape(N, G, g).sum(axis=2).T        # int64 [G, N]
    return {"w_eff": w_eff, "q": qw, "scale": sw, "offsum": rowsum.astype(np.float64),
            "rowsum": rowsum, "codes": pack_weight_codes(qw)}


# ---------------------------------------------------------------------------
# W4A4 GEMM and epilogue
# ---------------------------------------------------------------------------

def int_gemm(qa: np.ndarray, qw: np.ndarray) -> np.ndarray:
    """acc[t, n] = sum_k qa[t, k] * qw[n, k] exactly, as int64.

    A float64 BLAS product on integer-valued arrays is exact here: every partial
    sum is an integer of magnitude <= 49 * K < 2**53.
    """
    qa = np.asarray(qa, dtype=np.int64)
    qw = np.asarray(qw, dtype=np.int64)
    if 49 * qa.shape[1] >= 2 ** 53:
        raise ValueError("K too large for an exact float64 product")
    acc = qa.astype(np.float64) @ qw.astype(np.float64).T
    return np.rint(acc).astype(np.int64)


def int_gemm_loops(qa: np.ndarray, qw: np.ndarray) -> np.ndarray:
    """Triple-loop int64 GEMM for tiny shapes (a cross-check of :func:`int_gemm`)."""
    T, K = qa.shape
    N = qw.shape[0]
    acc = np.zeros((T, N), dtype=np.int64)
    for t in range(T):
        for n in range(N):
            a = 0
            for k in range(K):
                a += int(qa[t, k]) * int(qw[n, k])
            acc[t, n] = a
    return acc


def epilogue(acc: np.ndarray, s_a: np.ndarray, o: np.ndarray, s_w: np.ndarray,
             R: np.ndarray) -> np.ndarray:
    """y[t, n] = s_a[t] s_w[n] acc[t, n] + s_w[n] sum_b o[t, b] R[b, n], in float64.

    The second term is the offset's rank-G correction: each block's constant
    offset meets the block row sums of the dequantized weights.
    """
    s_w = np.asarray(s_w, np.float64)[None, :]
    return (np.asarray(s_a, np.float64)[:, None] * s_w * np.asarray(acc, np.float64)
            + s_w * (np.asarray(o, np.float64) @ np.asarray(R, np.float64)))


def w4a4_linear(qa: np.ndarray, s_a: np.ndarray, o: np.ndarray, qw: np.ndarray,
                s_w: np.ndarray, R: np.ndarray) -> Dict[str, np.ndarray]:
    """Integer GEMM of the codes plus the dequant + offset epilogue."""
    acc = int_gemm(qa, qw)
    return {"acc": acc, "y": epilogue(acc, s_a, o, s_w, R)}


def linear_reference(x: np.ndarray, w: np.ndarray) -> np.ndarray:
    """Unquantized y = X W^T in float64 (for the quality report, not parity)."""
    return np.asarray(x, np.float64) @ np.asarray(w, np.float64).T


# ---------------------------------------------------------------------------
# KV-cache 4-bit quantization  (Sec. 3.3 Step 2 (2)-(3): per-head H3, KV group = head dim)
# ---------------------------------------------------------------------------

def kv4_quantize(kv: np.ndarray, rotate: bool = True, offset: bool = True) -> Dict[str, np.ndarray]:
    """Per-(token, head) rotate/offset/quantize of KV vectors [T, H, hd] with g = hd.

    The head is one block: the per-head online Hadamard H3 of the keys
    (Sec. 3.3 Step 2 (3)), one offset and one scale per (token, head).
    """
    kv = np.asarray(kv, dtype=np.float64)
    T, H, hd = kv.shape
    res = quantize_act(kv.reshape(T * H, hd), hd, rotate=rotate, offset=offset)
    return {"q": res["q"].reshape(T, H, hd), "scale": res["scale"].reshape(T, H),
            "offset": res["offset"].reshape(T, H), "codes": res["codes"].reshape(T, H, hd // 2),
            "residual": res["residual"].reshape(T, H, hd)}


# ---------------------------------------------------------------------------
# Key cache with a dense per-head rotation  (Sec. 3.3 Step 2 (3): U3 P3 H3)
# ---------------------------------------------------------------------------
#
# With bias-induced outliers in the keys, the per-head online Hadamard H3 is
# replaced by M = U3 P3 H3: a per-head top-1 PCA rotation U3, a permutation
# P3 and H3 (Sec. 3.3 Step 1 (2), Step 2 (3)). It is applied to the
# RoPE-encoded outputs of W_Q and W_K, so Q K^T is unchanged (M orthonormal),
# and the key cache is quantized per (token, head) as before: M's last factor
# has an all-ones first row, so the concentrated outlier leaves as the head's
# constant offset (Eq. 5).


def rotate_heads(x: np.ndarray, rot: np.ndarray) -> np.ndarray:
    """y[t, h, :] = x[t, h, :] @ rot[h] for x [T, H, hd] and rot [H, hd, hd], float64."""
    x = np.asarray(x, np.float64)
    rot = np.asarray(rot, np.float64)
    return np.einsum("thi,hij->thj", x, rot)


def kv4_quantize_dense(kv: np.ndarray, rot: np.ndarray, offset: bool = True) -> Dict[str, np.ndarray]:
    """Per-(token, head) 4-bit keys after the dense rotation: offset = mean of the
    rotated head (Eq. 5), symmetric scale max|r| / 7, q = clamp(rne(r / s), -7, 7)."""
    y = rotate_heads(kv, rot)
    T, H, hd = y.shape
    flat = y.reshape(T * H, hd)
    o = np.array([math.fsum(r) / hd for r in flat]) if offset else np.zeros(T * H)
    r = flat - o[:, None]
    q, s = quantize_rows(r)
    return {"y": y, "q": q.reshape(T, H, hd), "scale": s.reshape(T, H), "offset": o.reshape(T, H),
            "residual": r.reshape(T, H, hd), "codes": pack_act_codes(q).reshape(T, H, hd // 2)}


def householder_to_first(v: np.ndarray) -> np.ndarray:
    """Symmetric orthonormal U with U e_1 = v / |v| (a reflection): a row vector k
    rotated as k U carries k . v / |v| in channel 0, the role of U3's top-1 PCA
    direction (Sec. 3.3 Step 1 (2))."""
    v = np.asarray(v, np.float64)
    v = v / np.linalg.norm(v)
    e = np.zeros_like(v)
    e[0] = 1.0
    w = v - e
    nw = np.dot(w, w)
    if nw < 1e-30:
        return np.eye(len(v))
    return np.eye(len(v)) - 2.0 * np.outer(w, w) / nw


def top1_pca_direction(x: np.ndarray) -> np.ndarray:
    """Leading right singular vector of the (uncentred) rows of x: the top-1 PCA
    direction of Sec. 3.3 Step 1, sign fixed so its largest entry is positive."""
    _, _, vt = np.linalg.svd(np.asarray(x, np.float64), full_matrices=False)
    v = vt[0]
    return v if v[np.argmax(np.abs(v))] > 0 else -v


def key_rotation(keys: np.ndarray, perm: Optional[np.ndarray] = None) -> np.ndarray:
    """Per-head M = U3 P3 H3 from key samples [T, H, hd]: U3 the reflection taking
    channel 0 to the head's top-1 PCA direction, P3 the permutation ``perm``
    (new channel c takes old channel perm[c]; identity by default), H3 the
    normalised Sylvester Hadamard. Returns [H, hd, hd].

    P3 keeps channel 0 first: the concentrated channel must stay block-leading
    to meet the Hadamard's all-ones first row and leave as the offset (Eq. 5,
    group-wise offsetting of Sec. 3.2)."""
    keys = np.asarray(keys, np.float64)
    T, H, hd = keys.shape
    if perm is not None and perm[0] != 0:
        raise ValueError("P3 must keep the concentrated channel 0 first")
    Hs = _hadamard_f64(hd) / math.sqrt(hd)
    P = np.eye(hd)[:, perm] if perm is not None else np.eye(hd)
    out = np.empty((H, hd, hd))
    for h in range(H):
        U = householder_to_first(top1_pca_direction(keys[:, h, :]))
        out[h] = U @ P @ Hs
    return out


# ---------------------------------------------------------------------------
# Offline transform builder  (Sec. 3.1 top-1 PCA; Sec. 3.2 group-wise
# offsetting; Sec. 3.3 Steps 1-2)
# ---------------------------------------------------------------------------
#
# From calibration activations [S sequences, L tokens, D channels]:
#   1. per sequence, the token with the largest L-infinity norm (Sec. 3.1,
#      "top-1"): X [S, D];
#   2. the leading eigenvector v of C = X^T X / S (Eq. 6);
#   3. U1: the reflection with U1 e_1 = v, so x U1 carries x . v in channel 0
#      (the paper's full eigenvector matrix is read as any orthonormal U1
#      whose first column is v: only the leading direction is concentrated);
#   4. P1: sorted grouping of the channels of X U1 by their absolute maxima
#      (Sec. 3.2): the G largest lead the G groups in descending order, the
#      rest fill the groups in ascending order;
#   5. the block Hadamard H1 of size g = D / G; the weights become W U1 P1 H1
#      (Sec. 3.3 Step 2 (1)), so W x = (W M)(x M)^T for M = U1 P1 H1.


def top1_tokens(x: np.ndarray):
    """Per sequence of x [S, L, D], the token of largest max_d |x| (first on
    ties). Returns (index [S] int64, rows [S, D] float64)."""
    x = np.asarray(x, np.float64)
    linf = np.max(np.abs(x), axis=2)
    idx = np.argmax(linf, axis=1)
    return idx, x[np.arange(x.shape[0]), idx]


def top1_pca(X: np.ndarray):
    """Leading eigenpair of C = X^T X / N by a symmetric eigensolver; the
    eigenvector's sign makes its largest-magnitude entry positive."""
    X = np.asarray(X, np.float64)
    C = X.T @ X / X.shape[0]
    lam, U = np.linalg.eigh(C)
    v = U[:, -1]
    if v[np.argmax(np.abs(v))] < 0:
        v = -v
    return v, lam[-1], lam[-2] if len(lam) > 1 else 0.0


def sorted_grouping(mag: np.ndarray, G: int) -> np.ndarray:
    """Permutation of D channels into G groups of D / G (Sec. 3.2): the G
    largest |mag| lead the groups (largest first), the remaining channels fill
    the groups in ascending order of |mag|. New channel c takes old channel
    perm[c]; ties keep channel order."""
    mag = np.abs(np.asarray(mag, np.float64))
    D = len(mag)
    if D % G:
        raise ValueError("G must divide D")
    order = np.argsort(-mag, kind="stable")
    leaders, rest = order[:G], order[G:]
    rest = rest[np.argsort(mag[rest], kind="stable")]
    size = D // G
    perm = np.empty(D, dtype=np.int64)
    for gi in range(G):
        perm[gi * size] = leaders[gi]
        perm[gi * size + 1:(gi + 1) * size] = rest[gi * (size - 1):(gi + 1) * (size - 1)]
    return perm


def offset_basis(v: np.ndarray, perm: np.ndarray, g: int) -> np.ndarray:
    """M = U1 P1 blockdiag(H_g) / sqrt(g) as a dense [D, D] matrix."""
    D = len(v)
    U = householder_to_first(v)
    P = np.eye(D)[:, perm]
    Hb = np.zeros((D, D))
    Hs = _hadamard_f64(g) / math.sqrt(g)
    for b in range(D // g):
        Hb[b * g:(b + 1) * g, b * g:(b + 1) * g] = Hs
    return U @ P @ Hb


def build_offset_transform(x: np.ndarray, G: int) -> Dict[str, np.ndarray]:
    """Steps 1-5 on calibration activations x [S, L, D]."""
    idx, X = top1_tokens(x)
    v, lam1, lam2 = top1_pca(X)
    Xr = X @ householder_to_first(v)
    perm = sorted_grouping(np.max(np.abs(Xr), axis=0), G)
    D = x.shape[2]
    return {"index": idx, "X": X, "v": v, "lam1": lam1, "lam2": lam2, "perm": perm,
            "M": offset_basis(v, perm, D // G)}


def fuse_rotation(w: np.ndarray, M: np.ndarray) -> np.ndarray:
    """W M: the weight that meets activations rotated as x M (Sec. 3.3 Step 2 (1))."""
    return np.asarray(w, np.float64) @ np.asarray(M, np.float64)


# ---------------------------------------------------------------------------
# Per-group asymmetric activations  (Sec. 3 Eq. 1 with its zero-point; Sec. 3.2
# footnote at Eq. 5; Sec. 4 settings: groups of 128 activations)
# ---------------------------------------------------------------------------
#
# The paper's evaluated activation quantizer. Eq. 1 with the zero-point z is
# applied to every group of GROUP consecutive channels of a (rotated) token
# row. After the Hadamard rotation the outlier is a constant offset over a
# whole block (Eq. 5); a zero-point absorbs it because the grid need not hold
# 0 (Sec. 3.2 footnote), so this path keeps no explicit offset. Readings:
#
# * s = (max - min) / 15 over the group (the 2^b - 1 steps of Eq. 1's range
#   [0, 2^b - 1] span the group's range); z = -rne(min / s), any integer
#   (0 need not lie in the range); q = clamp(rne(y / s) + z, 0, 15).
# * A constant group (max == min) gets s = 0, z = 0 and q = 0.
# * Storage: s and z in float32 (z integer-valued); the paper's 16-bit storage
#   (Sec. 3.4) is an accounting choice left out here.
# * Codes: the unsigned 4-bit q is the nibble itself, two per byte, even
#   channel low (the layout of :func:`pack_act_codes`).
# * Weights: the per-channel symmetric codes of :func:`prepare_weight` (Sec. 4
#   settings), with integer row sums per activation group.

GROUP = 128  # activation group size of the evaluated setting (Sec. 4)
UMAX = 15    # largest code of Eq. 1's unsigned grid for b = 4


def quantize_groups_asym(y: np.ndarray, group: int):
    """Eq. 1 with a zero-point for every group of ``group`` channels of each row.

    Returns q (int64 [T, K], in [0, 15]), s (float64 [T, K/group]) and z
    (float64, integer-valued, [T, K/group]). The decisions are taken in
    float64: z = -rne(min / s) and q = clamp(rne(y / s) + z, 0, 15).

    The ratio y / s of Eq. 1, with s = (max - min) / 15, is the real number
    15 y / (max - min); it is evaluated in that form, so s is not rounded
    before the division. For values of bf16, f16 or f32 inputs (and their
    float64 Hadamard transforms) 15 y and max - min are exact in float64, so a
    ratio that is exactly a half-integer is seen as one and rounds half to
    even. Such ties are frequent: on a bf16 grid max - min and y share few
    significant bits.
    """
    y = np.asarray(y, dtype=np.float64)
    T, K = y.shape
    if K % group != 0:
        raise ValueError("group must divide K")
    yg = y.reshape(T, K // group, group)
    mn, mx = yg.min(axis=2), yg.max(axis=2)
    rng = mx - mn
    s = rng / UMAX
    z = np.zeros_like(s)
    q = np.zeros(yg.shape, dtype=np.int64)
    nz = rng > 0
    z[nz] = -np.rint(UMAX * mn[nz] / rng[nz])
    q[nz] = np.clip(np.rint(UMAX * yg[nz] / rng[nz][:, None]) + z[nz][:, None], 0, UMAX).astype(np.int64)
    return q.reshape(T, K), s, z


def pack_unsigned_codes(q: np.ndarray) -> np.ndarray:
    """Unsigned codes in [0, 15] -> nibbles, two per byte, even channel low."""
    q = np.asarray(q, dtype=np.int64)
    if np.any((q < 0) | (q > UMAX)):
        raise ValueError("code out of range")
    if q.shape[-1] % 2:
        raise ValueError("K must be even")
    u = q.astype(np.uint8)
    return (u[..., 0::2] | (u[..., 1::2] << 4)).astype(np.uint8)


def quantize_act_group(x: np.ndarray, g: int, group: int = GROUP, rotate: bool = True) -> Dict[str, np.ndarray]:
    """Rotate -> per-group asymmetric quantize -> pack one batch of token rows X [T, K].

    Steps, in the paper's order:
      1. Y = X H / sqrt(g) block-wise when ``rotate`` (Eq. 4); else Y = X.
      2. Per group of ``group`` channels: s, z, q of Eq. 1 (readings above).
      3. Two codes per byte.

    As in :func:`quantize_act`, the codes are taken from the unnormalised
    product X H (y / s is the same ratio), so the decisions see no 1/sqrt(g)
    rounding.
    """
    x = np.asarray(x, dtype=np.float64)
    T, K = x.shape
    if K % g != 0 or K % group != 0:
        raise ValueError("g and group must divide K")
    if rotate:
        H = _hadamard_f64(g)
        yu = np.empty_like(x)
        for b in range(K // g):
            sl = slice(b * g, (b + 1) * g)
            yu[:, sl] = x[:, sl] @ H
        norm = math.sqrt(g)
    else:
        yu = x.copy()
        norm = 1.0
    q, su, z = quantize_groups_asym(yu, group)
    return {"y": yu / norm, "q": q, "scale": su / norm, "zero": z, "codes": pack_unsigned_codes(q)}


def dequantize_act_group(q: np.ndarray, s: np.ndarray, z: np.ndarray, group: int) -> np.ndarray:
    """X_hat[t, k] = s[t, k // group] * (q[t, k] - z[t, k // group]) (Eq. 1 inverted)."""
    T, K = q.shape
    qg = np.asarray(q, np.float64).reshape(T, K // group, group)
    return (np.asarray(s, np.float64)[:, :, None] * (qg - np.asarray(z, np.float64)[:, :, None])).reshape(T, K)


def weight_group_sums(qw: np.ndarray, group: int) -> np.ndarray:
    """R[j, n] = sum_{k in group j} Qw[n, k]: integer row sums per activation group."""
    qw = np.asarray(qw, dtype=np.int64)
    N, K = qw.shape
    return qw.reshape(N, K // group, group).sum(axis=2).T


def w4a4_linear_group(q: np.ndarray, s: np.ndarray, z: np.ndarray, qw: np.ndarray, s_w: np.ndarray,
                      R: np.ndarray, group: int) -> Dict[str, np.ndarray]:
    """y[t, n] = s_w[n] sum_j s[t, j] (P_j[t, n] - z[t, j] R[j, n]), in float64.

    P_j = sum_{k in group j} q[t, k] Qw[n, k] is each group's exact integer
    product; subtracting z R removes the zero-point (Eq. 1 inverted), and the
    per-group scale leaves the sum over groups as floating point.
    """
    q = np.asarray(q, np.int64)
    qw = np.asarray(qw, np.int64)
    T, K = q.shape
    G = K // group
    P = np.stack([int_gemm(q[:, j * group:(j + 1) * group], qw[:, j * group:(j + 1) * group]) for j in range(G)])
    s = np.asarray(s, np.float64)
    z = np.asarray(z, np.float64)
    acc = np.zeros((T, qw.shape[0]))
    for j in range(G):
        acc += s[:, j, None] * (P[j].astype(np.float64) - z[:, j, None] * np.asarray(R, np.float64)[j][None, :])
    return {"P": P, "y": np.asarray(s_w, np.float64)[None, :] * acc}


# ---------------------------------------------------------------------------
# Storage accounting  (Sec. 3.4 "Efficiency of Per-Group Activation Quantization")
# ---------------------------------------------------------------------------

def effective_bits(group: int, code_bits: int = 4, param_bits: int = 16, n_params: int = 2) -> float:
    """Bits per activation when each group of ``group`` codes stores ``n_params`` parameters."""
    return (code_bits * group + param_bits * n_params) / group


def effective_bits_per_token_offset(K: int, g: int, code_bits: int = 4, param_bits: int = 32) -> float:
    """Bits per activation of this path's layout: one scale per token and one offset per block."""
    return (code_bits * K + param_bits * (1 + K // g)) / K


# ---------------------------------------------------------------------------
# MXFP4 activations and weights with the offset as zero-point
# (Sec. 3.4 "Generality on Data Formats": micro-scaling formats extended with
# a zero-point absorb the outlier the same way; the paper leaves it to future
# work, so the readings below are this implementation's own)
# ---------------------------------------------------------------------------
#
# Element format: MXFP4's E2M1 (OCP Microscaling Formats v1.0): sign, 2-bit
# exponent, 1-bit mantissa; magnitudes 0, 0.5, 1, 1.5, 2, 3, 4, 6 for the
# 3-bit codes 0..7, the sign in bit 3 of the nibble.
# Readings:
# * Zero-point: the offsetting block's offset (Eq. 5), one per block of g
#   channels as in the main path, subtracted before the micro-scaled residual is
#   quantized; it leaves through the weights' dequantized block sums.
# * Scale: one power of two 2^X per 32 consecutive channels of a row (MXFP4's
#   shared exponent), X = floor(log2(amax)) - 2, so that amax / 2^X lies in
#   [4, 8); values round to the nearest E2M1 magnitude, ties to the even
#   mantissa, and saturate at 6.
# * Span: within a row no block exponent is more than 6 below the row's
#   largest one (X = max(X, Xmax - 6); an all-zero block takes Xmax - 6). Every
#   code times its block's power of two relative to 2^(Xmax - 6) is then an exact
#   E4M3 value (at most 6 * 2^6 = 384), the form the GEMM multiplies in.

MX_BLOCK = 32
MX_SPAN = 6
E2M1_MAG = np.array([0.0, 0.5, 1.0, 1.5, 2.0, 3.0, 4.0, 6.0])


def e2m1_value(code: np.ndarray) -> np.ndarray:
    """Value of 4-bit E2M1 codes (sign in bit 3, magnitude code in bits 0-2)."""
    code = np.asarray(code, dtype=np.int64)
    return np.where(code & 8, -1.0, 1.0) * E2M1_MAG[code & 7]


def rne_e2m1(v: np.ndarray) -> np.ndarray:
    """Nearest E2M1 code of each value, ties to the even mantissa (magnitude code
    with bit 0 clear), magnitudes above 6 saturating to 6. Returns int64 codes."""
    v = np.asarray(v, dtype=np.float64)
    a = np.abs(v)
    d = np.abs(a[..., None] - E2M1_MAG)              # distance to each magnitude
    best = d.min(axis=-1, keepdims=True)
    cand = d <= best                                 # nearest magnitudes (two at a tie)
    even = cand & (np.arange(8) % 2 == 0)
    pick = np.where(even.any(axis=-1), np.argmax(even, axis=-1), np.argmax(cand, axis=-1))
    pick = np.where(a >= 6.0, 7, pick)
    return np.where((v < 0) & (pick > 0), pick | 8, pick).astype(np.int64)


def mx_block_exponents(r: np.ndarray, block: int = MX_BLOCK, span: int = MX_SPAN):
    """Shared exponents X [T, K/block] of the readings above and the row's Xmax [T]."""
    T, K = r.shape
    amax = np.abs(r.reshape(T, K // block, block)).max(axis=2)
    with np.errstate(divide="ignore"):
        X = np.where(amax > 0, np.floor(np.log2(np.where(amax > 0, amax, 1.0))) - 2, -np.inf)
    xmax = X.max(axis=1)
    xmax = np.where(np.isfinite(xmax), xmax, 0.0)     # an all-zero row: any exponent
    X = np.maximum(X, xmax[:, None] - span)
    return X.astype(np.int64), xmax.astype(np.int64)


def quantize_mx_rows(r: np.ndarray, block: int = MX_BLOCK, span: int = MX_SPAN) -> Dict[str, np.ndarray]:
    """MXFP4 codes of rows r [T, K] (float64): per block 2^X and E2M1 codes."""
    T, K = r.shape
    X, xmax = mx_block_exponents(r, block, span)
    scale = np.repeat(np.ldexp(1.0, X), block, axis=1)
    codes = rne_e2m1(r / scale)
    return {"code": codes, "X": X, "xmax": xmax, "value": e2m1_value(codes) * scale,
            "shift": X - (xmax[:, None] - span), "row_scale": np.ldexp(1.0, xmax - span)}


def quantize_act_mx(x: np.ndarray, g: int, rotate: bool = True, offset: bool = True) -> Dict[str, np.ndarray]:
    """Rotate -> offset -> MXFP4 residual for token rows X [T, K].

      1. Y = X H / sqrt(g) block-wise when ``rotate`` (Eq. 4).
      2. o[t, b] = mean of block b of Y when ``offset`` (Eq. 5).
      3. R = Y - o, quantized per 32 channels (quantize_mx_rows).
    X_hat = R_hat + o is what the activation stands for.
    """
    x = np.asarray(x, dtype=np.float64)
    T, K = x.shape
    if K % g != 0 or K % MX_BLOCK != 0:
        raise ValueError("g and 32 must divide K")
    G = K // g
    if rotate:
        H = _hadamard_f64(g)
        yu = np.empty_like(x)
        for b in range(G):
            sl = slice(b * g, (b + 1) * g)
            yu[:, sl] = x[:, sl] @ H
        norm = math.sqrt(g)
    else:
        yu = x.copy()
        norm = 1.0
    ou = block_offsets(yu, g) if offset else np.zeros((T, G))
    r = subtract_offsets(yu, ou, g) / norm
    res = quantize_mx_rows(r)
    res.update({"y": yu / norm, "offset": ou / norm, "residual": r})
    return res


def prepare_weight_mx(w: np.ndarray, g: int, rotate: bool = True) -> Dict[str, np.ndarray]:
    """MXFP4 weights W [N, K] per output row (no offset): W_eff = W blockdiag(H_g) / sqrt(g)
    when the input takes the online rotation, then quantize_mx_rows. ``offsum[b, n]`` is the
    block sum of the operand values code * 2^shift (the dequantized weights over the row's
    2^(Xmax - 6)), which the offsets meet in the GEMM."""
    res = quantize_act_mx(w, g, rotate=rotate, offset=False)
    N, K = res["code"].shape
    opv = e2m1_value(res["code"]) * np.repeat(np.ldexp(1.0, res["shift"]), MX_BLOCK, axis=1)
    res["operand"] = opv
    res["offsum"] = opv.reshape(N, K // g, g).sum(axis=2).T
    return res


def mx_linear(a: Dict[str, np.ndarray], w: Dict[str, np.ndarray], g: int) -> Dict[str, np.ndarray]:
    """y = (R_hat + o) W_hat^T in float64, from the codes of quantize_act_mx and
    prepare_weight_mx: the residual product plus the offsets' block-sum term."""
    K = a["code"].shape[1]
    ra = a["value"]
    wv = w["value"]
    T = ra.shape[0]
    o = np.repeat(a["offset"], g, axis=1)
    y = ra @ wv.T + o @ wv.T
    # The same value in the factored form the kernels use.
    opa = e2m1_value(a["code"]) * np.repeat(np.ldexp(1.0, a["shift"]), MX_BLOCK, axis=1)
    acc = opa @ w["operand"].T
    y2 = np.outer(a["row_scale"], w["row_scale"]) * acc + w["row_scale"][None, :] * (a["offset"] @ w["offsum"])
    return {"y": y, "y_factored": y2, "acc": acc}


def pack_mx_codes(code: np.ndarray) -> np.ndarray:
    """E2M1 codes [.., K] (int 0..15) -> bytes [.., K/2], even channel in the low nibble."""
    code = np.asarray(code, dtype=np.int64)
    if np.any((code < 0) | (code > 15)):
        raise ValueError("code out of range")
    u = code.astype(np.uint8)
    return (u[..., 0::2] | (u[..., 1::2] << 4)).astype(np.uint8)


def unpack_mx_codes(packed: np.ndarray) -> np.ndarray:
    p = np.asarray(packed, dtype=np.uint8).astype(np.int64)
    out = np.empty(p.shape[:-1] + (2 * p.shape[-1],), dtype=np.int64)
    out[..., 0::2] = p & 0xF
    out[..., 1::2] = p >> 4
    return out


def tile_mx_shifts(shift: np.ndarray) -> np.ndarray:
    """Block shifts [R, K/32] (0..6) -> the tiled byte layout the GEMM reads: rows padded
    to 32, for 32-row block rb and k-tile kt (4 blocks of 32 channels) the 4 shifts of
    row r at ((rb * (K/128) + kt) * 32 + r % 32) * 4 + (block % 4)."""
    s = np.asarray(shift, dtype=np.int64)
    R, B = s.shape
    if B % 4:
        raise ValueError("K must be a multiple of 128")
    Rp = -(-R // TILE_ROWS) * TILE_ROWS
    t = np.zeros((Rp, B), dtype=np.uint8)
    t[:R] = s.astype(np.uint8)
    return t.reshape(Rp // TILE_ROWS, TILE_ROWS, B // 4, 4).transpose(0, 2, 1, 3).reshape(-1).copy()


def untile_mx_shifts(tiled: np.ndarray, R: int, K: int) -> np.ndarray:
    t = np.asarray(tiled, dtype=np.uint8).reshape(-1)
    Rp = -(-R // TILE_ROWS) * TILE_ROWS
    B = K // MX_BLOCK
    return t[:Rp * B].reshape(Rp // TILE_ROWS, B // 4, TILE_ROWS, 4).transpose(0, 2, 1, 3).reshape(Rp, B)[:R].astype(np.int64)
