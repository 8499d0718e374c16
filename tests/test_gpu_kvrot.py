"""GPU parity of the key cache under a dense per-head rotation M = U3 P3 H3
(offq_kv4_quantize_rotated) and of the query-side rotation (offq_rotate_heads)
against the oracle.

Both sides use the same fp32 matrix M.
* fp32 / fp16 keys: each rotated value is an fp32 chain of head_dim
  multiply-adds in input-channel order, at most (hd + 1) u sum_i |x_i| |M_ij|
  from the float64 value.
* bf16 keys (tensor cores): M is split into three bf16 parts (exact to 2^-24
  relative), every bf16 x bf16 product is exact, and the 3 hd products are
  summed in the tensor core's fp32 accumulator; allowing each addition a full
  ulp (truncation), the bound is (2 * 3 hd + 8) u sum_i |x_i| |M_ij|. The
  offset is then a sequential 128-term fp32 sum in one thread.
The offset and the scale inherit the bound, and a code may differ only where
the oracle's r / s lies within the bound (in code units) of a rounding tie."""

import math

import numpy as np
import pytest
import torch

import oracle as O
from paper_2606_07116_gb300 import build as B
from paper_2606_07116_gb300 import offq as Q
from parity import U32

pytestmark = pytest.mark.gpu

HD = 128


@pytest.fixture(scope="module", autouse=True)
def _lib():
    B.build()
    Q.load_library()


def _keys(T, H, seed, outlier=True):
    rng = np.random.default_rng(seed)
    k = rng.standard_normal((T, H, HD))
    if outlier:
        dirs = rng.standard_normal((H, HD))
        dirs /= np.linalg.norm(dirs, axis=1, keepdims=True)
        k += rng.uniform(20, 80, size=(T, H, 1)) * dirs[None]
    return k


def _rotation(k, seed):
    perm = np.concatenate([[0], 1 + np.random.default_rng(seed).permutation(HD - 1)])
    return O.key_rotation(k, perm).astype(np.float32)


def _bound_y(x, M, tc=False):
    factor = 2 * 3 * HD + 8 if tc else HD + 1
    return factor * U32 * np.einsum("thi,hij->thj", np.abs(x), np.abs(M.astype(np.float64)))


def _check_key_cache(codes, scale, off, x, M, offset=True, tc=False, by=None):
    T, H, _ = x.shape
    ref = O.kv4_quantize_dense(x, M.astype(np.float64), offset=offset)
    if by is None:
        by = _bound_y(x, M, tc).max(axis=2)            # per (t, h)
    y_abs = np.abs(ref["y"]).sum(axis=2)
    bo = by + (HD + 2 if tc else 8) * U32 * y_abs / HD if offset else np.zeros_like(by)
    s_gpu, s_ref = scale.cpu().numpy().astype(np.float64), ref["scale"]
    assert np.all(np.abs(s_gpu - s_ref) <= (by + bo) / 7 + 4 * U32 * s_ref), "scales out of bound"
    if offset:
        o_gpu = off.cpu().numpy().astype(np.float64)
        assert np.all(np.abs(o_gpu - ref["offset"]) <= bo + 1e-30), "offsets out of bound"
    q_gpu = O.unpack_act_codes(codes.cpu().numpy())
    mism = q_gpu != ref["q"]
    if mism.any():
        assert np.all(np.abs(q_gpu - ref["q"])[mism] <= 1)
        with np.errstate(divide="ignore", invalid="ignore"):
            t = np.where(s_ref[..., None] > 0, ref["residual"] / s_ref[..., None], 0.0)
            win = np.where(s_ref > 0, (by + bo) / s_ref, 0.0)[..., None] * 2 + 1e-6
        dist = np.abs(np.abs(t) - np.floor(np.abs(t)) - 0.5)
        assert np.all((dist < np.broadcast_to(win, dist.shape))[mism]), "code mismatch away from a rounding tie"
        assert mism.sum() <= max(1, 1e-4 * mism.size)
    return int(mism.sum())


@pytest.mark.parametrize("dt", [torch.float32, torch.bfloat16, torch.float16])
def test_rotated_key_cache_parity(dt):
    T, H = 300, 8
    k = _keys(T, H, seed=90)
    M = _rotation(k, 91)
    kt = torch.from_numpy(k).to(dt)
    codes, scale, off = Q.kv4_quantize_rotated(kt.cuda(), torch.from_numpy(M).cuda())
    torch.cuda.synchronize()
    assert Q.offq_get_device_status() == Q.OFFQ_OK
    _check_key_cache(codes, scale, off, kt.to(torch.float64).numpy(), M, tc=dt == torch.bfloat16)


def test_rotated_key_cache_ragged_and_strided():
    """One token, 45 tokens (a partial tile), a token stride past the heads, no offset."""
    for T in (1, 45):
        H = 4
        k = _keys(T, H, seed=92 + T)
        M = _rotation(k, 93)
        big = torch.zeros((T, H * HD + 64), dtype=torch.bfloat16)
        big[:, :H * HD] = torch.from_numpy(k.reshape(T, H * HD)).to(torch.bfloat16)
        dev = big.cuda()
        codes = torch.empty((T, H, HD // 2), dtype=torch.uint8, device="cuda")
        scale = torch.empty((T, H), dtype=torch.float32, device="cuda")
        Q.offq_kv4_quantize_rotated(dev, T, H, HD, dev.stride(0), torch.from_numpy(M).cuda(), 0, codes, scale, None)
        torch.cuda.synchronize()
        x = big[:, :H * HD].to(torch.float64).numpy().reshape(T, H, HD)
        _check_key_cache(codes, scale, None, x, M, offset=False, tc=True)


def test_hadamard_matrix_reproduces_h3_path():
    """M = H / sqrt(128) gives the per-head Hadamard key cache (offq_kv4_quantize
    with OFFQ_ROTATE | OFFQ_OFFSET) up to rounding ties."""
    T, H = 64, 4
    k = torch.from_numpy(_keys(T, H, seed=94, outlier=False)).to(torch.bfloat16).cuda()
    Hm = (O.sylvester_hadamard(HD).astype(np.float64) / math.sqrt(HD)).astype(np.float32)
    rot = torch.from_numpy(np.stack([Hm] * H)).cuda()
    c1, s1, o1 = Q.kv4_quantize_rotated(k, rot)
    c2, s2, o2 = Q.kv4_quantize(k, rotate=True, offset=True)
    torch.cuda.synchronize()
    # Both are within their own bounds of the float64 values: the tensor-core
    # product here, the (log2 128 + 2)-stage butterfly there.
    x = k.to(torch.float64).cpu().numpy()
    b_tc = _bound_y(x, rot.cpu().numpy(), tc=True).max(axis=2)
    b_fwht = (7 + 2) * U32 * np.abs(x).sum(axis=2) / math.sqrt(HD)
    s1n, s2n = s1.cpu().numpy().astype(np.float64), s2.cpu().numpy().astype(np.float64)
    assert np.all(np.abs(s1n - s2n) <= 2 * (b_tc + b_fwht) / 7 + 8 * U32 * s2n)
    o_tol = 2 * (b_tc + b_fwht) + (HD + 8) * U32 * np.abs(x).sum(axis=2) / HD
    assert np.all(np.abs(o1.cpu().numpy() - o2.cpu().numpy()) <= o_tol)
    q1, q2 = O.unpack_act_codes(c1.cpu().numpy()), O.unpack_act_codes(c2.cpu().numpy())
    assert np.mean(q1 != q2) < 1e-3 and np.all(np.abs(q1 - q2) <= 1)


@pytest.mark.parametrize("odt", [torch.float32, torch.bfloat16])
def test_rotate_heads_parity_and_scores(odt):
    T, H = 200, 8
    k = _keys(T, H, seed=95)
    q = np.random.default_rng(96).standard_normal((T, H, HD))
    M = _rotation(k, 97)
    qt = torch.from_numpy(q).to(torch.bfloat16)
    y = Q.rotate_heads(qt.cuda(), torch.from_numpy(M).cuda(), out_dtype=odt)
    torch.cuda.synchronize()
    x = qt.to(torch.float64).numpy()
    ref = O.rotate_heads(x, M.astype(np.float64))
    tol = _bound_y(x, M, tc=True) + (2.0 ** -8 * np.abs(ref) if odt == torch.bfloat16 else 0.0)
    err = np.abs(y.float().cpu().numpy().astype(np.float64) - ref)
    assert np.all(err <= tol + 1e-30), f"worst {np.max(err / (tol + 1e-30)):.3g}x the bound"


def test_rotated_key_cache_full_size():
    """The workload's key tensor: 2048 tokens x 32 heads."""
    T, H = 2048, 32
    k = _keys(T, H, seed=98)
    M = _rotation(k, 99)
    kt = torch.from_numpy(k).to(torch.bfloat16)
    codes, scale, off = Q.kv4_quantize_rotated(kt.cuda(), torch.from_numpy(M).cuda())
    torch.cuda.synchronize()
    assert Q.offq_get_device_status() == Q.OFFQ_OK
    _check_key_cache(codes, scale, off, kt.to(torch.float64).numpy(), M, tc=True)


def _bf16_rne(a):
    """float32 -> bf16 (round to nearest even) -> float32, on the host."""
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(torch.bfloat16).float().numpy()


def _decode_prepared(prep, H):
    """The prepared image back to the parts [H][3][k][n] as float32, undoing
    the chunk swizzle: chunk c (k = 8c .. 8c+7) of row n sits in atom column
    c // 8, slot (c % 8) ^ (n % 8) of the row's 128 bytes."""
    u = prep.cpu().numpy().view(np.uint16).reshape(H, 3, 2, HD, 8, 8)
    n = np.arange(HD)[:, None]
    c = np.arange(16)[None, :]
    g = u[:, :, c >> 3, n, (c & 7) ^ (n & 7), :]          # [H, 3, n, c, e]
    parts = g.reshape(H, 3, HD, HD).transpose(0, 1, 3, 2)  # [H, 3, k = 8c + e, n]
    return (parts.astype(np.uint32) << 16).view(np.float32)


def test_prepared_image_is_the_three_part_split():
    H = 3
    k = _keys(16, H, seed=100)
    M = _rotation(k, 101)
    M[2] = (O.sylvester_hadamard(HD) / math.sqrt(HD)).astype(np.float32)
    prep = Q.prepare_key_rotation(torch.from_numpy(M).cuda())
    torch.cuda.synchronize()
    parts = _decode_prepared(prep, H)
    hi = _bf16_rne(M)
    r1 = (M - hi).astype(np.float32)
    mid = _bf16_rne(r1)
    lo = _bf16_rne((r1 - mid).astype(np.float32))
    assert np.array_equal(parts[:, 0], hi) and np.array_equal(parts[:, 1], mid) and np.array_equal(parts[:, 2], lo)
    rebuilt = parts[:, 0].astype(np.float64) + parts[:, 1] + parts[:, 2]
    assert np.all(np.abs(rebuilt - M) <= 2.0 ** -26 * np.abs(M))


@pytest.mark.parametrize("T,H", [(1, 4), (45, 4), (300, 8), (600, 160)])
def test_prepared_key_cache_parity(T, H):
    """The prepared parts give the in-kernel split's outputs bit for bit and
    stay within the tensor-core bound of the oracle. With 160 heads each CTA
    takes all of its head's tiles, so every warpgroup loops over several."""
    k = _keys(T, H, seed=102 + T)
    M = _rotation(k, 103)
    kt = torch.from_numpy(k).to(torch.bfloat16).cuda()
    rot = torch.from_numpy(M).cuda()
    prep = Q.prepare_key_rotation(rot)
    for offset in (True, False):
        c1, s1, o1 = Q.kv4_quantize_prepared(kt, prep, offset=offset)
        c2, s2, o2 = Q.kv4_quantize_rotated(kt, rot, offset=offset)
        torch.cuda.synchronize()
        assert Q.offq_get_device_status() == Q.OFFQ_OK
        assert torch.equal(c1, c2) and torch.equal(s1, s2)
        if offset:
            assert torch.equal(o1, o2)
        _check_key_cache(c1, s1, o1 if offset else None, kt.to(torch.float64).cpu().numpy(), M, offset=offset,
                         tc=True)


@pytest.mark.parametrize("odt", [torch.float32, torch.bfloat16, torch.float16])
def test_rotate_heads_prepared(odt):
    T, H = 333, 160
    q = np.random.default_rng(104).standard_normal((T, H, HD))
    M = _rotation(_keys(8, H, seed=105), 106)
    qt = torch.from_numpy(q).to(torch.bfloat16)
    rot = torch.from_numpy(M).cuda()
    y1 = Q.rotate_heads_prepared(qt.cuda(), Q.prepare_key_rotation(rot), out_dtype=odt)
    y2 = Q.rotate_heads(qt.cuda(), rot, out_dtype=odt)
    torch.cuda.synchronize()
    assert torch.equal(y1, y2)
    if odt == torch.float32:
        x = qt.to(torch.float64).numpy()
        err = np.abs(y1.cpu().numpy().astype(np.float64) - O.rotate_heads(x, M.astype(np.float64)))
        assert np.all(err <= _bound_y(x, M, tc=True) + 1e-30)


def test_prepared_key_cache_full_size():
    """The workload's key tensor, 2048 tokens x 32 heads, through the prepared call."""
    T, H = 2048, 32
    k = _keys(T, H, seed=107)
    M = _rotation(k, 108)
    kt = torch.from_numpy(k).to(torch.bfloat16)
    prep = Q.prepare_key_rotation(torch.from_numpy(M).cuda())
    codes, scale, off = Q.kv4_quantize_prepared(kt.cuda(), prep)
    torch.cuda.synchronize()
    assert Q.offq_get_device_status() == Q.OFFQ_OK
    _check_key_cache(codes, scale, off, kt.to(torch.float64).numpy(), M, tc=True)


# ---------------------------------------------------------------------------
# The structured form M = U3 P3 H3 (offq_prepare_key_reflection and the
# *_reflected calls): y = fma(acc, fp32(1/sqrt(128)), fl(-2 d w'')) with
# acc = sqrt(128) x P3 H3 (exact +-1 products, fp32 sum over 128 terms) and
# d = x . w (exact products with w's three bf16 parts, fp32 sums). With A =
# sum |x_i|, Bw = sum |x_i w_i|, u = x P3 H3, each y_j is within
#   u32 [ (2 hd + 8) A / sqrt(hd) + 2 |u_j| + 2 |w''_j| (2 hd + 12) Bw + 4 |d| |w''_j| + |y_j| ]
# of its float64 value: the accumulations (a full ulp per addition), fp32(1/sqrt(128)),
# fp32(w) and fp32(w''), the product -2 d w''_j and the final fma.
# ---------------------------------------------------------------------------
def _reflection_case(T, H, seed, e0_head=False):
    k = _keys(T, H, seed)
    rng = np.random.default_rng(seed + 1)
    perm = np.stack([np.concatenate([[0], 1 + rng.permutation(HD - 1)]) for _ in range(H)]).astype(np.int32)
    v = np.stack([O.top1_pca_direction(k[:, h, :]) for h in range(H)]).astype(np.float32)
    if e0_head:
        v[0] = 0.0
        v[0, 0] = 1.0                                  # U3 = I for head 0
    Hs = O.sylvester_hadamard(HD).astype(np.float64) / math.sqrt(HD)
    PH = np.stack([np.eye(HD)[:, perm[h]] @ Hs for h in range(H)])
    U = np.stack([O.householder_to_first(v[h].astype(np.float64)) for h in range(H)])
    M = np.einsum("hij,hjk->hik", U, PH)
    return k, v, perm, M, U, PH


def _bound_reflected(x, U, PH):
    T, H, _ = x.shape
    W = np.zeros((H, HD))
    for h in range(H):
        lam, vec = np.linalg.eigh(U[h])               # U = I - 2 w w^T: w is the eigenvector of eigenvalue -1
        if lam[0] < 0:
            W[h] = vec[:, 0]
    w2 = np.einsum("hkn,hk->hn", PH, W)
    A = np.abs(x).sum(axis=2)
    Bw = np.einsum("thi,hi->th", np.abs(x), np.abs(W))
    d = np.einsum("thi,hi->th", x, W)
    u = np.einsum("thi,hij->thj", x, PH)
    y = u - 2 * d[..., None] * w2[None]
    return U32 * ((2 * HD + 8) * A[..., None] / math.sqrt(HD) + 2 * np.abs(u)
                  + 2 * np.abs(w2)[None] * (2 * HD + 12) * Bw[..., None]
                  + 4 * np.abs(d)[..., None] * np.abs(w2)[None] + np.abs(y))


@pytest.mark.parametrize("T,H,e0", [(1, 4, False), (45, 4, True), (300, 8, False), (600, 160, True)])
def test_reflected_key_cache_parity(T, H, e0):
    k, v, perm, M, U, PH = _reflection_case(T, H, seed=110 + T, e0_head=e0)
    kt = torch.from_numpy(k).to(torch.bfloat16)
    x = kt.to(torch.float64).numpy()
    prep = Q.prepare_key_reflection(torch.from_numpy(v), torch.from_numpy(perm), device="cuda")
    by = _bound_reflected(x, U, PH).max(axis=2)
    for offset in (True, False):
        codes, scale, off = Q.kv4_quantize_reflected(kt.cuda(), prep, offset=offset)
        torch.cuda.synchronize()
        assert Q.offq_get_device_status() == Q.OFFQ_OK
        _check_key_cache(codes, scale, off if offset else None, x, M, offset=offset, by=by)


@pytest.mark.parametrize("odt", [torch.float32, torch.bfloat16, torch.float16])
def test_rotate_heads_reflected_parity(odt):
    T, H = 333, 8
    k, v, perm, M, U, PH = _reflection_case(64, H, seed=120)
    q = np.random.default_rng(121).standard_normal((T, H, HD)) * 3.0
    qt = torch.from_numpy(q).to(torch.bfloat16)
    x = qt.to(torch.float64).numpy()
    prep = Q.prepare_key_reflection(torch.from_numpy(v), torch.from_numpy(perm), device="cuda")
    y = Q.rotate_heads_reflected(qt.cuda(), prep, out_dtype=odt)
    torch.cuda.synchronize()
    ref = O.rotate_heads(x, M)
    rnd = {torch.float32: 0.0, torch.bfloat16: 2.0 ** -8, torch.float16: 2.0 ** -11}[odt]
    tol = _bound_reflected(x, U, PH) * (1 + rnd) + rnd * np.abs(ref)
    err = np.abs(y.float().cpu().numpy().astype(np.float64) - ref)
    assert np.all(err <= tol + 1e-30), f"worst {np.max(err / (tol + 1e-30)):.3g}x the bound"


def test_reflected_key_cache_full_size():
    """The workload's key tensor, 2048 tokens x 32 heads, with the structured M."""
    T, H = 2048, 32
    k, v, perm, M, U, PH = _reflection_case(T, H, seed=130)
    kt = torch.from_numpy(k).to(torch.bfloat16)
    x = kt.to(torch.float64).numpy()
    prep = Q.prepare_key_reflection(torch.from_numpy(v), torch.from_numpy(perm), device="cuda")
    codes, scale, off = Q.kv4_quantize_reflected(kt.cuda(), prep)
    torch.cuda.synchronize()
    assert Q.offq_get_device_status() == Q.OFFQ_OK
    _check_key_cache(codes, scale, off, x, M, by=_bound_reflected(x, U, PH).max(axis=2))


@pytest.mark.parametrize("odt", [torch.bfloat16, torch.float16])
def test_rotate_heads_staged_store_ragged_and_padded(odt):
    """16-bit outputs leave by TMA stores of 128-token boxes: one token and 45
    tokens (partial boxes), an output row pitch past the heads whose padding
    must stay untouched, and the same values as the fp32 output rounded once."""
    for T in (1, 45):
        H = 4
        k, v, perm, M, U, PH = _reflection_case(16, H, seed=140 + T)
        x = torch.from_numpy(np.random.default_rng(141 + T).standard_normal((T, H, HD))).to(torch.bfloat16).cuda()
        rot = torch.from_numpy(M.astype(np.float32)).cuda()
        prep = Q.prepare_key_rotation(rot)
        refl = Q.prepare_key_reflection(torch.from_numpy(v), torch.from_numpy(perm), device="cuda")
        ld = H * HD + 72
        for call, img in ((Q.offq_rotate_heads_prepared, prep), (Q.offq_rotate_heads_reflected, refl)):
            out = torch.full((T, ld), 7.0, dtype=odt, device="cuda")
            call(x, T, H, HD, x.stride(0), img, out, ld)
            ref = torch.empty((T, H, HD), dtype=torch.float32, device="cuda")
            call(x, T, H, HD, x.stride(0), img, ref, H * HD)
            torch.cuda.synchronize()
            assert Q.offq_get_device_status() == Q.OFFQ_OK
            assert torch.all(out[:, H * HD:] == 7.0), "padding written"
            assert torch.equal(out[:, :H * HD], ref.reshape(T, H * HD).to(odt))
