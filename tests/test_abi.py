"""The C-ABI library loads, exports every symbol include/offq.h declares, and
rejects bad arguments on the host (no GPU needed: no call here reaches a
CUDA runtime function)."""

import ctypes
import math

import numpy as np
import pytest
import torch

from paper_2606_07116_gb300 import build as B
from paper_2606_07116_gb300 import offq as Q


@pytest.fixture(scope="module")
def lib():
    B.build()
    return Q.load_library()


def test_exports_every_declared_symbol(lib):
    declared = Q.declared_symbols()
    assert {"offq_quantize_act", "offq_w4a4_linear", "offq_kv4_quantize", "offq_prepare_weight",
            "offq_get_device_status", "offq_status_string", "offq_abi_version"} <= set(declared)
    for name in declared:
        assert hasattr(lib, name), name


def test_wait_budget_hook_arguments(lib):
    assert lib.offq_set_wait_cycles(-1) == Q.OFFQ_ERR_INVALID_ARG
    assert lib.offq_set_wait_cycles(0) == Q.OFFQ_OK


def test_status_strings_and_version(lib):
    assert Q.abi_version() == 1
    for code, name in [(0, "OFFQ_OK"), (-1, "OFFQ_ERR_INVALID_ARG"), (-2, "OFFQ_ERR_UNSUPPORTED"),
                       (-3, "OFFQ_ERR_MISALIGNED"), (-4, "OFFQ_ERR_CUDA"), (-5, "OFFQ_ERR_TIMEOUT")]:
        assert Q.status_string(code) == name
    assert Q.status_string(12345) == "OFFQ_UNKNOWN_STATUS"


def test_missing_library_fails_loudly(tmp_path):
    with pytest.raises(RuntimeError):
        Q.load_library(str(tmp_path / "nope.so"))


P = ctypes.c_void_p
A16 = P(0x10000)      # a 16-byte aligned (never dereferenced) address
A8 = P(0x10008)       # only 8-byte aligned


def quant(lib, x=A16, dt=Q.OFFQ_BF16, T=4, K=1024, ldx=1024, g=256, flags=3, codes=A16, scale=A16, off=A16):
    return lib.offq_quantize_act(x, dt, T, K, ldx, g, flags, codes, scale, off, None)


def test_quantize_argument_checks(lib):
    assert quant(lib, g=33) == Q.OFFQ_ERR_INVALID_ARG          # g not a power of two
    assert quant(lib, g=16) == Q.OFFQ_ERR_INVALID_ARG          # g below 32
    assert quant(lib, g=16384, K=16384) == Q.OFFQ_ERR_INVALID_ARG
    assert quant(lib, K=1000) == Q.OFFQ_ERR_INVALID_ARG        # g does not divide K
    assert quant(lib, K=0) == Q.OFFQ_ERR_INVALID_ARG
    assert quant(lib, K=65536, ldx=65536) == Q.OFFQ_ERR_UNSUPPORTED
    assert quant(lib, g=32, K=8192, ldx=8192) == Q.OFFQ_ERR_UNSUPPORTED  # K > 128 g
    assert quant(lib, ldx=1000) == Q.OFFQ_ERR_INVALID_ARG      # ldx < K
    assert quant(lib, dt=7) == Q.OFFQ_ERR_INVALID_ARG
    assert quant(lib, flags=4) == Q.OFFQ_ERR_INVALID_ARG
    assert quant(lib, T=-1) == Q.OFFQ_ERR_INVALID_ARG
    assert quant(lib, x=None) == Q.OFFQ_ERR_INVALID_ARG
    assert quant(lib, off=None) == Q.OFFQ_ERR_INVALID_ARG      # OFFSET needs an offset buffer
    assert quant(lib, x=A8) == Q.OFFQ_ERR_MISALIGNED
    assert quant(lib, codes=A8) == Q.OFFQ_ERR_MISALIGNED
    assert quant(lib, ldx=1028) == Q.OFFQ_ERR_MISALIGNED       # row pitch not a multiple of 16 bytes
    assert quant(lib, T=0) == Q.OFFQ_OK                        # nothing to do, nothing launched
    assert quant(lib, T=0, x=None, codes=None) == Q.OFFQ_OK


def gemm(lib, a=A16, sa=A16, oa=A16, T=8, N=64, K=1024, g=256, w=A16, sw=A16, R=A16, out=A16, dt=Q.OFFQ_BF16,
         ldo=64, dbg=None):
    return lib.offq_w4a4_linear(a, sa, oa, T, N, K, g, w, sw, R, out, dt, ldo, dbg, None)


def test_gemm_argument_checks(lib):
    assert gemm(lib, g=100) == Q.OFFQ_ERR_INVALID_ARG
    assert gemm(lib, K=1000) == Q.OFFQ_ERR_INVALID_ARG
    assert gemm(lib, N=0) == Q.OFFQ_ERR_INVALID_ARG
    assert gemm(lib, ldo=32) == Q.OFFQ_ERR_INVALID_ARG
    assert gemm(lib, dt=9) == Q.OFFQ_ERR_INVALID_ARG
    assert gemm(lib, K=131072, g=4096) == Q.OFFQ_ERR_UNSUPPORTED
    assert gemm(lib, w=None) == Q.OFFQ_ERR_INVALID_ARG
    assert gemm(lib, a=A8) == Q.OFFQ_ERR_MISALIGNED
    assert gemm(lib, out=A8) == Q.OFFQ_ERR_MISALIGNED
    assert gemm(lib, ldo=65) == Q.OFFQ_ERR_MISALIGNED
    assert gemm(lib, T=0) == Q.OFFQ_OK


def test_kv_and_weight_argument_checks(lib):
    kv = lib.offq_kv4_quantize
    assert kv(A16, Q.OFFQ_BF16, 4, 0, 128, 128, 3, A16, A16, A16, None) == Q.OFFQ_ERR_INVALID_ARG    # H = 0
    assert kv(A16, Q.OFFQ_BF16, 4, 8, 96, 768, 3, A16, A16, A16, None) == Q.OFFQ_ERR_INVALID_ARG     # head_dim
    assert kv(A16, Q.OFFQ_BF16, 4, 8, 128, 512, 3, A16, A16, A16, None) == Q.OFFQ_ERR_INVALID_ARG    # ld_token
    assert kv(A8, Q.OFFQ_BF16, 4, 8, 128, 1024, 3, A16, A16, A16, None) == Q.OFFQ_ERR_MISALIGNED
    assert kv(A16, Q.OFFQ_BF16, 0, 8, 128, 1024, 3, A16, A16, A16, None) == Q.OFFQ_OK
    pw = lib.offq_prepare_weight
    assert pw(A16, Q.OFFQ_F32, 0, 1024, 256, 1, A16, A16, A16, None) == Q.OFFQ_ERR_INVALID_ARG      # N = 0
    assert pw(A16, Q.OFFQ_F32, 8, 1000, 256, 1, A16, A16, A16, None) == Q.OFFQ_ERR_INVALID_ARG
    assert pw(A16, Q.OFFQ_F32, 8, 1024, 256, 1, A16, A16, None, None) == Q.OFFQ_ERR_INVALID_ARG
    assert pw(A8, Q.OFFQ_F32, 8, 1024, 256, 1, A16, A16, A16, None) == Q.OFFQ_ERR_MISALIGNED


def test_code_buffer_sizes(lib):
    assert Q.offq_act_codes_bytes(1, 4096) == 32 * 2048
    assert Q.offq_act_codes_bytes(64, 4096) == 64 * 2048
    assert Q.offq_act_codes_bytes(65, 64) == 96 * 32
    assert Q.offq_act_codes_bytes(0, 64) == 0
    assert Q.offq_act_codes_bytes(4, 48) == -1
    assert Q.offq_weight_codes_bytes(11008, 4096) == 11008 * 2048
    assert Q.offq_weight_codes_bytes(300, 1024) == 320 * 512
    assert Q.offq_weight_codes_bytes(0, 1024) == -1


def test_mx_argument_checks(lib):
    def qm(x=A16, dt=Q.OFFQ_BF16, T=8, K=1024, ldx=1024, g=256, flags=3, c=A16, sh=A16, s=A16, o=A16):
        return lib.offq_quantize_act_mx(x, dt, T, K, ldx, g, flags, c, sh, s, o, None)
    assert qm(g=100) == Q.OFFQ_ERR_INVALID_ARG
    assert qm(g=16) == Q.OFFQ_ERR_INVALID_ARG
    assert qm(K=1000, ldx=1000) == Q.OFFQ_ERR_INVALID_ARG      # g does not divide K
    assert qm(K=1088, ldx=1088, g=64) == Q.OFFQ_ERR_INVALID_ARG  # K not a multiple of 128
    assert qm(K=65536, ldx=65536, g=4096) == Q.OFFQ_ERR_UNSUPPORTED
    assert qm(ldx=512) == Q.OFFQ_ERR_INVALID_ARG
    assert qm(flags=4) == Q.OFFQ_ERR_INVALID_ARG
    assert qm(o=None) == Q.OFFQ_ERR_INVALID_ARG                # OFFSET needs an offset buffer
    assert qm(sh=None) == Q.OFFQ_ERR_INVALID_ARG
    assert qm(x=A8) == Q.OFFQ_ERR_MISALIGNED
    assert qm(T=0) == Q.OFFQ_OK
    pm = lib.offq_prepare_weight_mx
    assert pm(A16, Q.OFFQ_F32, 0, 1024, 256, 1, A16, A16, A16, A16, None) == Q.OFFQ_ERR_INVALID_ARG  # N = 0
    assert pm(A16, Q.OFFQ_F32, 8, 1024, 256, 1, A16, A16, A16, None, None) == Q.OFFQ_ERR_INVALID_ARG
    assert pm(A16, Q.OFFQ_F32, 8, 1000, 200, 1, A16, A16, A16, A16, None) == Q.OFFQ_ERR_INVALID_ARG

    def lm(T=8, N=64, K=1024, g=256, a=A16, sh=A16, w=A16, out=A16, dt=Q.OFFQ_BF16, ldo=64):
        return lib.offq_mx_linear(a, sh, A16, A16, T, N, K, g, w, A16, A16, A16, out, dt, ldo, None)
    assert lm(K=1000) == Q.OFFQ_ERR_INVALID_ARG
    assert lm(K=1088, g=64) == Q.OFFQ_ERR_INVALID_ARG
    assert lm(N=0) == Q.OFFQ_ERR_INVALID_ARG
    assert lm(ldo=32) == Q.OFFQ_ERR_INVALID_ARG
    assert lm(dt=9) == Q.OFFQ_ERR_INVALID_ARG
    assert lm(K=131072, g=4096) == Q.OFFQ_ERR_UNSUPPORTED
    assert lm(sh=None) == Q.OFFQ_ERR_INVALID_ARG
    assert lm(a=A8) == Q.OFFQ_ERR_MISALIGNED
    assert lm(T=0) == Q.OFFQ_OK
    assert Q.mx_shift_bytes(1, 4096) == 32 * 128
    assert Q.mx_shift_bytes(33, 128) == 64 * 4
    assert Q.mx_shift_bytes(4, 96) == -1


def test_group_path_argument_checks(lib):
    qg = lambda x=A16, dt=Q.OFFQ_BF16, T=4, K=1024, ldx=1024, g=256, group=128, flags=1, c=A16, s=A16, z=A16: \
        lib.offq_quantize_act_group(x, dt, T, K, ldx, g, group, flags, c, s, z, None)
    assert qg(group=64) == Q.OFFQ_ERR_UNSUPPORTED          # the library quantizes groups of 128
    assert qg(group=0) == Q.OFFQ_ERR_INVALID_ARG
    assert qg(K=1000, ldx=1000) == Q.OFFQ_ERR_INVALID_ARG  # group does not divide K
    assert qg(g=100) == Q.OFFQ_ERR_INVALID_ARG             # rotation block not a power of two
    assert qg(g=2048) == Q.OFFQ_ERR_INVALID_ARG            # rotation block does not divide K
    assert qg(flags=2) == Q.OFFQ_ERR_INVALID_ARG           # no explicit offset on this path
    assert qg(ldx=1000) == Q.OFFQ_ERR_INVALID_ARG
    assert qg(z=None) == Q.OFFQ_ERR_INVALID_ARG
    assert qg(x=A8) == Q.OFFQ_ERR_MISALIGNED
    assert qg(ldx=1028) == Q.OFFQ_ERR_MISALIGNED
    assert qg(T=0) == Q.OFFQ_OK
    ws = lambda w=A16, N=64, K=1024, group=128, out=A16: lib.offq_weight_group_sums(w, N, K, group, out, None)
    assert ws(group=100) == Q.OFFQ_ERR_INVALID_ARG
    assert ws(K=1000) == Q.OFFQ_ERR_INVALID_ARG
    assert ws(N=0) == Q.OFFQ_ERR_INVALID_ARG
    assert ws(out=None) == Q.OFFQ_ERR_INVALID_ARG
    assert ws(w=A8) == Q.OFFQ_ERR_MISALIGNED
    lg = lambda a=A16, sa=A16, za=A16, T=8, N=64, K=1024, group=128, w=A16, sw=A16, R=A16, out=A16, \
        dt=Q.OFFQ_BF16, ldo=64: lib.offq_w4a4_linear_group(a, sa, za, T, N, K, group, w, sw, R, out, dt, ldo, None)
    assert lg(group=256) == Q.OFFQ_ERR_UNSUPPORTED
    assert lg(K=1000) == Q.OFFQ_ERR_INVALID_ARG
    assert lg(N=0) == Q.OFFQ_ERR_INVALID_ARG
    assert lg(ldo=32) == Q.OFFQ_ERR_INVALID_ARG
    assert lg(dt=9) == Q.OFFQ_ERR_INVALID_ARG
    assert lg(K=131072) == Q.OFFQ_ERR_UNSUPPORTED
    assert lg(za=None) == Q.OFFQ_ERR_INVALID_ARG
    assert lg(a=A8) == Q.OFFQ_ERR_MISALIGNED
    assert lg(ldo=65) == Q.OFFQ_ERR_MISALIGNED
    assert lg(T=0) == Q.OFFQ_OK


def test_rotated_key_cache_argument_checks(lib):
    kq = lambda kv=A16, dt=Q.OFFQ_BF16, T=4, H=8, hd=128, ld=1024, rot=A16, flags=2, c=A16, s=A16, o=A16: \
        lib.offq_kv4_quantize_rotated(kv, dt, T, H, hd, ld, rot, flags, c, s, o, None)
    assert kq(hd=64, ld=512) == Q.OFFQ_ERR_UNSUPPORTED     # the library rotates heads of 128
    assert kq(H=0) == Q.OFFQ_ERR_INVALID_ARG
    assert kq(ld=512) == Q.OFFQ_ERR_INVALID_ARG            # ld_token < H * head_dim
    assert kq(flags=1) == Q.OFFQ_ERR_INVALID_ARG           # the rotation is M, not a flag
    assert kq(rot=None) == Q.OFFQ_ERR_INVALID_ARG
    assert kq(o=None) == Q.OFFQ_ERR_INVALID_ARG            # OFFSET needs an offset buffer
    assert kq(kv=A8) == Q.OFFQ_ERR_MISALIGNED
    assert kq(rot=A8) == Q.OFFQ_ERR_MISALIGNED
    assert kq(c=A8) == Q.OFFQ_ERR_MISALIGNED               # codes take 16-byte stores
    assert kq(dt=7) == Q.OFFQ_ERR_INVALID_ARG
    assert kq(T=0) == Q.OFFQ_OK
    rh = lambda x=A16, T=4, H=8, hd=128, ld=1024, rot=A16, out=A16, odt=Q.OFFQ_F32, ldo=1024: \
        lib.offq_rotate_heads(x, Q.OFFQ_BF16, T, H, hd, ld, rot, out, odt, ldo, None)
    assert rh(ldo=512) == Q.OFFQ_ERR_INVALID_ARG
    assert rh(odt=9) == Q.OFFQ_ERR_INVALID_ARG
    assert rh(out=None) == Q.OFFQ_ERR_INVALID_ARG
    assert rh(out=A8) == Q.OFFQ_ERR_MISALIGNED
    assert rh(T=0) == Q.OFFQ_OK


def test_prepared_key_rotation_argument_checks(lib):
    pr = lambda rot=A16, H=8, hd=128, prep=A16: lib.offq_prepare_key_rotation(rot, H, hd, prep, None)
    assert pr(hd=64) == Q.OFFQ_ERR_UNSUPPORTED
    assert pr(H=0) == Q.OFFQ_ERR_INVALID_ARG
    assert pr(H=70000) == Q.OFFQ_ERR_UNSUPPORTED
    assert pr(rot=None) == Q.OFFQ_ERR_INVALID_ARG
    assert pr(prep=None) == Q.OFFQ_ERR_INVALID_ARG
    assert pr(rot=A8) == Q.OFFQ_ERR_MISALIGNED
    assert pr(prep=A8) == Q.OFFQ_ERR_MISALIGNED
    kp = lambda kv=A16, dt=Q.OFFQ_BF16, T=4, H=8, hd=128, ld=1024, prep=A16, flags=2, c=A16, s=A16, o=A16: \
        lib.offq_kv4_quantize_prepared(kv, dt, T, H, hd, ld, prep, flags, c, s, o, None)
    assert kp(dt=Q.OFFQ_F32) == Q.OFFQ_ERR_UNSUPPORTED     # the prepared parts serve bf16 inputs
    assert kp(dt=Q.OFFQ_F16) == Q.OFFQ_ERR_UNSUPPORTED
    assert kp(hd=64, ld=512) == Q.OFFQ_ERR_UNSUPPORTED
    assert kp(prep=None) == Q.OFFQ_ERR_INVALID_ARG
    assert kp(prep=A8) == Q.OFFQ_ERR_MISALIGNED
    assert kp(flags=1) == Q.OFFQ_ERR_INVALID_ARG
    assert kp(o=None) == Q.OFFQ_ERR_INVALID_ARG
    assert kp(c=A8) == Q.OFFQ_ERR_MISALIGNED
    assert kp(T=0) == Q.OFFQ_OK
    rp = lambda x=A16, dt=Q.OFFQ_BF16, T=4, prep=A16, out=A16, odt=Q.OFFQ_F32, ldo=1024: \
        lib.offq_rotate_heads_prepared(x, dt, T, 8, 128, 1024, prep, out, odt, ldo, None)
    assert rp(dt=Q.OFFQ_F32) == Q.OFFQ_ERR_UNSUPPORTED
    assert rp(prep=None) == Q.OFFQ_ERR_INVALID_ARG
    assert rp(ldo=512) == Q.OFFQ_ERR_INVALID_ARG
    assert rp(out=None) == Q.OFFQ_ERR_INVALID_ARG
    assert rp(out=A8) == Q.OFFQ_ERR_MISALIGNED
    assert rp(T=0) == Q.OFFQ_OK


def test_builder_argument_checks(lib):
    assert lib.offq_top1_tokens(A16, Q.OFFQ_BF16, 4, 8, 64, 32, 512, A16, A16, None) == Q.OFFQ_ERR_INVALID_ARG
    assert lib.offq_top1_tokens(A16, Q.OFFQ_BF16, 4, 8, 64, 64, 256, A16, A16, None) == Q.OFFQ_ERR_INVALID_ARG
    assert lib.offq_top1_tokens(A16, Q.OFFQ_BF16, 0, 8, 64, 64, 512, None, None, None) == Q.OFFQ_OK
    assert lib.offq_top1_direction(A16, 4, 64, 0, A16, A16, A16, None) == Q.OFFQ_ERR_INVALID_ARG
    assert lib.offq_top1_direction(A16, 4, 64, 10, None, A16, A16, None) == Q.OFFQ_ERR_INVALID_ARG
    assert lib.offq_reflect_rows(A16, 4, 32768, A16, A16, None) == Q.OFFQ_ERR_UNSUPPORTED
    assert lib.offq_reflect_rows(A16, 0, 64, A16, A16, None) == Q.OFFQ_OK
    assert lib.offq_fuse_rotation(A16, 4, 64, A16, A16, 48, A16, None) == Q.OFFQ_ERR_INVALID_ARG
    assert lib.offq_fuse_rotation(A16, 4, 64, A16, None, 64, A16, None) == Q.OFFQ_ERR_INVALID_ARG
    assert lib.offq_column_absmax(A16, 0, 64, A16, None) == Q.OFFQ_ERR_INVALID_ARG
    assert lib.offq_sorted_grouping(None, 6, 2, None) == Q.OFFQ_ERR_INVALID_ARG


def test_sorted_grouping_host_matches_oracle(lib):
    """The host grouping is plain C++: exact against the oracle, including the
    paper's example and ties."""
    import numpy as np
    import torch
    import oracle as O
    vals = torch.tensor([1, 2, 3, 4, 50, 60], dtype=torch.float32)
    perm = Q.sorted_grouping(vals, 2).numpy()
    assert list(vals.numpy()[perm]) == [60, 1, 2, 50, 3, 4]
    rng = np.random.default_rng(70)
    for D, G in [(256, 4), (4096, 32), (64, 1), (12, 3)]:
        m = rng.standard_normal(D).astype(np.float32)
        m[rng.integers(0, D, size=D // 8)] = 0.5  # ties
        np.testing.assert_array_equal(Q.sorted_grouping(torch.from_numpy(m), G).numpy(),
                                      O.sorted_grouping(m.astype(np.float64), G))


def _decode_reflection(img, H):
    """The structured image back to B [H][144][128] (float64) and w'' [H][128]."""
    u = np.frombuffer(img.numpy().tobytes(), dtype=np.uint8).reshape(H, -1)
    b = u[:, :36864].copy().view(np.uint16).reshape(H, 2, 144, 8, 8)   # [h][half][row][slot][e]
    n = np.arange(144)[:, None]
    c = np.arange(16)[None, :]
    g = b[:, c >> 3, n, (c & 7) ^ (n & 7), :]                           # [H, 144, 16, 8]
    B = ((g.reshape(H, 144, 128).astype(np.uint32) << 16).view(np.float32)).astype(np.float64)
    wpp = u[:, 36864:].copy().view(np.float32).astype(np.float64)
    return B, wpp


def test_key_reflection_image_matches_the_oracle_rotation(lib):
    """Host prepare of M = U3 P3 H3: the +-1 rows are sqrt(128) (P3 H3)^T, the
    three parts of w rebuild the reflection, and w'' = (P3 H3)^T w, so the image
    gives the oracle's M back (Sec. 3.3 Step 2 (3))."""
    import oracle as O
    H, hd = 3, 128
    rng = np.random.default_rng(5)
    keys = rng.standard_normal((64, H, hd))
    keys[:, :, 5] += 30.0                            # a concentrated channel per head
    keys[:, 2, :] = 0.01 * rng.standard_normal((64, hd))
    keys[:, 2, 0] += 40.0                            # head 2: direction ~ e_0 (U3 close to I)
    perm = np.stack([np.concatenate([[0], 1 + rng.permutation(hd - 1)]) for _ in range(H)]).astype(np.int32)
    v = np.stack([O.top1_pca_direction(keys[:, h, :]) for h in range(H)]).astype(np.float32)
    img = Q.prepare_key_reflection(torch.from_numpy(v), torch.from_numpy(perm))
    B, wpp = _decode_reflection(img, H)
    Hs = O.sylvester_hadamard(hd).astype(np.float64) / math.sqrt(hd)
    for h in range(H):
        PH = np.eye(hd)[:, perm[h]] @ Hs
        assert np.array_equal(B[h, :hd], np.sign(PH.T))  # sqrt(128) (P3 H3)[k][n] = +-1 at row n
        assert np.all(B[h, hd + 3:] == 0)
        w = B[h, hd] + B[h, hd + 1] + B[h, hd + 2]
        U = np.eye(hd) - 2.0 * np.outer(w, w)
        M_img = U @ PH
        M_ref = O.householder_to_first(v[h].astype(np.float64)) @ PH
        assert np.max(np.abs(M_img - M_ref)) < 1e-6
        # w'' from the float64 w, rounded once; w here is fp32(w) (its parts'
        # sum), at most 2^-24 |w_k| from the float64 w in each entry.
        tol = 2.0 ** -24 * (np.abs(PH.T @ w) + np.abs(PH.T) @ np.abs(w)) * 2
        assert np.all(np.abs(wpp[h] - PH.T @ w) <= tol)


def test_key_reflection_argument_checks(lib):
    hd = 128
    v = torch.ones((2, hd), dtype=torch.float32)
    perm = torch.arange(hd, dtype=torch.int32).repeat(2, 1)
    out = torch.empty((2, Q.KEY_REFLECTION_BYTES), dtype=torch.uint8)
    call = lambda v=v, perm=perm, H=2, hd=hd: lib.offq_prepare_key_reflection(
        ctypes.c_void_p(v.data_ptr()), ctypes.c_void_p(perm.data_ptr()), H, hd, ctypes.c_void_p(out.data_ptr()))
    assert call() == Q.OFFQ_OK
    assert call(hd=64) == Q.OFFQ_ERR_UNSUPPORTED
    assert call(H=0) == Q.OFFQ_ERR_INVALID_ARG
    bad = perm.clone(); bad[1, 7] = 3                # not a permutation
    assert call(perm=bad) == Q.OFFQ_ERR_INVALID_ARG
    zero = v.clone(); zero[1] = 0.0                   # no direction
    assert call(v=zero) == Q.OFFQ_ERR_INVALID_ARG
    assert lib.offq_prepare_key_reflection(None, None, 2, hd, None) == Q.OFFQ_ERR_INVALID_ARG
    kr = lambda dt=Q.OFFQ_BF16, prep=A16, flags=2, T=4: \
        lib.offq_kv4_quantize_reflected(A16, dt, T, 8, 128, 1024, prep, flags, A16, A16, A16, None)
    assert kr(dt=Q.OFFQ_F32) == Q.OFFQ_ERR_UNSUPPORTED
    assert kr(prep=None) == Q.OFFQ_ERR_INVALID_ARG
    assert kr(prep=A8) == Q.OFFQ_ERR_MISALIGNED
    assert kr(flags=1) == Q.OFFQ_ERR_INVALID_ARG
    assert kr(T=0) == Q.OFFQ_OK
    rr = lambda dt=Q.OFFQ_BF16, out=A16, T=4: \
        lib.offq_rotate_heads_reflected(A16, dt, T, 8, 128, 1024, A16, out, Q.OFFQ_F32, 1024, None)
    assert rr(dt=Q.OFFQ_F16) == Q.OFFQ_ERR_UNSUPPORTED
    assert rr(out=A8) == Q.OFFQ_ERR_MISALIGNED
    assert rr(T=0) == Q.OFFQ_OK
