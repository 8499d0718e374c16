"""Python binding of liboffq.so (the OffQ W4A4 linear path on GB300).

The functions named ``offq_*`` mirror the C ABI in ``include/offq.h`` one to
one: they take torch CUDA tensors, pass their device pointers, sizes and the
current CUDA stream to the library, and raise :class:`OffqError` on a non-zero
status. All computation happens in the library's kernels; torch supplies device
memory and streams only. The helpers without the prefix (``quantize_act``,
``w4a4_linear``, ...) allocate the outputs with torch and call the same entry
points. Activation and weight code buffers are [ceil(R/32)*32, K/2] uint8
tensors holding the tiled operand layout of include/offq.h.
"""

from __future__ import annotations

import ctypes
import os
import re
from typing import Optional, Tuple

import torch

from . import build as _build

OFFQ_OK = 0
OFFQ_ERR_INVALID_ARG = -1
OFFQ_ERR_UNSUPPORTED = -2
OFFQ_ERR_MISALIGNED = -3
OFFQ_ERR_CUDA = -4
OFFQ_ERR_TIMEOUT = -5

OFFQ_F32, OFFQ_BF16, OFFQ_F16 = 0, 1, 2
OFFQ_ROTATE, OFFQ_OFFSET = 1, 2

_DTYPE_CODE = {torch.float32: OFFQ_F32, torch.bfloat16: OFFQ_BF16, torch.float16: OFFQ_F16}
_CODE_DTYPE = {v: k for k, v in _DTYPE_CODE.items()}

_c_vp = ctypes.c_void_p
_c_i64 = ctypes.c_int64
_c_i32 = ctypes.c_int32
_c_int = ctypes.c_int

_SIGNATURES = {
    "offq_quantize_act": (_c_int, [_c_vp, _c_int, _c_i64, _c_i64, _c_i64, _c_i32, _c_i32, _c_vp, _c_vp, _c_vp, _c_vp]),
    "offq_w4a4_linear": (_c_int, [_c_vp, _c_vp, _c_vp, _c_i64, _c_i64, _c_i64, _c_i32, _c_vp, _c_vp, _c_vp, _c_vp,
                                  _c_int, _c_i64, _c_vp, _c_vp]),
    "offq_kv4_quantize": (_c_int, [_c_vp, _c_int, _c_i64, _c_i32, _c_i32, _c_i64, _c_i32, _c_vp, _c_vp, _c_vp, _c_vp]),
    "offq_prepare_weight": (_c_int, [_c_vp, _c_int, _c_i64, _c_i64, _c_i32, _c_i32, _c_vp, _c_vp, _c_vp, _c_vp]),
    "offq_get_device_status": (_c_int, [_c_vp]),
    "offq_set_wait_cycles": (_c_int, [_c_i64]),
    "offq_quantize_act_mx": (_c_int, [_c_vp, _c_int, _c_i64, _c_i64, _c_i64, _c_i32, _c_i32, _c_vp, _c_vp, _c_vp,
                                      _c_vp, _c_vp]),
    "offq_prepare_weight_mx": (_c_int, [_c_vp, _c_int, _c_i64, _c_i64, _c_i32, _c_i32, _c_vp, _c_vp, _c_vp, _c_vp,
                                        _c_vp]),
    "offq_mx_linear": (_c_int, [_c_vp, _c_vp, _c_vp, _c_vp, _c_i64, _c_i64, _c_i64, _c_i32, _c_vp, _c_vp, _c_vp,
                                _c_vp, _c_vp, _c_int, _c_i64, _c_vp]),
    "offq_mx_shift_bytes": (_c_i64, [_c_i64, _c_i64]),
    "offq_status_string": (ctypes.c_char_p, [_c_int]),
    "offq_abi_version": (_c_int, []),
    "offq_act_codes_bytes": (_c_i64, [_c_i64, _c_i64]),
    "offq_weight_codes_bytes": (_c_i64, [_c_i64, _c_i64]),
    "offq_quantize_act_group": (_c_int, [_c_vp, _c_int, _c_i64, _c_i64, _c_i64, _c_i32, _c_i32, _c_i32, _c_vp, _c_vp,
                                         _c_vp, _c_vp]),
    "offq_weight_group_sums": (_c_int, [_c_vp, _c_i64, _c_i64, _c_i32, _c_vp, _c_vp]),
    "offq_w4a4_linear_group": (_c_int, [_c_vp, _c_vp, _c_vp, _c_i64, _c_i64, _c_i64, _c_i32, _c_vp, _c_vp, _c_vp,
                                        _c_vp, _c_int, _c_i64, _c_vp]),
    "offq_kv4_quantize_rotated": (_c_int, [_c_vp, _c_int, _c_i64, _c_i32, _c_i32, _c_i64, _c_vp, _c_i32, _c_vp,
                                           _c_vp, _c_vp, _c_vp]),
    "offq_rotate_heads": (_c_int, [_c_vp, _c_int, _c_i64, _c_i32, _c_i32, _c_i64, _c_vp, _c_vp, _c_int, _c_i64,
                                   _c_vp]),
    "offq_prepare_key_rotation": (_c_int, [_c_vp, _c_i32, _c_i32, _c_vp, _c_vp]),
    "offq_kv4_quantize_prepared": (_c_int, [_c_vp, _c_int, _c_i64, _c_i32, _c_i32, _c_i64, _c_vp, _c_i32, _c_vp,
                                            _c_vp, _c_vp, _c_vp]),
    "offq_rotate_heads_prepared": (_c_int, [_c_vp, _c_int, _c_i64, _c_i32, _c_i32, _c_i64, _c_vp, _c_vp, _c_int,
                                            _c_i64, _c_vp]),
    "offq_prepare_key_reflection": (_c_int, [_c_vp, _c_vp, _c_i32, _c_i32, _c_vp]),
    "offq_kv4_quantize_reflected": (_c_int, [_c_vp, _c_int, _c_i64, _c_i32, _c_i32, _c_i64, _c_vp, _c_i32, _c_vp,
                                             _c_vp, _c_vp, _c_vp]),
    "offq_rotate_heads_reflected": (_c_int, [_c_vp, _c_int, _c_i64, _c_i32, _c_i32, _c_i64, _c_vp, _c_vp, _c_int,
                                             _c_i64, _c_vp]),
    "offq_top1_tokens": (_c_int, [_c_vp, _c_int, _c_i64, _c_i64, _c_i64, _c_i64, _c_i64, _c_vp, _c_vp, _c_vp]),
    "offq_top1_direction": (_c_int, [_c_vp, _c_i64, _c_i64, _c_i32, _c_vp, _c_vp, _c_vp, _c_vp]),
    "offq_reflect_rows": (_c_int, [_c_vp, _c_i64, _c_i64, _c_vp, _c_vp, _c_vp]),
    "offq_column_absmax": (_c_int, [_c_vp, _c_i64, _c_i64, _c_vp, _c_vp]),
    "offq_sorted_grouping": (_c_int, [_c_vp, _c_i64, _c_i32, _c_vp]),
    "offq_fuse_rotation": (_c_int, [_c_vp, _c_i64, _c_i64, _c_vp, _c_vp, _c_i32, _c_vp, _c_vp]),
}

_lib = None


class OffqError(RuntimeError):
    def __init__(self, fn: str, status: int):
        self.status = status
        super().__init__(f"{fn} failed: {status_string(status)} ({status})")


def library_path() -> str:
    return _build.LIB_PATH


def load_library(path: Optional[str] = None) -> ctypes.CDLL:
    """Loads liboffq.so (raises if it was not built: there is no fallback)."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = path or library_path()
    if not os.path.exists(p):
        raise RuntimeError(f"liboffq.so not found at {p}; build it with "
                           "paper_2606_07116_gb300.build.build() (no CPU fallback exists)")
    lib = ctypes.CDLL(p)
    for name, (res, args) in _SIGNATURES.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    if path is None:
        _lib = lib
    return lib


def declared_symbols(header: Optional[str] = None):
    """Names of the functions include/offq.h declares."""
    header = header or os.path.join(_build.INCLUDE, "offq.h")
    with open(header) as f:
        text = f.read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(offq_[a-z0-9_]+)\s*\(", text)))


def status_string(status: int) -> str:
    return load_library().offq_status_string(status).decode()


def abi_version() -> int:
    return load_library().offq_abi_version()


def _check(fn: str, rc: int):
    if rc != OFFQ_OK:
        raise OffqError(fn, rc)


def _ptr(t: Optional[torch.Tensor]):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("tensors passed to liboffq must live on a CUDA device")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    if isinstance(stream, torch.cuda.Stream):
        return ctypes.c_void_p(stream.cuda_stream)
    return ctypes.c_void_p(int(stream))


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype not in _DTYPE_CODE:
        raise ValueError(f"unsupported dtype {t.dtype}")
    return _DTYPE_CODE[t.dtype]


# ---------------------------------------------------------------------------
# One-to-one wrappers of the C ABI.
# ---------------------------------------------------------------------------

def offq_quantize_act(x: torch.Tensor, T: int, K: int, ldx: int, g: int, flags: int,
                      codes: torch.Tensor, scale: torch.Tensor, offset: Optional[torch.Tensor],
                      stream=None) -> None:
    _check("offq_quantize_act", load_library().offq_quantize_act(
        _ptr(x), _dtype_code(x), T, K, ldx, g, flags, _ptr(codes), _ptr(scale), _ptr(offset), _stream(stream)))


def offq_w4a4_linear(a_codes: torch.Tensor, a_scale: torch.Tensor, a_offset: Optional[torch.Tensor],
                     T: int, N: int, K: int, g: int, w_codes: torch.Tensor, w_scale: torch.Tensor,
                     w_offsum: torch.Tensor, out: torch.Tensor, ldo: int,
                     acc_debug: Optional[torch.Tensor] = None, stream=None) -> None:
    _check("offq_w4a4_linear", load_library().offq_w4a4_linear(
        _ptr(a_codes), _ptr(a_scale), _ptr(a_offset), T, N, K, g, _ptr(w_codes), _ptr(w_scale),
        _ptr(w_offsum), _ptr(out), _dtype_code(out), ldo, _ptr(acc_debug), _stream(stream)))


def offq_kv4_quantize(kv: torch.Tensor, T: int, H: int, head_dim: int, ld_token: int, flags: int,
                      codes: torch.Tensor, scale: torch.Tensor, offset: Optional[torch.Tensor],
                      stream=None) -> None:
    _check("offq_kv4_quantize", load_library().offq_kv4_quantize(
        _ptr(kv), _dtype_code(kv), T, H, head_dim, ld_token, flags, _ptr(codes), _ptr(scale), _ptr(offset),
        _stream(stream)))


def offq_prepare_weight(w: torch.Tensor, N: int, K: int, g: int, rotate: bool, w_codes: torch.Tensor,
                        w_scale: torch.Tensor, w_offsum: torch.Tensor, stream=None) -> None:
    _check("offq_prepare_weight", load_library().offq_prepare_weight(
        _ptr(w), _dtype_code(w), N, K, g, 1 if rotate else 0, _ptr(w_codes), _ptr(w_scale), _ptr(w_offsum),
        _stream(stream)))


def offq_quantize_act_group(x: torch.Tensor, T: int, K: int, ldx: int, g: int, group: int, flags: int,
                            codes: torch.Tensor, scale: torch.Tensor, zero: torch.Tensor, stream=None) -> None:
    _check("offq_quantize_act_group", load_library().offq_quantize_act_group(
        _ptr(x), _dtype_code(x), T, K, ldx, g, group, flags, _ptr(codes), _ptr(scale), _ptr(zero), _stream(stream)))


def offq_weight_group_sums(w_codes: torch.Tensor, N: int, K: int, group: int, w_groupsum: torch.Tensor,
                           stream=None) -> None:
    _check("offq_weight_group_sums", load_library().offq_weight_group_sums(
        _ptr(w_codes), N, K, group, _ptr(w_groupsum), _stream(stream)))


def offq_w4a4_linear_group(a_codes: torch.Tensor, a_scale: torch.Tensor, a_zero: torch.Tensor, T: int, N: int,
                           K: int, group: int, w_codes: torch.Tensor, w_scale: torch.Tensor,
                           w_groupsum: torch.Tensor, out: torch.Tensor, ldo: int, stream=None) -> None:
    _check("offq_w4a4_linear_group", load_library().offq_w4a4_linear_group(
        _ptr(a_codes), _ptr(a_scale), _ptr(a_zero), T, N, K, group, _ptr(w_codes), _ptr(w_scale),
        _ptr(w_groupsum), _ptr(out), _dtype_code(out), ldo, _stream(stream)))


def offq_kv4_quantize_rotated(kv: torch.Tensor, T: int, H: int, head_dim: int, ld_token: int, rot: torch.Tensor,
                              flags: int, codes: torch.Tensor, scale: torch.Tensor, offset: Optional[torch.Tensor],
                              stream=None) -> None:
    _check("offq_kv4_quantize_rotated", load_library().offq_kv4_quantize_rotated(
        _ptr(kv), _dtype_code(kv), T, H, head_dim, ld_token, _ptr(rot), flags, _ptr(codes), _ptr(scale),
        _ptr(offset), _stream(stream)))


def offq_rotate_heads(x: torch.Tensor, T: int, H: int, head_dim: int, ld_token: int, rot: torch.Tensor,
                      out: torch.Tensor, ld_out: int, stream=None) -> None:
    _check("offq_rotate_heads", load_library().offq_rotate_heads(
        _ptr(x), _dtype_code(x), T, H, head_dim, ld_token, _ptr(rot), _ptr(out), _dtype_code(out), ld_out,
        _stream(stream)))


def offq_prepare_key_rotation(rot: torch.Tensor, H: int, head_dim: int, prepared: torch.Tensor,
                              stream=None) -> None:
    _check("offq_prepare_key_rotation", load_library().offq_prepare_key_rotation(
        _ptr(rot), H, head_dim, _ptr(prepared), _stream(stream)))


def offq_kv4_quantize_prepared(kv: torch.Tensor, T: int, H: int, head_dim: int, ld_token: int,
                               prepared: torch.Tensor, flags: int, codes: torch.Tensor, scale: torch.Tensor,
                               offset: Optional[torch.Tensor], stream=None) -> None:
    _check("offq_kv4_quantize_prepared", load_library().offq_kv4_quantize_prepared(
        _ptr(kv), _dtype_code(kv), T, H, head_dim, ld_token, _ptr(prepared), flags, _ptr(codes), _ptr(scale),
        _ptr(offset), _stream(stream)))


def offq_rotate_heads_prepared(x: torch.Tensor, T: int, H: int, head_dim: int, ld_token: int,
                               prepared: torch.Tensor, out: torch.Tensor, ld_out: int, stream=None) -> None:
    _check("offq_rotate_heads_prepared", load_library().offq_rotate_heads_prepared(
        _ptr(x), _dtype_code(x), T, H, head_dim, ld_token, _ptr(prepared), _ptr(out), _dtype_code(out), ld_out,
        _stream(stream)))


def offq_prepare_key_reflection(v: torch.Tensor, perm: torch.Tensor, H: int, head_dim: int,
                                prepared: torch.Tensor) -> None:
    """Host call: v [H, hd] float32, perm [H, hd] int32 and prepared (uint8) all in host memory."""
    for t in (v, perm, prepared):
        if t.device.type != "cpu" or not t.is_contiguous():
            raise ValueError("offq_prepare_key_reflection takes contiguous host tensors")
    _check("offq_prepare_key_reflection", load_library().offq_prepare_key_reflection(
        ctypes.c_void_p(v.data_ptr()), ctypes.c_void_p(perm.data_ptr()), H, head_dim,
        ctypes.c_void_p(prepared.data_ptr())))


def offq_kv4_quantize_reflected(kv: torch.Tensor, T: int, H: int, head_dim: int, ld_token: int,
                                prepared: torch.Tensor, flags: int, codes: torch.Tensor, scale: torch.Tensor,
                                offset: Optional[torch.Tensor], stream=None) -> None:
    _check("offq_kv4_quantize_reflected", load_library().offq_kv4_quantize_reflected(
        _ptr(kv), _dtype_code(kv), T, H, head_dim, ld_token, _ptr(prepared), flags, _ptr(codes), _ptr(scale),
        _ptr(offset), _stream(stream)))


def offq_rotate_heads_reflected(x: torch.Tensor, T: int, H: int, head_dim: int, ld_token: int,
                                prepared: torch.Tensor, out: torch.Tensor, ld_out: int, stream=None) -> None:
    _check("offq_rotate_heads_reflected", load_library().offq_rotate_heads_reflected(
        _ptr(x), _dtype_code(x), T, H, head_dim, ld_token, _ptr(prepared), _ptr(out), _dtype_code(out), ld_out,
        _stream(stream)))


def offq_get_device_status(stream=None) -> int:
    return load_library().offq_get_device_status(_stream(stream))


def offq_set_wait_cycles(cycles: int) -> None:
    """Test hook: budget of the persistent quantizers' waits for staged rows
    (0 restores the default)."""
    _check("offq_set_wait_cycles", load_library().offq_set_wait_cycles(cycles))


def offq_act_codes_bytes(T: int, K: int) -> int:
    return load_library().offq_act_codes_bytes(T, K)


def offq_weight_codes_bytes(N: int, K: int) -> int:
    return load_library().offq_weight_codes_bytes(N, K)


def padded_rows(R: int) -> int:
    """Rows a tiled code buffer holds for R rows (a multiple of 32)."""
    return (R + 31) // 32 * 32


# ---------------------------------------------------------------------------
# Allocating helpers (torch allocates; the entry points above compute).
# ---------------------------------------------------------------------------

def quantize_act(x: torch.Tensor, g: int, rotate: bool = True, offset: bool = True,
                 stream=None) -> Tuple[torch.Tensor, torch.Tensor, torch.Tensor]:
    T, K = x.shape
    codes = torch.empty((padded_rows(T), K // 2), dtype=torch.uint8, device=x.device)
    scale = torch.empty((T,), dtype=torch.float32, device=x.device)
    off = torch.empty((T, K // g), dtype=torch.float32, device=x.device)
    flags = (OFFQ_ROTATE if rotate else 0) | (OFFQ_OFFSET if offset else 0)
    offq_quantize_act(x, T, K, x.stride(0), g, flags, codes, scale, off, stream)
    return codes, scale, off


def kv4_quantize(kv: torch.Tensor, rotate: bool = True, offset: bool = True,
                 stream=None) -> Tuple[torch.Tensor, torch.Tensor, torch.Tensor]:
    T, H, hd = kv.shape
    if kv.stride(2) != 1 or kv.stride(1) != hd:
        raise ValueError("heads of a token must be contiguous")
    codes = torch.empty((T, H, hd // 2), dtype=torch.uint8, device=kv.device)
    scale = torch.empty((T, H), dtype=torch.float32, device=kv.device)
    off = torch.empty((T, H), dtype=torch.float32, device=kv.device)
    flags = (OFFQ_ROTATE if rotate else 0) | (OFFQ_OFFSET if offset else 0)
    offq_kv4_quantize(kv, T, H, hd, kv.stride(0), flags, codes, scale, off, stream)
    return codes, scale, off


def prepare_weight(w: torch.Tensor, g: int, rotate: bool = True,
                   stream=None) -> Tuple[torch.Tensor, torch.Tensor, torch.Tensor]:
    N, K = w.shape
    w = w.contiguous()
    codes = torch.empty((padded_rows(N), K // 2), dtype=torch.uint8, device=w.device)
    scale = torch.empty((N,), dtype=torch.float32, device=w.device)
    rowsum = torch.empty((K // g, N), dtype=torch.float32, device=w.device)
    offq_prepare_weight(w, N, K, g, rotate, codes, scale, rowsum, stream)
    return codes, scale, rowsum


def w4a4_linear(a_codes: torch.Tensor, a_scale: torch.Tensor, a_offset: Optional[torch.Tensor],
                w_codes: torch.Tensor, w_scale: torch.Tensor, w_offsum: torch.Tensor, g: int,
                out_dtype: torch.dtype = torch.bfloat16, out: Optional[torch.Tensor] = None,
                acc_debug: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    T = a_scale.shape[0]
    K = a_codes.shape[1] * 2
    N = w_scale.shape[0]
    if out is None:
        out = torch.empty((T, N), dtype=out_dtype, device=a_codes.device)
    offq_w4a4_linear(a_codes, a_scale, a_offset, T, N, K, g, w_codes, w_scale, w_offsum, out, out.stride(0),
                     acc_debug, stream)
    return out


GROUP = 128  # activation group size of the per-group path (the paper's evaluated setting)


def quantize_act_group(x: torch.Tensor, g: int, group: int = GROUP, rotate: bool = True,
                       stream=None) -> Tuple[torch.Tensor, torch.Tensor, torch.Tensor]:
    """Per-group asymmetric codes, scales and zero-points of token rows x [T, K]."""
    T, K = x.shape
    codes = torch.empty((padded_rows(T), K // 2), dtype=torch.uint8, device=x.device)
    scale = torch.empty((T, K // group), dtype=torch.float32, device=x.device)
    zero = torch.empty((T, K // group), dtype=torch.float32, device=x.device)
    offq_quantize_act_group(x, T, K, x.stride(0), g, group, OFFQ_ROTATE if rotate else 0, codes, scale, zero,
                            stream)
    return codes, scale, zero


def weight_group_sums(w_codes: torch.Tensor, N: int, K: int, group: int = GROUP, stream=None) -> torch.Tensor:
    """Integer row sums of the weight codes per activation group, [K/group, N] float32."""
    sums = torch.empty((K // group, N), dtype=torch.float32, device=w_codes.device)
    offq_weight_group_sums(w_codes, N, K, group, sums, stream)
    return sums


def w4a4_linear_group(a_codes: torch.Tensor, a_scale: torch.Tensor, a_zero: torch.Tensor,
                      w_codes: torch.Tensor, w_scale: torch.Tensor, w_groupsum: torch.Tensor,
                      group: int = GROUP, out_dtype: torch.dtype = torch.bfloat16,
                      out: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    T = a_scale.shape[0]
    K = a_codes.shape[1] * 2
    N = w_scale.shape[0]
    if out is None:
        out = torch.empty((T, N), dtype=out_dtype, device=a_codes.device)
    offq_w4a4_linear_group(a_codes, a_scale, a_zero, T, N, K, group, w_codes, w_scale, w_groupsum, out,
                           out.stride(0), stream)
    return out


def kv4_quantize_rotated(kv: torch.Tensor, rot: torch.Tensor, offset: bool = True,
                         stream=None) -> Tuple[torch.Tensor, torch.Tensor, torch.Tensor]:
    """Key-cache codes, scales and offsets of kv [T, H, hd] under per-head rotations rot [H, hd, hd]."""
    T, H, hd = kv.shape
    if kv.stride(2) != 1 or kv.stride(1) != hd:
        raise ValueError("heads of a token must be contiguous")
    codes = torch.empty((T, H, hd // 2), dtype=torch.uint8, device=kv.device)
    scale = torch.empty((T, H), dtype=torch.float32, device=kv.device)
    off = torch.empty((T, H), dtype=torch.float32, device=kv.device)
    offq_kv4_quantize_rotated(kv, T, H, hd, kv.stride(0), rot.contiguous(), OFFQ_OFFSET if offset else 0, codes,
                              scale, off, stream)
    return codes, scale, off


def rotate_heads(x: torch.Tensor, rot: torch.Tensor, out_dtype: torch.dtype = torch.float32,
                 stream=None) -> torch.Tensor:
    """x [T, H, hd] rotated per head by rot [H, hd, hd] (y = x rot[h])."""
    T, H, hd = x.shape
    if x.stride(2) != 1 or x.stride(1) != hd:
        raise ValueError("heads of a token must be contiguous")
    out = torch.empty((T, H, hd), dtype=out_dtype, device=x.device)
    offq_rotate_heads(x, T, H, hd, x.stride(0), rot.contiguous(), out, out.stride(0), stream)
    return out


KEY_ROTATION_BYTES = 98304  # OFFQ_KEY_ROTATION_BYTES: one head's prepared rotation


def prepare_key_rotation(rot: torch.Tensor, stream=None) -> torch.Tensor:
    """rot [H, hd, hd] float32 -> the prepared image [H, KEY_ROTATION_BYTES] (uint8)."""
    H, hd, _ = rot.shape
    prep = torch.empty((H, KEY_ROTATION_BYTES), dtype=torch.uint8, device=rot.device)
    offq_prepare_key_rotation(rot.contiguous(), H, hd, prep, stream)
    return prep


def kv4_quantize_prepared(kv: torch.Tensor, prepared: torch.Tensor, offset: bool = True,
                          stream=None) -> Tuple[torch.Tensor, torch.Tensor, torch.Tensor]:
    """kv4_quantize_rotated for bf16 kv [T, H, hd] with M given as prepare_key_rotation's image."""
    T, H, hd = kv.shape
    if kv.stride(2) != 1 or kv.stride(1) != hd:
        raise ValueError("heads of a token must be contiguous")
    codes = torch.empty((T, H, hd // 2), dtype=torch.uint8, device=kv.device)
    scale = torch.empty((T, H), dtype=torch.float32, device=kv.device)
    off = torch.empty((T, H), dtype=torch.float32, device=kv.device)
    offq_kv4_quantize_prepared(kv, T, H, hd, kv.stride(0), prepared, OFFQ_OFFSET if offset else 0, codes, scale,
                               off, stream)
    return codes, scale, off


def rotate_heads_prepared(x: torch.Tensor, prepared: torch.Tensor, out_dtype: torch.dtype = torch.float32,
                          stream=None) -> torch.Tensor:
    """rotate_heads for bf16 x [T, H, hd] with M given as prepare_key_rotation's image."""
    T, H, hd = x.shape
    if x.stride(2) != 1 or x.stride(1) != hd:
        raise ValueError("heads of a token must be contiguous")
    out = torch.empty((T, H, hd), dtype=out_dtype, device=x.device)
    offq_rotate_heads_prepared(x, T, H, hd, x.stride(0), prepared, out, out.stride(0), stream)
    return out


KEY_REFLECTION_BYTES = 37376  # OFFQ_KEY_REFLECTION_BYTES: one head's structured rotation


def prepare_key_reflection(v: torch.Tensor, perm: torch.Tensor, device=None) -> torch.Tensor:
    """Top-1 directions v [H, hd] and permutations perm [H, hd] -> the structured
    image [H, KEY_REFLECTION_BYTES] (uint8), built on the host and copied to `device`."""
    H, hd = v.shape
    vh = v.detach().to("cpu", torch.float32).contiguous()
    ph = perm.detach().to("cpu", torch.int32).contiguous()
    img = torch.empty((H, KEY_REFLECTION_BYTES), dtype=torch.uint8)
    offq_prepare_key_reflection(vh, ph, H, hd, img)
    return img.to(device) if device is not None else img


def kv4_quantize_reflected(kv: torch.Tensor, prepared: torch.Tensor, offset: bool = True,
                           stream=None) -> Tuple[torch.Tensor, torch.Tensor, torch.Tensor]:
    """Key-cache codes, scales and offsets of bf16 kv [T, H, hd] under the structured M = U3 P3 H3."""
    T, H, hd = kv.shape
    if kv.stride(2) != 1 or kv.stride(1) != hd:
        raise ValueError("heads of a token must be contiguous")
    codes = torch.empty((T, H, hd // 2), dtype=torch.uint8, device=kv.device)
    scale = torch.empty((T, H), dtype=torch.float32, device=kv.device)
    off = torch.empty((T, H), dtype=torch.float32, device=kv.device)
    offq_kv4_quantize_reflected(kv, T, H, hd, kv.stride(0), prepared, OFFQ_OFFSET if offset else 0, codes, scale,
                                off, stream)
    return codes, scale, off


def rotate_heads_reflected(x: torch.Tensor, prepared: torch.Tensor, out_dtype: torch.dtype = torch.float32,
                           stream=None) -> torch.Tensor:
    """bf16 x [T, H, hd] rotated per head by the structured M = U3 P3 H3."""
    T, H, hd = x.shape
    if x.stride(2) != 1 or x.stride(1) != hd:
        raise ValueError("heads of a token must be contiguous")
    out = torch.empty((T, H, hd), dtype=out_dtype, device=x.device)
    offq_rotate_heads_reflected(x, T, H, hd, x.stride(0), prepared, out, out.stride(0), stream)
    return out


# ---------------------------------------------------------------------------
# Offline transform builder
# ---------------------------------------------------------------------------

def top1_tokens(x: torch.Tensor, stream=None) -> Tuple[torch.Tensor, torch.Tensor]:
    """x [S, L, D] (contiguous tokens): per sequence the token of largest L-inf norm."""
    S, L, D = x.shape
    if x.stride(2) != 1:
        raise ValueError("channels must be contiguous")
    index = torch.empty((S,), dtype=torch.int32, device=x.device)
    rows = torch.empty((S, D), dtype=torch.float32, device=x.device)
    _check("offq_top1_tokens", load_library().offq_top1_tokens(
        _ptr(x), _dtype_code(x), S, L, D, x.stride(1), x.stride(0), _ptr(index), _ptr(rows), _stream(stream)))
    return index, rows


def top1_direction(X: torch.Tensor, iters: int = 100, v0: Optional[torch.Tensor] = None,
                   stream=None) -> Tuple[torch.Tensor, torch.Tensor]:
    """Leading eigenvector of X^T X / N by power iteration (and X v)."""
    N, D = X.shape
    X = X.contiguous()
    if v0 is None:
        v0 = torch.ones((D,), dtype=torch.float32, device=X.device)
    v = torch.empty((D,), dtype=torch.float32, device=X.device)
    proj = torch.empty((N,), dtype=torch.float32, device=X.device)
    _check("offq_top1_direction", load_library().offq_top1_direction(
        _ptr(X), N, D, iters, _ptr(v0.contiguous()), _ptr(v), _ptr(proj), _stream(stream)))
    return v, proj


def reflect_rows(A: torch.Tensor, v: torch.Tensor, stream=None) -> torch.Tensor:
    R, D = A.shape
    out = torch.empty((R, D), dtype=torch.float32, device=A.device)
    _check("offq_reflect_rows", load_library().offq_reflect_rows(
        _ptr(A.contiguous()), R, D, _ptr(v), _ptr(out), _stream(stream)))
    return out


def column_absmax(A: torch.Tensor, stream=None) -> torch.Tensor:
    R, D = A.shape
    mag = torch.empty((D,), dtype=torch.float32, device=A.device)
    _check("offq_column_absmax", load_library().offq_column_absmax(
        _ptr(A.contiguous()), R, D, _ptr(mag), _stream(stream)))
    return mag


def sorted_grouping(mag: torch.Tensor, G: int) -> torch.Tensor:
    """Host call: the sorted-grouping permutation (int32, on the host)."""
    m = mag.detach().to("cpu", torch.float32).contiguous()
    perm = torch.empty((m.numel(),), dtype=torch.int32)
    _check("offq_sorted_grouping", load_library().offq_sorted_grouping(
        ctypes.c_void_p(m.data_ptr()), m.numel(), G, ctypes.c_void_p(perm.data_ptr())))
    return perm


def fuse_rotation(W: torch.Tensor, v: torch.Tensor, perm: torch.Tensor, g: int, stream=None) -> torch.Tensor:
    N, D = W.shape
    out = torch.empty((N, D), dtype=torch.float32, device=W.device)
    _check("offq_fuse_rotation", load_library().offq_fuse_rotation(
        _ptr(W.contiguous()), N, D, _ptr(v), _ptr(perm.to(W.device, torch.int32).contiguous()), g, _ptr(out),
        _stream(stream)))
    return out


# ---------------------------------------------------------------------------
# MXFP4 residuals with the offset as zero-point
# ---------------------------------------------------------------------------

def offq_quantize_act_mx(x: torch.Tensor, T: int, K: int, ldx: int, g: int, flags: int, codes: torch.Tensor,
                         shifts: torch.Tensor, row_scale: torch.Tensor, offset: Optional[torch.Tensor],
                         stream=None) -> None:
    _check("offq_quantize_act_mx", load_library().offq_quantize_act_mx(
        _ptr(x), _dtype_code(x), T, K, ldx, g, flags, _ptr(codes), _ptr(shifts), _ptr(row_scale), _ptr(offset),
        _stream(stream)))


def offq_prepare_weight_mx(w: torch.Tensor, N: int, K: int, g: int, rotate: int, w_codes: torch.Tensor,
                           w_shifts: torch.Tensor, w_scale: torch.Tensor, w_offsum: torch.Tensor,
                           stream=None) -> None:
    _check("offq_prepare_weight_mx", load_library().offq_prepare_weight_mx(
        _ptr(w), _dtype_code(w), N, K, g, rotate, _ptr(w_codes), _ptr(w_shifts), _ptr(w_scale), _ptr(w_offsum),
        _stream(stream)))


def offq_mx_linear(a_codes, a_shifts, a_scale, a_offset, T: int, N: int, K: int, g: int, w_codes, w_shifts,
                   w_scale, w_offsum, out: torch.Tensor, ldo: int, stream=None) -> None:
    _check("offq_mx_linear", load_library().offq_mx_linear(
        _ptr(a_codes), _ptr(a_shifts), _ptr(a_scale), _ptr(a_offset), T, N, K, g, _ptr(w_codes), _ptr(w_shifts),
        _ptr(w_scale), _ptr(w_offsum), _ptr(out), _dtype_code(out), ldo, _stream(stream)))


def mx_shift_bytes(R: int, K: int) -> int:
    return load_library().offq_mx_shift_bytes(R, K)


def quantize_act_mx(x: torch.Tensor, g: int, rotate: bool = True, offset: bool = True):
    """Allocating wrapper: (codes, shifts, row_scale, offset) for rows x [T, K]."""
    T, K = x.shape
    dev = x.device
    codes = torch.empty((padded_rows(T), K // 2), dtype=torch.uint8, device=dev)
    shifts = torch.empty((mx_shift_bytes(T, K),), dtype=torch.uint8, device=dev)
    scale = torch.empty((T,), dtype=torch.float32, device=dev)
    off = torch.empty((T, K // g), dtype=torch.float32, device=dev)
    flags = (OFFQ_ROTATE if rotate else 0) | (OFFQ_OFFSET if offset else 0)
    offq_quantize_act_mx(x, T, K, x.stride(0), g, flags, codes, shifts, scale, off)
    return codes, shifts, scale, off


def prepare_weight_mx(w: torch.Tensor, g: int, rotate: bool = True):
    """Allocating wrapper: (codes, shifts, scale, offsum) for weights w [N, K]."""
    N, K = w.shape
    dev = w.device
    codes = torch.empty((padded_rows(N), K // 2), dtype=torch.uint8, device=dev)
    shifts = torch.empty((mx_shift_bytes(N, K),), dtype=torch.uint8, device=dev)
    scale = torch.empty((N,), dtype=torch.float32, device=dev)
    offsum = torch.empty((K // g, N), dtype=torch.float32, device=dev)
    offq_prepare_weight_mx(w.contiguous(), N, K, g, 1 if rotate else 0, codes, shifts, scale, offsum)
    return codes, shifts, scale, offsum
