"""The bounded waits' failure path, on the GPU, without a fault.

The persistent row quantizers stage rows in shared memory by bulk copies and
wait for them with a bounded wait. With a test budget set by
offq_set_wait_cycles, those waits act as waits for a flag that nothing sets
and give up after a few cycles: the kernel must let the copies in flight land,
return, and leave OFFQ_ERR_TIMEOUT in the device status word, which
offq_get_device_status reports once and clears. With the default budget restored, the same call must then produce the
oracle's codes on the same device and context, with a clean status."""

import numpy as np
import pytest
import torch

import oracle as O
import workloads as W
from paper_2606_07116_gb300 import build as B
from paper_2606_07116_gb300 import offq as Q
from parity import act_q, check_codes, check_scales, code_window, tensor_core_form

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    B.build()
    Q.load_library()


@pytest.mark.parametrize("T,K,g,rotate", [
    (4096, 2048, 1024, True),    # the warp-per-block kernel of g = 1024 with the rotation
    (8192, 2048, 512, True),     # the ring form of the block-Hadamard kernel (g <= 1024)
    (2048, 8192, 4096, True),    # the ring form of the wide kernel (g >= 2048)
    (8192, 4096, 4096, False),   # the shared-memory ring kernel of rotation-free rows (per-warp rings)
    (2048, 14336, 1024, True),   # the tensor-core form of g = 1024 (its register warps' wait for the MMAs)
])
def test_shortened_wait_times_out_and_the_device_recovers(T, K, g, rotate):
    x = torch.from_numpy(W.activations(T, K, seed=T + K, n_out=3, mult=80.0)).to(torch.bfloat16)
    xd = x.cuda()
    flags = (Q.OFFQ_ROTATE if rotate else 0) | Q.OFFQ_OFFSET
    codes = torch.empty((Q.padded_rows(T), K // 2), dtype=torch.uint8, device="cuda")
    scale = torch.empty((T,), dtype=torch.float32, device="cuda")
    off = torch.empty((T, K // g), dtype=torch.float32, device="cuda")
    assert Q.offq_get_device_status() == Q.OFFQ_OK
    Q.offq_set_wait_cycles(1)
    try:
        Q.offq_quantize_act(xd, T, K, K, g, flags, codes, scale, off)
        torch.cuda.synchronize()
    finally:
        Q.offq_set_wait_cycles(0)
    assert Q.offq_get_device_status() == Q.OFFQ_ERR_TIMEOUT
    assert Q.offq_get_device_status() == Q.OFFQ_OK   # read once, then cleared

    Q.offq_quantize_act(xd, T, K, K, g, flags, codes, scale, off)
    torch.cuda.synchronize()
    assert Q.offq_get_device_status() == Q.OFFQ_OK
    rows = np.unique(np.concatenate([W.unit_index_sample(T, 64, seed=3), [0, T - 1]]))
    x64 = x.to(torch.float64).numpy()[rows]
    ref = O.quantize_act(x64, g, rotate=rotate, offset=True)
    tc = tensor_core_form(x, g, rotate)
    window = code_window(ref["scale"], x64, g, tc) if tc else None
    check_codes(act_q(codes, T, K)[rows], ref["q"], ref["residual"], ref["scale"], window=window)
    check_scales(scale.cpu().numpy()[rows], ref["scale"], x64, g, rotate, tc=tc)


def test_wait_budget_argument_checks():
    lib = Q.load_library()
    assert lib.offq_set_wait_cycles(-1) == Q.OFFQ_ERR_INVALID_ARG
    assert lib.offq_set_wait_cycles(0) == Q.OFFQ_OK


def test_shortened_wait_times_out_in_the_mx_quantizer():
    """The persistent MXFP4 quantizer (warp per 1024 channels) under the same test budget."""
    T, K, g = 4096, 2048, 1024
    x = torch.from_numpy(W.activations(T, K, seed=77, n_out=3, mult=80.0)).to(torch.bfloat16)
    xd = x.cuda()
    assert Q.offq_get_device_status() == Q.OFFQ_OK
    Q.offq_set_wait_cycles(1)
    try:
        codes, shifts, scale, off = Q.quantize_act_mx(xd, g, rotate=True, offset=True)
        torch.cuda.synchronize()
    finally:
        Q.offq_set_wait_cycles(0)
    assert Q.offq_get_device_status() == Q.OFFQ_ERR_TIMEOUT
    assert Q.offq_get_device_status() == Q.OFFQ_OK
    codes, shifts, scale, off = Q.quantize_act_mx(xd, g, rotate=True, offset=True)
    torch.cuda.synchronize()
    assert Q.offq_get_device_status() == Q.OFFQ_OK
    rows = np.unique(np.concatenate([W.unit_index_sample(T, 32, seed=4), [0, T - 1]]))
    ref = O.quantize_act_mx(x.to(torch.float64).numpy()[rows], g, rotate=True, offset=True)
    np.testing.assert_allclose(off.cpu().numpy()[rows], ref["offset"], rtol=1e-6)
    xlo = np.round(np.log2(scale.cpu().numpy()[rows].astype(np.float64)))
    assert np.all(np.abs(xlo - (ref["xmax"] - O.MX_SPAN)) <= 1)

