"""GPU parity of the per-group asymmetric path (the paper's evaluated
activation setting: groups of 128, Eq. 1 with zero-points) against the oracle.

* The quantizer decides codes in fp32; the oracle evaluates Eq. 1 as written,
  in float64 (rne(y / s) + z, z = -rne(min / s)). parity.check_group_quant
  allows a code or a zero-point to differ by 1 only within TIE_WINDOW of a
  rounding tie (a flipped zero-point moves the codes clamped at the grid's
  ends), and at most 1e-4 of the codes.
* Per-group weight row sums are integers and must match exactly.
* GEMM outputs from the GPU's own codes, scales and zero-points must lie
  within the fp32 bound of the per-group chain (parity.group_terms) of the
  oracle's float64 result, plus half an ulp of a bf16 / fp16 output."""

import numpy as np
import pytest
import torch

import oracle as O
import workloads as W
from paper_2606_07116_gb300 import build as B
from paper_2606_07116_gb300 import offq as Q
from parity import act_q, check_group_quant, check_outputs, group_terms, max_rel_err_floored, weight_q

pytestmark = pytest.mark.gpu

OUT_DT = {"f32": torch.float32, "bf16": torch.bfloat16, "f16": torch.float16}
IN_DT = {"f32": torch.float32, "bf16": torch.bfloat16, "f16": torch.float16}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    B.build()
    Q.load_library()


def _quant(x_np, g, rotate, in_dt="bf16"):
    xt = torch.from_numpy(x_np).to(IN_DT[in_dt])
    codes, scale, zero = Q.quantize_act_group(xt.cuda(), g, rotate=rotate)
    torch.cuda.synchronize()
    assert Q.offq_get_device_status() == Q.OFFQ_OK
    T, K = x_np.shape
    q = act_q(codes, T, K) + 8
    return xt.to(torch.float64).numpy(), codes, scale, zero, q


@pytest.mark.parametrize("in_dt", ["f32", "bf16", "f16"])
@pytest.mark.parametrize("rotate,g", [(False, 4096), (True, 128), (True, 256), (True, 512), (True, 32)])
def test_group_quantizer_parity(in_dt, rotate, g):
    T, K = 45, 4096
    x = W.activations(T, K, seed=60, n_out=3, mult=80.0)
    xe, codes, scale, zero, q = _quant(x, g, rotate, in_dt)
    ref = O.quantize_act_group(xe, g, 128, rotate=rotate)
    check_group_quant(q, scale.cpu().numpy(), zero.cpu().numpy(), ref, xe, g, rotate)


@pytest.mark.parametrize("g", [1024, 2048, 4096, 8192])
def test_group_quantizer_rotation_across_warps(g):
    """Rotation blocks of g >= 1024 span g / 512 warps of a CTA (index bits 9.. go through shared
    memory); 37 rows leave the last CTA with items past the end, and K = 3 g blocks for g <= 4096."""
    T = 37
    K = 3 * g if g <= 4096 else g
    x = W.activations(T, K, seed=64 + g, n_out=3, mult=120.0)
    xe, codes, scale, zero, q = _quant(x, g, True)
    ref = O.quantize_act_group(xe, g, 128, rotate=True)
    check_group_quant(q, scale.cpu().numpy(), zero.cpu().numpy(), ref, xe, g, True)


def test_group_quantizer_ragged_chunk_and_offsets():
    """K = 11008 (21.5 chunks of 512) with the g = 256 rotation of the
    down-projection input, and rows with large common offsets."""
    T, K, g = 37, 11008, 256
    x = W.activations(T, K, seed=61, n_out=4, mult=150.0)
    x[::3] += 40.0
    xe, codes, scale, zero, q = _quant(x, g, True)
    ref = O.quantize_act_group(xe, g, 128, rotate=True)
    check_group_quant(q, scale.cpu().numpy(), zero.cpu().numpy(), ref, xe, g, True)


def test_group_quantizer_constant_and_zero_groups():
    T, K = 8, 512
    x = np.random.default_rng(62).standard_normal((T, K)).astype(np.float32)
    x[0] = 0.0
    x[1, 128:256] = 2.5
    xe, codes, scale, zero, q = _quant(x, 512, False, "f32")
    s, z = scale.cpu().numpy(), zero.cpu().numpy()
    assert np.all(s[0] == 0) and np.all(z[0] == 0) and np.all(q[0] == 0)
    assert s[1, 1] == 0 and z[1, 1] == 0 and np.all(q[1, 128:256] == 0)
    ref = O.quantize_act_group(xe, 512, 128, rotate=False)
    check_group_quant(q, s, z, ref, xe, 512, False)


def test_group_quantizer_empty_input():
    x = torch.zeros((0, 1024), dtype=torch.bfloat16, device="cuda")
    codes, scale, zero = Q.quantize_act_group(x, 256)
    assert scale.shape == (0, 8)


@pytest.mark.parametrize("N,K,g", [(200, 512, 512), (4096, 4096, 4096), (300, 11008, 256)])
def test_weight_group_sums_exact(N, K, g):
    w = W.weights(N, K, seed=63)
    w_codes, w_scale, _ = Q.prepare_weight(torch.from_numpy(w).cuda(), g, rotate=True)
    sums = Q.weight_group_sums(w_codes, N, K)
    torch.cuda.synchronize()
    qw = weight_q(w_codes, N, K)
    np.testing.assert_array_equal(sums.cpu().numpy(), O.weight_group_sums(qw, 128).astype(np.float32))


def _check_group_layer(T, K, N, g, out_dt, rotate, seed=0, rows=None, ldo=None, mult=60.0, x=None):
    if x is None:
        x = W.activations(T, K, seed=seed, n_out=3, mult=mult)
    w = W.weights(N, K, seed=seed + 1)
    xt = torch.from_numpy(x).to(torch.bfloat16).cuda()
    a_codes, a_scale, a_zero = Q.quantize_act_group(xt, g, rotate=rotate)
    w_codes, w_scale, _ = Q.prepare_weight(torch.from_numpy(w).cuda(), g, rotate=rotate)
    gsum = Q.weight_group_sums(w_codes, N, K)
    ldo = N if ldo is None else ldo
    out = torch.full((T, ldo), float("nan"), dtype=OUT_DT[out_dt], device="cuda")
    Q.offq_w4a4_linear_group(a_codes, a_scale, a_zero, T, N, K, 128, w_codes, w_scale, gsum, out, ldo)
    torch.cuda.synchronize()
    assert Q.offq_get_device_status() == Q.OFFQ_OK
    y = out[:, :N].float().cpu().numpy().astype(np.float64)
    sel = np.arange(T) if rows is None else rows
    q = (act_q(a_codes, T, K) + 8)[sel]
    qw = weight_q(w_codes, N, K)
    s = a_scale.cpu().numpy().astype(np.float64)[sel]
    z = a_zero.cpu().numpy().astype(np.float64)[sel]
    sw = w_scale.cpu().numpy().astype(np.float64)
    R = gsum.cpu().numpy().astype(np.float64)
    res = O.w4a4_linear_group(q, s, z, qw, sw, R, 128)
    terms = group_terms(res["P"].astype(np.float64), s, z, R, sw)
    check_outputs(y[sel], res["y"], terms, 2 * (K // 128), out_dt)
    if ldo > N:
        assert torch.isnan(out[:, N:]).all(), "columns past N were written"
    return y[sel], res["y"], x[sel], w


@pytest.mark.parametrize("out_dt", ["f32", "bf16", "f16"])
@pytest.mark.parametrize("rotate", [False, True])
def test_group_gemm_ragged(out_dt, rotate):
    """T, N off every tile size (two m-pairs, a partial n-tile), 4 groups."""
    _check_group_layer(300, 512, 200, 512, out_dt, rotate, seed=70)


@pytest.mark.parametrize("K", [128, 256])
def test_group_gemm_one_and_two_groups(K):
    """K = 128 (one group per tile: the prefetch runs two tiles ahead) and
    K = 256, over more tiles than clusters."""
    _check_group_layer(600, K, 2000, K, "bf16", False, seed=80)


def test_group_gemm_leading_dimension():
    _check_group_layer(40, 1024, 96, 256, "bf16", True, seed=71, ldo=136)


@pytest.mark.parametrize("T", [1, 8, 64])
def test_group_gemm_decode(T):
    _check_group_layer(T, 4096, 1024, 4096, "bf16", False, seed=72)


def test_group_gemm_many_tiles_f16_bound():
    """More pair tiles than clusters (persistent loop), with the 2e-3 bound of
    fp16 outputs."""
    y, y_ref, x, w = _check_group_layer(1024, 1024, 4096, 1024, "f16", False, seed=73)
    assert max_rel_err_floored(y, y_ref) <= 2e-3


def test_group_gemm_llama2_7b_gate_sampled():
    """The bench's gate projection (T = 2048, 4096 -> 11008) on sampled rows."""
    rows = np.sort(np.random.default_rng(74).choice(2048, 64, replace=False))
    y, y_ref, x, w = _check_group_layer(2048, 4096, 11008, 4096, "bf16", False, seed=75, rows=rows)
    ref = O.linear_reference(x, w)
    assert np.linalg.norm(y - ref) < 0.3 * np.linalg.norm(ref)


def test_group_gemm_llama2_7b_down_sampled():
    """The bench's down projection (T = 2048, 11008 -> 4096, rotation g = 256)."""
    rows = np.sort(np.random.default_rng(76).choice(2048, 48, replace=False))
    _check_group_layer(2048, 11008, 4096, 256, "bf16", True, seed=77, rows=rows)


def test_group_gemm_is_repeatable():
    x = W.activations(256, 1024, seed=78, n_out=2, mult=60.0)
    w = W.weights(512, 1024, seed=79)
    a = Q.quantize_act_group(torch.from_numpy(x).to(torch.bfloat16).cuda(), 1024, rotate=False)
    wc, ws, _ = Q.prepare_weight(torch.from_numpy(w).cuda(), 1024, rotate=False)
    gs = Q.weight_group_sums(wc, 512, 1024)
    y1 = Q.w4a4_linear_group(*a, wc, ws, gs)
    y2 = Q.w4a4_linear_group(*a, wc, ws, gs)
    torch.cuda.synchronize()
    assert torch.equal(y1, y2)


def test_group_gemm_zero_points_outside_the_code_range():
    """Groups that do not straddle zero have z = -rne(min/s) outside [0, 15]:
    the kernel subtracts clamp(z, 0, 15) in the operand and the rest through
    the weight group sums. Shifted groups are mixed with ordinary ones within
    each warp's 32 rows."""
    T, K, N = 300, 1024, 640
    x = W.activations(T, K, seed=90, n_out=3, mult=60.0)
    rng = np.random.default_rng(91)
    for t in range(T):
        if t % 3 == 0:
            j = rng.integers(0, K // 128)
            x[t, 128 * j:128 * (j + 1)] += rng.choice([-1.0, 1.0]) * rng.uniform(20.0, 200.0)
    x[7] = np.abs(x[7]) + 1.0                          # every group of a row positive
    x[8] = -np.abs(x[8]) - 1.0                         # every group negative
    xt = torch.from_numpy(x).to(torch.bfloat16).cuda()
    _, _, zero = Q.quantize_act_group(xt, 1024, rotate=False)
    z = zero.cpu().numpy()
    assert (z < 0).any() and (z > 15).any() and ((z >= 0) & (z <= 15)).any()
    _check_group_layer(T, K, N, 1024, "f32", False, x=x)
