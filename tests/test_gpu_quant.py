"""GPU parity of the row quantizers (offq_quantize_act, offq_kv4_quantize,
offq_prepare_weight) against the float64 oracle, on seeded synthetic inputs."""

import math

import numpy as np
import pytest
import torch

import oracle as O
import workloads as W
from paper_2606_07116_gb300 import build as B
from paper_2606_07116_gb300 import offq as Q
from parity import act_q, check_codes, check_offsets, check_scales, code_window, tensor_core_form, weight_q

pytestmark = pytest.mark.gpu

TORCH_DT = {"bf16": torch.bfloat16, "f16": torch.float16, "f32": torch.float32}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    B.build()
    Q.load_library()


def _host(x32: np.ndarray, dt: str) -> torch.Tensor:
    """The input as the kernel sees it, made on the CPU (RNE cast)."""
    return torch.from_numpy(np.ascontiguousarray(x32)).to(TORCH_DT[dt])


def _quant_and_check(x_host: torch.Tensor, g: int, rotate: bool, offset: bool, rows=None, ldx=None):
    T, K = x_host.shape
    tc = tensor_core_form(x_host, g, rotate, ldx)
    if ldx is None:
        xd = x_host.cuda()
    else:
        buf = torch.zeros((T, ldx), dtype=x_host.dtype)
        buf[:, :K] = x_host
        xd = buf.cuda()[:, :K]
    codes, scale, off = Q.quantize_act(xd, g, rotate=rotate, offset=offset)
    torch.cuda.synchronize()
    assert Q.offq_get_device_status() == Q.OFFQ_OK
    x64 = x_host.to(torch.float64).numpy()
    sel = np.arange(T) if rows is None else rows
    ref = O.quantize_act(x64[sel], g, rotate=rotate, offset=offset)
    q_gpu = act_q(codes, T, K)[sel]
    window = code_window(ref["scale"], x64[sel], g, tc) if tc else None
    nmis = check_codes(q_gpu, ref["q"], ref["residual"], ref["scale"], window=window)
    check_scales(scale.cpu().numpy()[sel], ref["scale"], x64[sel], g, rotate, tc=tc)
    o = off.cpu().numpy()[sel]
    if offset:
        check_offsets(o, ref["offset"], x64[sel], g, rotate)
    else:
        assert np.all(o == 0.0)
    return nmis


@pytest.mark.parametrize("g", [32, 64, 128, 256, 512, 1024, 2048, 4096, 8192])
@pytest.mark.parametrize("G", [1, 3])
def test_quantize_every_block_size(g, G):
    T = 37
    x = W.activations(T, g * G, seed=100 + g + G, n_out=2, mult=50.0)
    _quant_and_check(_host(x, "bf16"), g, True, True)


@pytest.mark.parametrize("dt", ["bf16", "f16", "f32"])
@pytest.mark.parametrize("rotate,offset", [(True, True), (True, False), (False, True), (False, False)])
def test_quantize_flags_and_dtypes(dt, rotate, offset):
    x = W.activations(29, 512, seed=7, n_out=2, mult=30.0)
    _quant_and_check(_host(x, dt), 256, rotate, offset)


@pytest.mark.parametrize("T,K,g,dist", [
    (16, 512, 512, "normal"),          # toy layer (fp32 in the workload; bf16 here)
    (64, 11008, 256, "normal"),        # down-proj input, 43 blocks
    (48, 14336, 1024, "student_t3"),   # Llama-3-8B down-proj input, 14 blocks
    (8, 28672, 1024, "normal"),        # Llama-2-70B down-proj input, 28 blocks
    (40, 8192, 8192, "normal"),        # Llama-2-70B hidden
])
def test_quantize_workload_shapes(T, K, g, dist):
    x = W.activations(T, K, seed=11, dist=dist, n_out=4, mult=100.0)
    _quant_and_check(_host(x, "bf16"), g, True, True)


def _device_rows(T, K, dist, n_out, mult, seed):
    """A full prefill input drawn on the host from the workload recipe, bf16."""
    return _host(W.activations(T, K, seed=seed, dist=dist, n_out=n_out, mult=mult), "bf16")


@pytest.mark.parametrize("T,K,g,rotate,dist,n_out,mult", [
    (8192, 8192, 8192, False, "normal", 6, 200.0),       # Llama-2-70B attention / MLP input
    (8192, 28672, 1024, True, "normal", 6, 200.0),       # Llama-2-70B down-proj input, 28 blocks
    (4096, 14336, 1024, True, "student_t3", 3, 100.0),   # Llama-3-8B down-proj input, 14 blocks
])
def test_quantize_config_sites_sampled(T, K, g, rotate, dist, n_out, mult):
    """The bench's prefill launches at full size, checked on sampled rows (first and last included)."""
    rows = np.unique(np.concatenate([W.unit_index_sample(T, 96, seed=K % 89), [0, T - 1]]))
    _quant_and_check(_device_rows(T, K, dist, n_out, mult, seed=K + 3), g, rotate, True, rows=rows)


@pytest.mark.parametrize("K,dt", [(1024, "bf16"), (4096, "bf16"), (4096, "f16"), (4096, "f32"), (8192, "bf16"),
                                  (8192, "f32")])
@pytest.mark.parametrize("offset", [True, False])
def test_quantize_whole_row_block_without_rotation(K, dt, offset):
    """One offset block per row and no rotation (the q/k/v, o and gate/up sites); 45 rows leave
    warps without a row. Rows up to 24 KB take the shared-memory ring kernel; K = 8192 fp32 rows
    take the register kernel's two-sweep path."""
    x = W.activations(45, K, seed=31 + K, n_out=4, mult=100.0)
    _quant_and_check(_host(x, dt), K, False, offset)


@pytest.mark.parametrize("T,K,dt", [(40000, 1024, "bf16"), (5003, 8192, "bf16"), (4099, 4096, "f32")])
def test_quantize_whole_row_many_rows_per_warp(T, K, dt):
    """Enough rows that every warp of the persistent ring kernel quantizes several, so each slot
    is refilled and its barrier phase flips more than once; checked on sampled rows including
    the first and the last."""
    x = W.activations(T, K, seed=57 + K, n_out=4, mult=100.0)
    rows = np.unique(np.concatenate([W.unit_index_sample(T, 384, seed=5), [0, 1, T - 2, T - 1]]))
    _quant_and_check(_host(x, dt), K, False, True, rows=rows)


@pytest.mark.parametrize("g", [32, 64, 128, 256, 512, 1024, 2048, 4096, 8192])
@pytest.mark.parametrize("G", [1, 3])
def test_quantize_persistent_ring(g, G):
    """Enough rows (about 2^24 channels) that the row groups outnumber the SMs, so the
    persistent form stages each CTA's groups through its shared-memory slot; sampled rows,
    including the first and the last, against the oracle."""
    K = g * G
    T = max(700, 2 ** 24 // K)
    x = W.activations(T, K, seed=300 + g + G, n_out=3, mult=80.0)
    rows = np.unique(np.concatenate([W.unit_index_sample(T, 160, seed=9), [0, 1, T - 2, T - 1]]))
    _quant_and_check(_host(x, "bf16"), g, True, True, rows=rows)


@pytest.mark.parametrize("dt,ld_pad", [("f32", 0), ("bf16", 64), ("f16", 0)])
def test_quantize_persistent_ring_dtypes_and_stride(dt, ld_pad):
    """The persistent form on the down-proj shape (43 blocks of 256) with fp32 / fp16 rows, and
    with padded rows that take one bulk copy per row."""
    T, K, g = 1600, 11008, 256
    x = W.activations(T, K, seed=41, n_out=4, mult=100.0)
    rows = np.unique(np.concatenate([W.unit_index_sample(T, 160, seed=10), [0, T - 1]]))
    _quant_and_check(_host(x, dt), g, True, True, rows=rows, ldx=(K + ld_pad) if ld_pad else None)


@pytest.mark.parametrize("T,K,dt,ld_pad,offset", [
    (1700, 5120, "f32", 0, True),      # 5 blocks, one row per CTA and one slot of fp32 rows
    (900, 14336, "f16", 0, True),      # Llama-3-8B down-proj width: two rows of 14 warps per CTA
    (3001, 2048, "bf16", 64, True),    # padded rows (one bulk copy per row), a ragged last group
    (4500, 1024, "bf16", 0, False),    # 28 rows of one block per CTA, no offsets
    (760, 28672, "bf16", 0, False),    # Llama-2-70B down-proj width, no offsets
])
def test_quantize_warp_per_block_kernel(T, K, dt, ld_pad, offset):
    """The persistent g = 1024 kernel (a warp per block, rows held in registers) across dtypes,
    row counts per CTA, padded rows and the offset flag; sampled rows including the first and
    the last."""
    x = W.activations(T, K, seed=61 + K, n_out=4, mult=100.0)
    rows = np.unique(np.concatenate([W.unit_index_sample(T, 160, seed=12), [0, 1, T - 2, T - 1]]))
    _quant_and_check(_host(x, dt), 1024, True, offset, rows=rows, ldx=(K + ld_pad) if ld_pad else None)


@pytest.mark.parametrize("T,K,g,rotate", [
    (300, 32768, 1024, True),    # the largest K, 32 blocks of 1024: past the warp-per-block kernel's 28
    (40, 32768, 32768 // 4, False),  # the largest K without rotation, 4 offset blocks
    (33, 32768, 32768 // 4, True),   # the largest K with the widest rotation block (8192)
])
def test_quantize_maximum_k(T, K, g, rotate):
    x = W.activations(T, K, seed=83 + T, n_out=4, mult=100.0)
    rows = np.unique(np.concatenate([W.unit_index_sample(T, 48, seed=14), [0, T - 1]]))
    _quant_and_check(_host(x, "bf16"), g, rotate, True, rows=rows)


def test_quantize_toy_fp32():
    w = W.WORKLOADS["toy"]
    x = W.layer_inputs(w, w.layers[0])
    _quant_and_check(_host(x, "f32"), 512, True, True)


def test_quantize_full_llama2_7b_sampled():
    """Full 2048 x 4096 bf16 launch, checked on 256 sampled rows."""
    x = W.activations(2048, 4096, seed=0, n_out=4, mult=100.0)
    rows = W.unit_index_sample(2048, 256, seed=3)
    _quant_and_check(_host(x, "bf16"), 4096, True, True, rows=rows)


def test_quantize_strided_rows():
    x = W.activations(21, 1024, seed=12, n_out=1, mult=20.0)
    _quant_and_check(_host(x, "bf16"), 1024, True, True, ldx=1024 + 64)


@pytest.mark.parametrize("G,extra,offset,ld_pad", [
    (1, 37, True, 0),      # 64 tokens of one block per tile, a ragged last tile
    (2, 5, True, 64),      # padded rows
    (3, 0, True, 0),       # 21 tokens x 3 blocks: 63 of a half's 64 rows
    (5, 11, False, 0),     # no offsets
    (14, 3, True, 0),      # Llama-3-8B down-proj width
    (28, 1, False, 8),     # Llama-2-70B down-proj width, pitch K + 8
    (32, 1, True, 0),      # the largest K (32768): 2 tokens per tile
])
def test_quantize_tensor_core_form(G, extra, offset, ld_pad):
    """The tensor-core form of g = 1024 (bf16 rows, at least one tile per SM) across block
    counts per row, tile fill, ragged last tiles, padded rows and the offset flag; sampled
    rows plus every row of the first and the last tile."""
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    P = 64 // G
    T, K = sms * P + extra, 1024 * G
    x = _host(W.activations(T, K, seed=90 + G, n_out=4, mult=100.0), "bf16")
    ldx = K + ld_pad if ld_pad else None
    assert tensor_core_form(x, 1024, True, ldx)
    last0 = (T - 1) // P * P
    rows = np.unique(np.concatenate([W.unit_index_sample(T, 96, seed=G), np.arange(P), np.arange(last0, T)]))
    _quant_and_check(x, 1024, True, offset, rows=rows, ldx=ldx)


def test_quantize_tensor_core_form_degenerate_rows():
    """Zero rows, rows whose only nonzero channels lead their blocks (zero residual), a unit
    channel, a constant row and one large value, inside a launch that takes the tensor cores."""
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    G = 4
    T, K = sms * 16, 4096
    x = W.activations(T, K, seed=17, n_out=2, mult=40.0).astype(np.float32)
    x[0] = 0.0
    x[1] = 0.0
    x[1, ::1024] = [3.0, -250.0, 0.5, 8192.0]
    x[2] = 0.0
    x[2, 1024 + 77] = 1.0
    x[3] = 2.5
    x[T - 1, 4000] = 3e4
    xh = _host(x, "bf16")
    assert tensor_core_form(xh, 1024, True)
    codes, scale, off = Q.quantize_act(xh.cuda(), 1024)
    torch.cuda.synchronize()
    q = act_q(codes, T, K)
    assert np.all(q[0] == 0) and scale[0].item() == 0.0 and np.all(off[0].cpu().numpy() == 0.0)
    assert np.all(q[1] == 0) and scale[1].item() == 0.0
    np.testing.assert_array_equal(off[1].cpu().numpy(), np.array([3.0, -250.0, 0.5, 8192.0]) / 32.0)
    H = O.sylvester_hadamard(1024)
    np.testing.assert_array_equal(q[2, 1024:2048], 7 * H[77])
    assert np.all(q[2, :1024] == 0) and np.all(q[2, 2048:] == 0)
    # A constant block c rotates to (32 c, 0, ..., 0): residual 32 c - c / 32 at channel 0.
    assert np.all(q[3, ::1024] == 7) and np.count_nonzero(q[3]) == 4
    rows = np.unique(np.concatenate([np.arange(8), W.unit_index_sample(T, 32, seed=5), [T - 1]]))
    _quant_and_check(xh, 1024, True, True, rows=rows)


def test_quantize_degenerate_rows():
    g, G = 256, 2
    x = W.activations(6, g * G, seed=13)
    x[0] = 0.0                                   # all-zero row: scale 0, codes 0
    x[1] = 0.0
    x[1, 0], x[1, g] = 123.0, -7.5               # only the block-leading channels: zero residual
    x[2, :] = 0.0
    x[2, 5] = 1.0                                # one unit channel
    xh = _host(x, "f32")
    codes, scale, off = Q.quantize_act(xh.cuda(), g)
    torch.cuda.synchronize()
    q = act_q(codes, 6, g * G)
    assert np.all(q[0] == 0) and scale[0].item() == 0.0 and np.all(off[0].cpu().numpy() == 0.0)
    assert np.all(q[1] == 0) and scale[1].item() == 0.0
    np.testing.assert_allclose(off[1].cpu().numpy(), [123.0 / math.sqrt(g), -7.5 / math.sqrt(g)], rtol=3e-7)
    H = O.sylvester_hadamard(g)
    np.testing.assert_array_equal(q[2, :g], 7 * H[5])   # x = e_5 rotates to H[5] / sqrt(g)
    np.testing.assert_array_equal(q[2, g:], 0)
    _quant_and_check(xh, g, True, True)


def test_quantize_exact_ties_round_half_even():
    """Without rotation and offset, scale 1 and half-integer inputs: ties resolve to even, bit-exact."""
    row = np.array([7.0, -7.0, 0.5, 1.5, 2.5, 3.5, -0.5, -1.5, -2.5, -3.5, 4.5, -4.5, 5.5, 6.5, -5.5, -6.5]
                   * 2, dtype=np.float32)
    x = np.tile(row, (5, 2))
    codes, scale, _ = Q.quantize_act(torch.from_numpy(x).cuda(), 32, rotate=False, offset=False)
    torch.cuda.synchronize()
    q = act_q(codes, x.shape[0], x.shape[1])
    ref = O.quantize_act(x.astype(np.float64), 32, rotate=False, offset=False)
    np.testing.assert_array_equal(q, ref["q"])
    np.testing.assert_array_equal(scale.cpu().numpy(), 1.0)
    assert list(q[0, :16]) == [7, -7, 0, 2, 2, 4, 0, -2, -2, -4, 4, -4, 6, 6, -6, -6]


def test_quantize_single_token():
    x = W.activations(1, 4096, seed=14, n_out=4, mult=100.0)
    _quant_and_check(_host(x, "bf16"), 4096, True, True)


# --------------------------------------------------------------------------
# KV4
# --------------------------------------------------------------------------

@pytest.mark.parametrize("T,H", [(1, 32), (5, 32), (64, 32), (33, 8)])
@pytest.mark.parametrize("flags", [3, 2])
def test_kv4_against_oracle(T, H, flags):
    hd = 128
    kv = W.kv_heads(T, H, hd, seed=2 + T)
    kvh = _host(kv.reshape(T, H * hd), "bf16").reshape(T, H, hd)
    rotate = bool(flags & 1)
    codes, scale, off = Q.kv4_quantize(kvh.cuda(), rotate=rotate, offset=True)
    torch.cuda.synchronize()
    ref = O.kv4_quantize(kvh.to(torch.float64).numpy(), rotate=rotate, offset=True)
    q = O.unpack_act_codes(codes.cpu().numpy())
    check_codes(q.reshape(T * H, hd), ref["q"].reshape(T * H, hd), ref["residual"].reshape(T * H, hd),
                ref["scale"].reshape(T * H))
    x64 = kvh.to(torch.float64).numpy().reshape(T * H, hd)
    check_scales(scale.cpu().numpy().reshape(-1), ref["scale"].reshape(-1), x64, hd, rotate)
    check_offsets(off.cpu().numpy().reshape(-1, 1), ref["offset"].reshape(-1, 1), x64, hd, rotate)


def test_kv4_llama2_70b_prefill():
    """KV4 of the Llama-2-70B keys and values at prefill size: 8192 tokens x 8 heads x 128, every
    (token, head) checked, with and without the per-head Hadamard."""
    T, H, hd = 8192, 8, 128
    kv = W.kv_heads(T, H, hd, seed=81)
    kvh = _host(kv.reshape(T, H * hd), "bf16").reshape(T, H, hd)
    x64 = kvh.to(torch.float64).numpy()
    for rotate in (True, False):
        codes, scale, off = Q.kv4_quantize(kvh.cuda(), rotate=rotate, offset=True)
        torch.cuda.synchronize()
        assert Q.offq_get_device_status() == Q.OFFQ_OK
        ref = O.kv4_quantize(x64, rotate=rotate, offset=True)
        q = O.unpack_act_codes(codes.cpu().numpy())
        check_codes(q.reshape(T * H, hd), ref["q"].reshape(T * H, hd), ref["residual"].reshape(T * H, hd),
                    ref["scale"].reshape(T * H))
        check_scales(scale.cpu().numpy().reshape(-1), ref["scale"].reshape(-1), x64.reshape(T * H, hd), hd, rotate)
        check_offsets(off.cpu().numpy().reshape(-1, 1), ref["offset"].reshape(-1, 1), x64.reshape(T * H, hd), hd,
                      rotate)


def test_kv4_padded_token_stride():
    T, H, hd = 7, 8, 128
    kv = W.kv_heads(T, H, hd, seed=9)
    host = _host(kv.reshape(T, H * hd), "bf16")
    buf = torch.zeros((T, H * hd + 256), dtype=torch.bfloat16)
    buf[:, :H * hd] = host
    dev = buf.cuda()
    codes = torch.empty((T, H, hd // 2), dtype=torch.uint8, device="cuda")
    scale = torch.empty((T, H), dtype=torch.float32, device="cuda")
    off = torch.empty((T, H), dtype=torch.float32, device="cuda")
    Q.offq_kv4_quantize(dev, T, H, hd, H * hd + 256, Q.OFFQ_ROTATE | Q.OFFQ_OFFSET, codes, scale, off)
    torch.cuda.synchronize()
    ref = O.kv4_quantize(host.to(torch.float64).numpy().reshape(T, H, hd))
    q = O.unpack_act_codes(codes.cpu().numpy()).reshape(T * H, hd)
    check_codes(q, ref["q"].reshape(T * H, hd), ref["residual"].reshape(T * H, hd), ref["scale"].reshape(-1))


# --------------------------------------------------------------------------
# Weight preparation (offline)
# --------------------------------------------------------------------------

@pytest.mark.parametrize("N,K,g,rotate", [(300, 1024, 256, True), (64, 512, 512, False), (40, 11008, 256, True),
                                          (24, 14336, 1024, True)])
def test_prepare_weight(N, K, g, rotate):
    w = W.weights(N, K, seed=21)
    wh = torch.from_numpy(w)
    codes, scale, rowsum = Q.prepare_weight(wh.cuda(), g, rotate=rotate)
    torch.cuda.synchronize()
    ref = O.prepare_weight(w.astype(np.float64), g, rotate=rotate)
    qg = weight_q(codes, N, K)
    # Padding rows of the last 32-row tile are zero bytes.
    full = codes.cpu().numpy()
    tail = O.untile_codes(full, full.shape[0], K)[N:]
    assert np.all(tail == 0)
    # Reuse the activation-path checks: weights are rows quantized without offset.
    ra = O.quantize_act(w.astype(np.float64), g, rotate=rotate, offset=False)
    check_codes(qg, ref["q"], ra["residual"], ra["scale"], what="weight codes")
    check_scales(scale.cpu().numpy(), ref["scale"], w.astype(np.float64), g, rotate, what="weight scale")
    # Row sums are exact integers of the GPU's own codes.
    np.testing.assert_array_equal(rowsum.cpu().numpy(), qg.reshape(N, K // g, g).sum(axis=2).T)
