"""GPU parity of the W4A4 GEMM (offq_w4a4_linear) against the oracle.

Integer accumulators must match bit for bit given identical codes; outputs
must lie within the fp32 epilogue bound (plus half an ulp of bf16/fp16) of the
oracle's float64 dequantized result from the same codes, scales and offsets."""

import numpy as np
import pytest
import torch

import oracle as O
import workloads as W
from paper_2606_07116_gb300 import build as B
from paper_2606_07116_gb300 import offq as Q
from parity import act_q, check_outputs, epilogue_terms, max_rel_err_floored, weight_q

pytestmark = pytest.mark.gpu

OUT_DT = {"f32": torch.float32, "bf16": torch.bfloat16, "f16": torch.float16}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    B.build()
    Q.load_library()


def _run_gemm(a_codes, a_scale, a_off, w_codes, w_scale, rowsum, g, out_dt, ldo=None, T=None, N=None):
    T = a_scale.shape[0] if T is None else T
    N = w_scale.shape[0] if N is None else N
    ldo = N if ldo is None else ldo
    out = torch.full((T, ldo), float("nan"), dtype=OUT_DT[out_dt], device="cuda")
    acc = torch.zeros((T, N), dtype=torch.int32, device="cuda")
    K = a_codes.shape[1] * 2
    Q.offq_w4a4_linear(a_codes, a_scale, a_off, T, N, K, g, w_codes, w_scale, rowsum, out, ldo, acc)
    torch.cuda.synchronize()
    assert Q.offq_get_device_status() == Q.OFFQ_OK
    return out[:, :N].float().cpu().numpy().astype(np.float64), acc.cpu().numpy()


def _check_layer(T, K, N, g, out_dt, rotate=True, seed=0, ldo=None, rows=None, n_out=2, mult=50.0,
                 dist="normal"):
    x = W.activations(T, K, seed=seed, dist=dist, n_out=n_out, mult=mult)
    w = W.weights(N, K, seed=seed + 1)
    xh = torch.from_numpy(x).to(torch.bfloat16)
    a_codes, a_scale, a_off = Q.quantize_act(xh.cuda(), g, rotate=rotate, offset=True)
    w_codes, w_scale, rowsum = Q.prepare_weight(torch.from_numpy(w).cuda(), g, rotate=rotate)
    y, acc = _run_gemm(a_codes, a_scale, a_off, w_codes, w_scale, rowsum, g, out_dt, ldo=ldo)
    sel = np.arange(T) if rows is None else rows
    qa = act_q(a_codes, T, K)[sel]
    qw = weight_q(w_codes, N, K)
    sa = a_scale.cpu().numpy().astype(np.float64)[sel]
    oa = a_off.cpu().numpy().astype(np.float64)[sel]
    sw = w_scale.cpu().numpy().astype(np.float64)
    R = rowsum.cpu().numpy().astype(np.float64)
    # The accumulator the tensor cores hold: sum_k (q_a + 8) q_w, exact.
    acc_ref = O.int_gemm(qa + 8, qw)
    np.testing.assert_array_equal(acc[sel], acc_ref)
    dot = O.int_gemm(qa, qw)
    y_ref = O.epilogue(dot, sa, oa, sw, R)
    terms = epilogue_terms(dot, sa, oa, sw, R)
    check_outputs(y[sel], y_ref, terms, K // g, out_dt)
    return y[sel], y_ref, x[sel], w


@pytest.mark.parametrize("out_dt", ["f32", "bf16", "f16"])
def test_toy_layer(out_dt):
    wl = W.WORKLOADS["toy"]
    T, K = wl.T, 512
    x = W.layer_inputs(wl, wl.layers[0])
    w = W.weights(512, K)
    a_codes, a_scale, a_off = Q.quantize_act(torch.from_numpy(x).cuda(), 512)
    w_codes, w_scale, rowsum = Q.prepare_weight(torch.from_numpy(w).cuda(), 512)
    y, acc = _run_gemm(a_codes, a_scale, a_off, w_codes, w_scale, rowsum, 512, out_dt)
    qa = act_q(a_codes, T, K)
    qw = weight_q(w_codes, 512, K)
    np.testing.assert_array_equal(acc, O.int_gemm(qa + 8, qw))
    sa, oa = a_scale.cpu().numpy().astype(np.float64), a_off.cpu().numpy().astype(np.float64)
    sw, R = w_scale.cpu().numpy().astype(np.float64), rowsum.cpu().numpy().astype(np.float64)
    y_ref = O.epilogue(O.int_gemm(qa, qw), sa, oa, sw, R)
    check_outputs(y, y_ref, epilogue_terms(O.int_gemm(qa, qw), sa, oa, sw, R), 1, out_dt)
    if out_dt == "f16":
        assert max_rel_err_floored(y, y_ref) <= 2e-3
    # Quality sanity against the unquantized layer (not parity).
    ref = O.linear_reference(x, w)
    assert np.linalg.norm(y - ref) < 0.25 * np.linalg.norm(ref)


def test_oracle_codes_through_gemm():
    """Codes, scales and offsets made by the oracle go through the GPU GEMM."""
    T, K, N, g = 45, 1024, 320, 256
    x = W.activations(T, K, seed=31, n_out=2, mult=60.0)
    w = W.weights(N, K, seed=32)
    xa = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    a = O.quantize_act(xa, g)
    wp = O.prepare_weight(w.astype(np.float64), g)
    dev = lambda arr, dt: torch.from_numpy(np.ascontiguousarray(arr)).to(dt).cuda()
    y, acc = _run_gemm(dev(O.tile_codes(a["codes"]).reshape(-1, K // 2), torch.uint8), dev(a["scale"], torch.float32),
                       dev(a["offset"], torch.float32), dev(O.tile_codes(wp["codes"]).reshape(-1, K // 2), torch.uint8),
                       dev(wp["scale"], torch.float32), dev(wp["offsum"], torch.float32), g, "f32")
    np.testing.assert_array_equal(acc, O.int_gemm(a["q"] + 8, wp["q"]))
    sa = a["scale"].astype(np.float32).astype(np.float64)
    oa = a["offset"].astype(np.float32).astype(np.float64)
    sw = wp["scale"].astype(np.float32).astype(np.float64)
    y_ref = O.epilogue(O.int_gemm(a["q"], wp["q"]), sa, oa, sw, wp["offsum"])
    check_outputs(y, y_ref, epilogue_terms(O.int_gemm(a["q"], wp["q"]), sa, oa, sw, wp["offsum"]), K // g, "f32")


@pytest.mark.parametrize("T,K,N,g,out_dt,ldo", [
    (33, 1024, 300, 256, "bf16", 304),     # ragged T and N, padded output rows
    (130, 11008, 264, 256, "bf16", None),  # 43 offset blocks
    (64, 14336, 512, 1024, "f16", None),   # 14 offset blocks
    (3, 4096, 1000, 4096, "f32", 1000),
    (1, 4096, 11008, 4096, "bf16", None),  # one decode token
    (200, 4096, 4096, 4096, "bf16", None),
    (129, 2048, 257, 2048, "f32", 260),
    (40, 4096, 512, 32, "f32", None),      # 128 offset blocks of 32 channels
    (300, 1024, 800, 128, "bf16", None),   # the paper's group size, 8 blocks; several tiles per CTA
    (50, 1024, 258, 256, "bf16", 264),     # N % 4 != 0 with 4 offset blocks (scalar epilogue loads)
    (5, 96, 200, 32, "f32", None),         # K = 96: a k-tile of three 32-channel chunks
    # 2 x 40 pair tiles: on 76 clusters the 4 tiles past the first wave are cut
    # along N into 64-column pieces (ragged N at the end), with 4 and 1 offset blocks.
    (512, 1024, 10200, 256, "bf16", None),
    (512, 1024, 10200, 1024, "f32", 10208),
    # Decode form (T <= 64): more weight blocks than 4 per SM, so each CTA makes two passes of its
    # accumulator; and a K that is not a multiple of the 4-k-tile bulk copies.
    (9, 1024, 28672, 1024, "bf16", None),
    (17, 1920, 640, 128, "f16", None),
    # Few-token form (T <= 4, dp4a on the CUDA cores): every token count class (1, 2, 4 with
    # 3 padded), K = 1056 (33 chunks: the eighths of K are uneven and the last warp has none),
    # K = 11008 at 4 tokens (43 KB of unpacked activations, 43 offset blocks), and a K whose
    # unpacked activations exceed its budget (4 x 32768 bytes: the tensor-core form). Then the
    # decode kernel at its smallest token counts (5 to 8: 11 to 14 padded MMA columns).
    (1, 1024, 300, 256, "f32", None),
    (2, 4096, 1000, 4096, "f16", 1000),
    (3, 1056, 520, 32, "bf16", None),
    (4, 11008, 264, 256, "bf16", 272),
    (4, 32768, 512, 1024, "bf16", None),
    (5, 11008, 4096, 256, "f32", None),
    (6, 1056, 700, 32, "f16", 704),
    (7, 4096, 1000, 1024, "bf16", 1008),
    (8, 11008, 520, 256, "f32", None),
])
def test_layers(T, K, N, g, out_dt, ldo):
    _check_layer(T, K, N, g, out_dt, ldo=ldo, seed=T + K)


def test_no_rotation_site():
    """q/k/v/gate/up sites: codes made without the online rotation."""
    _check_layer(64, 4096, 768, 4096, "bf16", rotate=False, seed=5)


def test_null_offset_means_zero():
    T, K, N, g = 16, 512, 256, 512
    x = W.activations(T, K, seed=41)
    a_codes, a_scale, _ = Q.quantize_act(torch.from_numpy(x).cuda(), g, rotate=True, offset=False)
    w_codes, w_scale, rowsum = Q.prepare_weight(torch.from_numpy(W.weights(N, K, seed=42)).cuda(), g)
    y, acc = _run_gemm(a_codes, a_scale, None, w_codes, w_scale, rowsum, g, "f32")
    qa = act_q(a_codes, T, K)
    qw = weight_q(w_codes, N, K)
    sa, sw = a_scale.cpu().numpy().astype(np.float64), w_scale.cpu().numpy().astype(np.float64)
    R = rowsum.cpu().numpy().astype(np.float64)
    zero = np.zeros((T, 1))
    y_ref = O.epilogue(O.int_gemm(qa, qw), sa, zero, sw, R)
    check_outputs(y, y_ref, epilogue_terms(O.int_gemm(qa, qw), sa, zero, sw, R), 1, "f32")


def test_accumulator_exact_at_largest_k():
    """K = 28672 with every code at +-7: the extreme integer sums stay exact."""
    T, N, K, g = 8, 256, 28672, 1024
    qa = np.full((T, K), 7, dtype=np.int64)
    qa[1::2] = -7
    qw = np.full((N, K), 7, dtype=np.int64)
    qw[::3] = -7
    dev = lambda arr, dt: torch.from_numpy(np.ascontiguousarray(arr)).to(dt).cuda()
    sa = np.ones(T, dtype=np.float32)
    sw = np.ones(N, dtype=np.float32)
    R = qw.reshape(N, K // g, g).sum(axis=2).T.astype(np.float32)
    y, acc = _run_gemm(dev(O.tile_codes(O.pack_act_codes(qa)).reshape(-1, K // 2), torch.uint8),
                       dev(sa, torch.float32), None,
                       dev(O.tile_codes(O.pack_weight_codes(qw)).reshape(-1, K // 2), torch.uint8), dev(sw, torch.float32),
                       dev(R, torch.float32),
                       g, "f32")
    np.testing.assert_array_equal(acc, O.int_gemm(qa + 8, qw))
    np.testing.assert_array_equal(y, O.int_gemm(qa, qw).astype(np.float64))


@pytest.mark.parametrize("T", [1, 8, 96])
def test_accumulator_exact_at_maximum_k(T):
    """K = 65536, the largest the ABI takes, with every code at +-7, through each form of the
    linear (CUDA-core at 1 token, the decode kernel at 8, the pair kernel at 96): the largest
    sum, 15 * 7 * 65536 < 2^24, stays exact."""
    N, K, g = 256, 65536, 8192
    qa = np.full((T, K), 7, dtype=np.int64)
    qa[1::2] = -7
    qa[:, ::5] = 3
    qw = np.full((N, K), 7, dtype=np.int64)
    qw[::3] = -7
    qw[:, ::7] = 0
    dev = lambda arr, dt: torch.from_numpy(np.ascontiguousarray(arr)).to(dt).cuda()
    sa = np.full(T, 0.5, dtype=np.float32)
    sw = np.full(N, 0.25, dtype=np.float32)
    R = qw.reshape(N, K // g, g).sum(axis=2).T.astype(np.float32)
    y, acc = _run_gemm(dev(O.tile_codes(O.pack_act_codes(qa)).reshape(-1, K // 2), torch.uint8),
                       dev(sa, torch.float32), None,
                       dev(O.tile_codes(O.pack_weight_codes(qw)).reshape(-1, K // 2), torch.uint8), dev(sw, torch.float32),
                       dev(R, torch.float32),
                       g, "f32")
    np.testing.assert_array_equal(acc, O.int_gemm(qa + 8, qw))
    np.testing.assert_array_equal(y, 0.125 * O.int_gemm(qa, qw).astype(np.float64))


def test_full_llama2_7b_gate_sampled():
    """Full 2048 x 4096 -> 11008 launch, checked on 128 sampled token rows."""
    rows = W.unit_index_sample(2048, 128, seed=4)
    _check_layer(2048, 4096, 11008, 4096, "bf16", rows=rows, n_out=4, mult=100.0)


def test_full_llama2_7b_down_sampled():
    rows = W.unit_index_sample(2048, 64, seed=5)
    _check_layer(2048, 11008, 4096, 256, "bf16", rows=rows, n_out=4, mult=100.0)


@pytest.mark.parametrize("T", [8, 32, 64])
def test_decode_sweep(T):
    """Decode batches of the Llama-2-7B up-projection shape (4096 -> 11008)."""
    _check_layer(T, 4096, 11008, 4096, "bf16", seed=60 + T, n_out=4, mult=100.0)


def test_llama3_8b_mlp_down_sampled():
    """4096 tokens x 14336 -> 4096 with 14 offset blocks of 1024, Student-t(3) inputs, 3 outliers."""
    rows = W.unit_index_sample(4096, 48, seed=6)
    _check_layer(4096, 14336, 4096, 1024, "bf16", rows=rows, n_out=3, mult=100.0, dist="student_t3")


def test_llama2_70b_down_shape_sampled():
    """K = 28672 in 28 offset blocks of 1024, 6 outliers at 200x (1024 tokens, 1024 outputs)."""
    rows = W.unit_index_sample(1024, 64, seed=7)
    _check_layer(1024, 28672, 1024, 1024, "bf16", rows=rows, n_out=6, mult=200.0)


def _check_config_layer(T, K, N, g, rows, dist, n_out, mult, seed):
    """A launch at a configuration's own shape (the bench's q/k/v/o/gate/up sites:
    codes made without the online rotation), checked on sampled token rows
    against all N outputs; only the sampled rows leave the device."""
    x = W.activations(T, K, seed=seed, dist=dist, n_out=n_out, mult=mult)
    gen = torch.Generator(device="cuda").manual_seed(seed + 1)
    w = torch.randn((N, K), generator=gen, device="cuda") * 0.02
    a_codes, a_scale, a_off = Q.quantize_act(torch.from_numpy(x).to(torch.bfloat16).cuda(), g, rotate=False,
                                             offset=True)
    w_codes, w_scale, rowsum = Q.prepare_weight(w, g, rotate=False)
    del w
    out = torch.full((T, N), float("nan"), dtype=torch.bfloat16, device="cuda")
    acc = torch.zeros((T, N), dtype=torch.int32, device="cuda")
    Q.offq_w4a4_linear(a_codes, a_scale, a_off, T, N, K, g, w_codes, w_scale, rowsum, out, N, acc)
    torch.cuda.synchronize()
    assert Q.offq_get_device_status() == Q.OFFQ_OK
    sel = torch.from_numpy(rows).cuda()
    y = out.index_select(0, sel).float().cpu().numpy().astype(np.float64)
    acc_s = acc.index_select(0, sel).cpu().numpy()
    del out, acc
    qa = act_q(a_codes, T, K)[rows]
    qw = weight_q(w_codes, N, K)
    sa = a_scale.cpu().numpy().astype(np.float64)[rows]
    oa = a_off.cpu().numpy().astype(np.float64)[rows]
    sw = w_scale.cpu().numpy().astype(np.float64)
    R = rowsum.cpu().numpy().astype(np.float64)
    acc_ref = O.int_gemm(qa + 8, qw)
    np.testing.assert_array_equal(acc_s, acc_ref)
    dot = O.int_gemm(qa, qw)
    y_ref = O.epilogue(dot, sa, oa, sw, R)
    check_outputs(y, y_ref, epilogue_terms(dot, sa, oa, sw, R), K // g, "bf16")


@pytest.mark.parametrize("T,K,N,g,nrows,dist,n_out,mult", [
    (2048, 8192, 8192, 8192, 48, "normal", 6, 200.0),       # Llama-2-70B q / o: one offset block of 8192
    (8192, 8192, 1024, 8192, 96, "normal", 6, 200.0),       # Llama-2-70B k / v (8 KV heads x 128), full prefill
    (2048, 8192, 28672, 8192, 32, "normal", 6, 200.0),      # Llama-2-70B gate / up: 112 output tiles
    (4096, 4096, 14336, 4096, 48, "student_t3", 3, 100.0),  # Llama-3-8B gate / up
])
def test_config_gemm_shapes_sampled(T, K, N, g, nrows, dist, n_out, mult):
    rows = np.unique(np.concatenate([W.unit_index_sample(T, nrows, seed=N % 97), [0, T - 1]]))
    _check_config_layer(T, K, N, g, rows, dist, n_out, mult, seed=K + N)


@pytest.mark.parametrize("K,g", [(4096, 4096), (11008, 256), (4096, 32)])
def test_outputs_near_zero_against_large_row_sums(K, g):
    """Weight rows of all +7 (row sums 7K) against activation rows whose codes add up to
    0, +-1, +-2, ...: every output is a small multiple of s_a s_w next to the 8 s_a R that the
    tensor cores carry in acc'. Removing that term in the integer domain leaves each fp32 output
    within a few rounding errors of the float64 result (max relative error 2e-3 with no floor,
    f32 out), for one block, 43 blocks, and the unstaged 128-block epilogue."""
    T, N = 64, 512
    rng = np.random.default_rng(K + g)
    qa = rng.integers(-7, 8, size=(T, K))
    # Make each row's code sum a small integer: move the excess onto channels with room.
    for t in range(T):
        target = t % 9 - 4
        excess = int(qa[t].sum()) - target
        while excess != 0:
            k = int(rng.integers(0, K))
            step = max(-7 - qa[t, k], min(7 - qa[t, k], -excess))
            qa[t, k] += step
            excess += step
    qw = rng.integers(-7, 8, size=(N, K))
    qw[::2] = 7                                            # every other weight row all +7
    sa = rng.uniform(0.5, 2.0, size=T).astype(np.float32)
    sw = rng.uniform(0.5, 2.0, size=N).astype(np.float32)
    R = qw.reshape(N, K // g, g).sum(axis=2).T.astype(np.float32)
    dev = lambda arr, dt: torch.from_numpy(np.ascontiguousarray(arr)).to(dt).cuda()
    y, acc = _run_gemm(dev(O.tile_codes(O.pack_act_codes(qa)).reshape(-1, K // 2), torch.uint8),
                       dev(sa, torch.float32), None,
                       dev(O.tile_codes(O.pack_weight_codes(qw)).reshape(-1, K // 2), torch.uint8),
                       dev(sw, torch.float32), dev(R, torch.float32), g, "f32")
    np.testing.assert_array_equal(acc, O.int_gemm(qa + 8, qw))
    dot = O.int_gemm(qa, qw)
    zero = np.zeros((T, K // g))
    y_ref = O.epilogue(dot, sa.astype(np.float64), zero, sw.astype(np.float64), R.astype(np.float64))
    np.testing.assert_array_equal(dot[:, ::2], np.repeat(7 * (np.arange(T) % 9 - 4)[:, None], N // 2, axis=1))
    check_outputs(y, y_ref, epilogue_terms(dot, sa, zero, sw, R), K // g, "f32")
    nz = y_ref != 0
    assert np.all(y[~nz] == 0)
    assert np.max(np.abs(y[nz] - y_ref[nz]) / np.abs(y_ref[nz])) <= 2e-3


def test_few_token_forms_agree():
    """4 tokens take the CUDA-core form, 5 to 9 the tensor-core decode kernel: on the same rows
    both give the same integer accumulators and, with the same epilogue chain, the same
    output bits."""
    T, K, N, g = 9, 4096, 11008, 4096
    x = W.activations(T, K, seed=71, n_out=4, mult=100.0)
    w = W.weights(N, K, seed=72)
    a_codes, a_scale, a_off = Q.quantize_act(torch.from_numpy(x).to(torch.bfloat16).cuda(), g, rotate=False)
    w_codes, w_scale, rowsum = Q.prepare_weight(torch.from_numpy(w).cuda(), g, rotate=False)
    for dt in ("bf16", "f32"):
        y9, acc9 = _run_gemm(a_codes, a_scale, a_off, w_codes, w_scale, rowsum, g, dt, T=9)
        for t in (8, 5, 4):
            yt, acct = _run_gemm(a_codes, a_scale[:t], a_off[:t], w_codes, w_scale, rowsum, g, dt, T=t)
            np.testing.assert_array_equal(acct, acc9[:t])
            np.testing.assert_array_equal(yt, y9[:t])

