"""The fp32 facts the kernels rely on, checked on the CPU with IEEE float32
arithmetic (numpy rounds each float32 operation to nearest even, as the
kernels' .rn instructions do). None of this is the oracle: these are the
arithmetic shortcuts the CUDA code takes, stated where a reader can check
them.

* The absmax of an H_2 stage (tensor-core quantizer): for outputs
  fl(u + t) and fl(u - t), the larger magnitude is exactly fl(|u| + |t|).
* Magic-number rounding (every quantizer): for |v| < 7.5 (the kernels' values
  are at most 7 (1 + 2^-24) in magnitude) the float32 sum
  fl(v + 1.5 * 2^23 + 8) holds round_half_even(v) + 8 in its low four bits,
  and bits 4-21 of its pattern are zero.
* The 4-bit integer operands of the GEMM: the bytes 0x00..0x0F read as E4M3
  are exactly 0, 1, ..., 15 times 2^-9 (subnormals up to 7, then exponent 1).
* The tensor-core quantizer's derived error bound stays a tight tie window on
  the inputs it serves.
"""

import numpy as np

F = np.float32


def _rand_f32(rng, n, lo_exp=-30, hi_exp=30):
    m = rng.uniform(1.0, 2.0, n).astype(np.float32)
    e = rng.integers(lo_exp, hi_exp, n)
    s = rng.choice(np.array([-1.0, 1.0], np.float32), n)
    return (s * np.ldexp(m, e)).astype(np.float32)


def test_h2_pair_absmax_is_abs_sum():
    rng = np.random.default_rng(0)
    n = 200_000
    u = _rand_f32(rng, n)
    t = _rand_f32(rng, n)
    # Near-equal magnitudes (heavy cancellation in one of the two outputs).
    t[: n // 4] = (u[: n // 4] * F(1.0 + 2.0 ** -20)).astype(np.float32)
    t[n // 4 : n // 2] = -u[n // 4 : n // 2]
    t[n // 2 : n // 2 + 1000] = 0.0
    with np.errstate(over="ignore"):
        s = (u + t).astype(np.float32)
        d = (u - t).astype(np.float32)
        a = (np.abs(u) + np.abs(t)).astype(np.float32)
    big = np.maximum(np.abs(s), np.abs(d))
    np.testing.assert_array_equal(big, a)


def test_magic_number_rounding_gives_the_code():
    magic = F(12582920.0)  # 1.5 * 2^23 + 8
    assert float(magic) == 1.5 * 2 ** 23 + 8
    # float32 values in (-7.5, 7.5) on a fine grid, the exact ties included.
    v = np.concatenate([
        np.linspace(-7.5, 7.5, 600_001).astype(np.float32),
        np.arange(-15, 16, dtype=np.float32) / F(2.0),            # the half-integers
        np.nextafter(np.arange(-15, 16, dtype=np.float32) / F(2.0), F(np.inf)),
        np.nextafter(np.arange(-15, 16, dtype=np.float32) / F(2.0), F(-np.inf)),
    ]).astype(np.float32)
    v = v[np.abs(v) < 7.5]
    r = (v + magic).astype(np.float32)
    bits = r.view(np.uint32)
    code = (bits & 0xF).astype(np.int64)
    np.testing.assert_array_equal(code, np.rint(v.astype(np.float64)).astype(np.int64) + 8)
    assert np.all((bits >> 4) & ((1 << 18) - 1) == 0)
    assert np.all(bits & ~np.uint32(0x3FFFFF) == 0x4B400000)


def test_small_integers_are_exact_e4m3_subnormals():
    def e4m3(byte):
        s = -1.0 if byte & 0x80 else 1.0
        e = (byte >> 3) & 0xF
        m = byte & 0x7
        return s * (m / 8.0) * 2.0 ** -6 if e == 0 else s * (1 + m / 8.0) * 2.0 ** (e - 7)

    for k in range(16):
        assert e4m3(k) == k * 2.0 ** -9
        # The weights' sign-magnitude bytes: bit 7 is the sign of the same value.
        if k < 8:
            assert e4m3(0x80 | k) == -k * 2.0 ** -9


def test_tensor_core_bound_keeps_the_tie_window_tight():
    """The tensor-core quantizer's error bound (TC_FACTOR u sum|x| per block) in code
    units, on the prefill recipes it serves (Llama-2-70B and Llama-3-8B down-proj
    inputs): a code may differ from the oracle's only within that window of a
    rounding tie, so the bound must stay far below half a code step."""
    import oracle as O
    import workloads as W
    from parity import code_window

    for K, dist, n_out, mult in [(28672, "normal", 6, 200.0), (14336, "student_t3", 3, 100.0)]:
        x = W.activations(16, K, seed=5, dist=dist, n_out=n_out, mult=mult).astype(np.float64)
        ref = O.quantize_act(x, 1024, rotate=True, offset=True)
        w = code_window(ref["scale"], x, 1024, tc=True)
        assert np.all(w < 2e-3), (K, float(w.max()))
