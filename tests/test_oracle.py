"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each test would fail under a plausible slip in the oracle: a wrong Hadamard
ordering or normalisation, a dropped or mis-indexed offset term, a wrong
rounding mode or scale, a transposed GEMM operand, or a wrong nibble layout.
"""

import json
import math
import os

import numpy as np
import pytest
import scipy.linalg

import oracle as O
import workloads as W


def _load(golden_dir, name):
    with open(os.path.join(golden_dir, name)) as f:
        return json.load(f)


# --------------------------------------------------------------------------
# Hadamard (Sec. 3.2): +-1 entries, orthogonal, first row all ones.
# --------------------------------------------------------------------------

@pytest.mark.parametrize("g", [1, 2, 4, 8, 32, 128, 512, 2048])
def test_hadamard_structure(g):
    H = O.sylvester_hadamard(g)
    assert H.shape == (g, g)
    assert set(np.unique(H)) <= {-1, 1}
    assert np.all(H[0] == 1)
    np.testing.assert_array_equal(H @ H.T, g * np.eye(g, dtype=np.int64))
    # Every row but the first sums to zero: the reason the offset is x_1 / sqrt(g).
    np.testing.assert_array_equal(H[1:].sum(axis=1), 0)


@pytest.mark.parametrize("g", [2, 16, 256, 1024])
def test_hadamard_matches_library(g):
    # scipy builds the Sylvester matrix independently.
    np.testing.assert_array_equal(O.sylvester_hadamard(g), scipy.linalg.hadamard(g))


def test_hadamard_h4_golden(golden_dir):
    d = _load(golden_dir, "hadamard_h4.json")
    np.testing.assert_array_equal(O.sylvester_hadamard(4), np.array(d["H4"]))


def test_rotation_against_butterfly():
    """The dense-matmul rotation equals an independent fast butterfly transform."""
    rng = np.random.default_rng(3)
    g, T = 64, 5
    x = rng.standard_normal((T, 3 * g))

    def fwht(v):
        v = v.copy()
        h = 1
        while h < len(v):
            for i in range(0, len(v), 2 * h):
                a = v[i:i + h].copy()
                b = v[i + h:i + 2 * h].copy()
                v[i:i + h] = a + b
                v[i + h:i + 2 * h] = a - b
            h *= 2
        return v

    y = O.rotate_blocks(x, g)
    for t in range(T):
        for b in range(3):
            blk = x[t, b * g:(b + 1) * g]
            np.testing.assert_allclose(y[t, b * g:(b + 1) * g], fwht(blk) / math.sqrt(g),
                                       rtol=0, atol=1e-12)


@pytest.mark.parametrize("g", [2, 8, 128, 1024])
def test_rotation_is_orthonormal(g):
    rng = np.random.default_rng(g)
    x = rng.standard_normal((4, 2 * g))
    y = O.rotate_blocks(x, g)
    # Parseval per block: a wrong normalisation (1/g, none) changes the norm.
    for b in range(2):
        sl = slice(b * g, (b + 1) * g)
        np.testing.assert_allclose(np.linalg.norm(y[:, sl], axis=1),
                                   np.linalg.norm(x[:, sl], axis=1), rtol=1e-12)
    # Applying it twice is the identity (H/sqrt(g) is symmetric and orthogonal).
    np.testing.assert_allclose(O.rotate_blocks(y, g), x, rtol=0, atol=1e-11)


# --------------------------------------------------------------------------
# Offsetting (Sec. 3.2, Eq. 4-5).
# --------------------------------------------------------------------------

def test_eq5_worked_example(golden_dir):
    d = _load(golden_dir, "eq5_two_channel.json")
    for c in d["cases"]:
        x = np.array([c["x"]])
        y = O.rotate_blocks(x, 2)
        np.testing.assert_allclose(y[0], c["y"], rtol=1e-15, atol=1e-15)
        res = O.quantize_act(x, 2, rotate=True, offset=True)
        np.testing.assert_allclose(res["offset"][0, 0], c["offset"], rtol=1e-15, atol=1e-15)
        np.testing.assert_allclose(res["residual"][0], c["residual"], rtol=1e-15, atol=1e-15)


@pytest.mark.parametrize("g", [2, 4, 32, 256, 1024])
def test_offset_is_first_channel_over_sqrt_g(g):
    """The block mean of X H / sqrt(g) is x_1 / sqrt(g) (Sec. 3.2)."""
    rng = np.random.default_rng(11 + g)
    G = 3
    x = rng.standard_normal((6, G * g)) * 3.0
    res = O.quantize_act(x, g, rotate=True, offset=True)
    expect = x[:, ::g] / math.sqrt(g)
    np.testing.assert_allclose(res["offset"], expect, rtol=1e-12, atol=1e-12)
    # The residual of every block sums to zero.
    np.testing.assert_allclose(res["residual"].reshape(6, G, g).sum(axis=2), 0.0, atol=1e-10)


def test_outlier_only_row_leaves_zero_residual():
    g = 128
    x = np.zeros((2, 2 * g))
    x[0, 0] = 300.0
    x[0, g] = -20.5
    x[1, 0] = 1e-3
    res = O.quantize_act(x, g, rotate=True, offset=True)
    assert np.all(res["residual"] == 0.0)
    assert np.all(res["q"] == 0) and np.all(res["scale"] == 0.0)
    np.testing.assert_allclose(res["offset"][0], [300.0 / math.sqrt(g), -20.5 / math.sqrt(g)], rtol=1e-15)


def test_unit_channel_gives_hadamard_row_codes():
    """x = e_j (j >= 1) rotates to H[j]/sqrt(g): offset 0, all codes +-7 in H's sign pattern."""
    g = 64
    H = O.sylvester_hadamard(g)
    for j in (1, 5, 63):
        x = np.zeros((1, g))
        x[0, j] = 1.0
        res = O.quantize_act(x, g, rotate=True, offset=True)
        assert res["offset"][0, 0] == 0.0
        np.testing.assert_array_equal(res["q"][0], 7 * H[j])
        np.testing.assert_allclose(res["scale"][0], 1.0 / (7.0 * math.sqrt(g)), rtol=1e-15)


def test_offset_without_rotation_is_block_mean():
    x = np.array([[1.0, 2.0, 3.0, 6.0, -1.0, -1.0, -1.0, -1.0]])
    res = O.quantize_act(x, 4, rotate=False, offset=True)
    np.testing.assert_array_equal(res["offset"], [[3.0, -1.0]])
    np.testing.assert_array_equal(res["residual"], [[-2.0, -1.0, 0.0, 3.0, 0.0, 0.0, 0.0, 0.0]])
    # Residual max is 3 -> scale 3/7; codes rne(r * 7/3).
    np.testing.assert_array_equal(res["q"], [[-5, -2, 0, 7, 0, 0, 0, 0]])


def test_offsetting_reduces_quantization_error():
    """Statistical property the method rests on (Sec. 3.2): with a concentrated
    outlier channel, offsetting lowers the 4-bit reconstruction error."""
    g = 512
    x = W.activations(64, g, seed=5, n_out=1, mult=100.0)
    with_off = O.quantize_act(x, g, rotate=True, offset=True)
    no_off = O.quantize_act(x, g, rotate=True, offset=False)
    y = with_off["y"]

    def mse(res):
        xh = O.dequantize_act(res["q"], res["scale"], res["offset"], g)
        return np.mean((xh - y) ** 2)

    assert mse(with_off) < 0.5 * mse(no_off)


# --------------------------------------------------------------------------
# Quantizer (Eq. 1, symmetric; readings: rne, s = max/7, [-7, 7]).
# --------------------------------------------------------------------------

def test_rtn_textbook_rows(golden_dir):
    d = _load(golden_dir, "rtn_textbook.json")
    for row in d["rows"]:
        x = np.array([row["x"]])
        res = O.quantize_act(x, 8, rotate=False, offset=False)
        np.testing.assert_array_equal(res["q"][0], row["q"])
        np.testing.assert_allclose(res["scale"][0], row["scale"], rtol=1e-15)
        assert np.all(res["offset"] == 0.0)


def test_quantization_error_bound():
    rng = np.random.default_rng(21)
    x = rng.standard_normal((32, 256)) * rng.uniform(0.1, 10, size=(32, 1))
    for rotate in (False, True):
        for offset in (False, True):
            res = O.quantize_act(x, 64, rotate=rotate, offset=offset)
            err = np.abs(res["residual"] - res["scale"][:, None] * res["q"])
            assert np.all(err <= res["scale"][:, None] / 2 * (1 + 1e-12))
            # The largest residual of each row lands on the grid's end.
            assert np.all(np.max(np.abs(res["q"]), axis=1) == 7)


def test_brute_force_eight_channels():
    """At D = 8, each code is the grid point nearest to R/s, ties to the even code."""
    rng = np.random.default_rng(8)
    grid = np.arange(-7, 8)
    for trial in range(200):
        x = rng.standard_normal((1, 8)) * rng.uniform(0.01, 100)
        if trial % 4 == 0:
            x[0, 0] += 50.0
        rotate = trial % 2 == 0
        res = O.quantize_act(x, 8, rotate=rotate, offset=True)
        r, s = res["residual"][0], res["scale"][0]
        for k in range(8):
            d = np.abs(r[k] / s - grid)
            best = grid[d <= d.min() + 1e-12]
            expect = best[0] if len(best) == 1 else best[best % 2 == 0][0]
            assert res["q"][0, k] == expect


def test_pack_layout_golden(golden_dir):
    d = _load(golden_dir, "pack_layout.json")
    codes = np.array([d["codes"]])
    np.testing.assert_array_equal(O.pack_act_codes(codes)[0], d["act_bytes"])
    np.testing.assert_array_equal(O.unpack_act_codes(np.array([d["act_bytes"]]))[0], d["codes"])
    np.testing.assert_array_equal(O.pack_weight_codes(codes)[0], d["weight_bytes"])
    np.testing.assert_array_equal(O.unpack_weight_codes(np.array([d["weight_bytes"]]))[0], d["codes"])


def test_pack_roundtrip_all_codes():
    rng = np.random.default_rng(1)
    q = rng.integers(-7, 8, size=(3, 256))
    np.testing.assert_array_equal(O.unpack_act_codes(O.pack_act_codes(q)), q)
    np.testing.assert_array_equal(O.unpack_weight_codes(O.pack_weight_codes(q)), q)
    with pytest.raises(ValueError):
        O.pack_act_codes(np.array([[8, 0]]))
    with pytest.raises(ValueError):
        O.pack_weight_codes(np.array([[-8, 0, 0, 0, 0, 0, 0, 0]]))


def test_tiled_layout_positions():
    """Hand-worked positions of the tiled operand layout (R = 33 rows, K = 64 codes)."""
    R, K = 33, 64
    p = np.zeros((R, K // 2), dtype=np.uint8)
    p[0, 0] = 1      # row 0, byte 0   -> tile (0, 0), row 0      -> 0
    p[1, 3] = 2      # row 1, byte 3   -> tile (0, 0), row 1      -> 16 + 3 = 19
    p[2, 17] = 3     # row 2, byte 17  -> tile (0, 1), row 2      -> 512 + 32 + 1 = 545
    p[31, 31] = 4    # row 31, byte 31 -> tile (0, 1), row 31     -> 512 + 496 + 15 = 1023
    p[32, 16] = 5    # row 32, byte 16 -> tile (1, 1), row 0      -> 3 * 512 = 1536
    t = O.tile_codes(p)
    assert t.size == 64 * 32                      # rows padded to 64
    expect = {0: 1, 19: 2, 545: 3, 1023: 4, 1536: 5}
    for pos, val in expect.items():
        assert t[pos] == val
    assert np.count_nonzero(t) == len(expect)
    np.testing.assert_array_equal(O.untile_codes(t, R, K), p)


# --------------------------------------------------------------------------
# Weights, GEMM and epilogue.
# --------------------------------------------------------------------------

def test_weight_rotation_cancels():
    """(X H)(W H)^T = X W^T for the symmetric orthonormal block Hadamard."""
    rng = np.random.default_rng(4)
    g, K, N = 32, 96, 7
    x = rng.standard_normal((5, K))
    w = rng.standard_normal((N, K))
    y = O.rotate_blocks(x, g)
    wp = O.prepare_weight(w, g, rotate=True)
    np.testing.assert_allclose(y @ wp["w_eff"].T, x @ w.T, rtol=1e-11, atol=1e-11)


def test_weight_table_is_block_rowsum():
    rng = np.random.default_rng(6)
    g, K, N = 16, 64, 9
    w = rng.standard_normal((N, K))
    wp = O.prepare_weight(w, g, rotate=True)
    q = O.unpack_weight_codes(wp["codes"])
    np.testing.assert_array_equal(q, wp["q"])
    for b in range(K // g):
        for n in range(N):
            assert wp["offsum"][b, n] == q[n, b * g:(b + 1) * g].sum()


def test_int_gemm_loops_match_blas():
    rng = np.random.default_rng(9)
    qa = rng.integers(-7, 8, size=(5, 40))
    qw = rng.integers(-7, 8, size=(6, 40))
    np.testing.assert_array_equal(O.int_gemm(qa, qw), O.int_gemm_loops(qa, qw))
    # Not transposed: a row of ones against a one-hot weight picks one column sum.
    e = np.zeros((1, 40), dtype=np.int64)
    e[0, 3] = 1
    np.testing.assert_array_equal(O.int_gemm(qa, e)[:, 0], qa[:, 3])


def test_int_gemm_exact_at_largest_k():
    K = 28672
    qa = np.full((2, K), 7)
    qw = np.full((3, K), -7)
    qw[1] = 7
    acc = O.int_gemm(qa, qw)
    assert acc[0, 0] == -49 * K and acc[0, 1] == 49 * K


def test_offset_identity_unquantized():
    """W x = W (x - o 1) + o W 1 per block, in float64 before any rounding."""
    rng = np.random.default_rng(10)
    g, G, N = 32, 3, 11
    x = rng.standard_normal((4, g * G)) * 5
    w = rng.standard_normal((N, g * G))
    o = rng.standard_normal((4, G)) * 20
    ob = np.repeat(o, g, axis=1)
    lhs = x @ w.T
    rhs = (x - ob) @ w.T + o @ w.reshape(N, G, g).sum(axis=2).T
    np.testing.assert_allclose(lhs, rhs, rtol=1e-12, atol=1e-10)


@pytest.mark.parametrize("rotate", [False, True])
def test_epilogue_equals_dequantized_product(rotate):
    """s_a s_w acc + o S equals X_hat W_hat^T computed from the dequantized matrices."""
    g, G, N, T = 64, 3, 13, 7
    x = W.activations(T, g * G, seed=12, n_out=2, mult=40.0)
    w = W.weights(N, g * G, seed=13)
    a = O.quantize_act(x, g, rotate=rotate, offset=True)
    wp = O.prepare_weight(w, g, rotate=rotate)
    out = O.w4a4_linear(a["q"], a["scale"], a["offset"], wp["q"], wp["scale"], wp["offsum"])
    xh = O.dequantize_act(a["q"], a["scale"], a["offset"], g)
    wh = wp["q"] * wp["scale"][:, None]
    np.testing.assert_allclose(out["y"], xh @ wh.T, rtol=1e-12, atol=1e-12 * np.abs(out["y"]).max())
    # And it approximates the unquantized layer.
    ref = O.linear_reference(x, w)
    assert np.linalg.norm(out["y"] - ref) < 0.3 * np.linalg.norm(ref)


def test_kv4_is_per_head_block():
    kv = W.kv_heads(3, 4, 128, seed=2)
    res = O.kv4_quantize(kv)
    for t in range(3):
        for h in range(4):
            one = O.quantize_act(kv[t, h][None, :], 128)
            np.testing.assert_array_equal(res["q"][t, h], one["q"][0])
            assert res["scale"][t, h] == one["scale"][0]
            assert res["offset"][t, h] == one["offset"][0, 0]


def test_storage_bits_golden(golden_dir):
    d = _load(golden_dir, "storage_bits.json")
    assert O.effective_bits(d["group"], d["code_bits"], d["param_bits"], d["n_params"]) == d["bits"]
    # This path: one fp32 scale per token + one fp32 offset per block.
    assert O.effective_bits_per_token_offset(4096, 4096) == pytest.approx(4 + 64 / 4096)


# --------------------------------------------------------------------------
# Per-group asymmetric activations (Eq. 1 with z; Sec. 3.2 footnote; Sec. 4:
# groups of 128). Readings: s = (max - min) / 15, z = -rne(min / s),
# q = clamp(rne(y / s) + z, 0, 15); a constant group has s = z = q = 0.
# --------------------------------------------------------------------------

def test_group_affine_grid_is_exact():
    """A group whose values sit on s0 * (j - z0), j covering 0..15, comes back
    exactly: s = s0, z = z0, q = j (powers of two keep every division exact)."""
    rng = np.random.default_rng(40)
    for trial in range(50):
        group = 16 * int(rng.integers(1, 5))
        s0 = 2.0 ** int(rng.integers(-6, 4))
        z0 = int(rng.integers(-40, 40))
        j = rng.integers(0, 16, size=group)
        j[rng.integers(0, group)] = 0
        j[(rng.integers(1, group) + 3) % group] = 15
        if j.min() != 0 or j.max() != 15:
            j[0], j[1] = 0, 15
        y = s0 * (j - z0).astype(np.float64)
        q, s, z = O.quantize_groups_asym(y[None, :], group)
        assert s[0, 0] == s0 and z[0, 0] == z0
        np.testing.assert_array_equal(q[0], j)
        np.testing.assert_array_equal(O.dequantize_act_group(q, s, z, group)[0], y)


def test_group_exact_ties_round_half_even():
    """Values exactly half-way between two grid points of Eq. 1 round to the
    even quotient: y / s = k + 1/2 - z0 goes to the even one of k - z0 and
    k + 1 - z0, for every k and for steps and zero-points that are powers of
    two, bf16-sized grids and shifted ranges alike."""
    for s0 in (2.0 ** -3, 0.75, 1.0, 3.0, 2.0 ** 5):
        for z0 in (-9, -1, 0, 3, 8, 21):
            ks = np.arange(15)
            y = s0 * np.concatenate([[0 - z0, 15 - z0], ks + 0.5 - z0])
            q, s, z = O.quantize_groups_asym(y[None, :], y.size)
            assert s[0, 0] == s0 and z[0, 0] == z0
            even = (ks - z0) % 2 == 0
            np.testing.assert_array_equal(q[0, 2:], np.where(even, ks, ks + 1))
            assert q[0, 0] == 0 and q[0, 1] == 15
    # A tie on the zero-point itself: min / s = -(z + 1/2) takes the even z.
    for zt in (2.5, 3.5, -4.5):
        mn = -zt
        y = np.array([mn, mn + 15.0, mn + 0.25])
        q, s, z = O.quantize_groups_asym(y[None, :], 3)
        assert s[0, 0] == 1.0 and z[0, 0] == (np.floor(zt) if np.floor(zt) % 2 == 0 else np.ceil(zt))


def test_group_eq5_two_channel_example(golden_dir):
    """Eq. 5's two-channel token: after H/sqrt(2) the outlier x1 is a common
    offset, so with one group of 2 the step is 2|x2| / (15 sqrt 2) whatever x1
    is, and the two channels take the ends of the grid."""
    d = _load(golden_dir, "eq5_two_channel.json")
    for case in d["cases"]:
        x = np.array([case["x"]], dtype=np.float64)
        res = O.quantize_act_group(x, 2, group=2, rotate=True)
        x2 = case["x"][1]
        np.testing.assert_allclose(res["y"][0], case["y"], rtol=1e-14)
        np.testing.assert_allclose(res["scale"][0, 0], 2 * abs(x2) / (15 * math.sqrt(2)), rtol=1e-12)
        # x2 = 0 leaves a constant group: s = z = q = 0 (the reading).
        expect = [15, 0] if x2 > 0 else [0, 15] if x2 < 0 else [0, 0]
        np.testing.assert_array_equal(res["q"][0], expect)


def test_group_rotation_absorbs_outlier():
    """A channel-0 outlier adds the same constant to every rotated channel of
    its block (Eq. 5): the group scales do not move, unlike the symmetric
    per-token scale, and the reconstruction stays within s / 2."""
    rng = np.random.default_rng(41)
    K, group = 512, 128
    base = rng.standard_normal((16, K))
    spiked = base.copy()
    spiked[:, 0] += rng.uniform(400, 2000, size=16)
    a = O.quantize_act_group(base, K, group, rotate=True)
    b = O.quantize_act_group(spiked, K, group, rotate=True)
    np.testing.assert_allclose(b["scale"], a["scale"], rtol=1e-9)
    err = np.abs(O.dequantize_act_group(b["q"], b["scale"], b["zero"], group) - b["y"])
    assert np.all(err <= np.repeat(b["scale"], group, axis=1) * (0.5 + 1e-9))
    sym = O.quantize_act(spiked, K, rotate=True, offset=False)
    assert np.all(sym["scale"] > 5 * b["scale"].max(axis=1))


def test_group_error_bound_and_ends():
    rng = np.random.default_rng(42)
    x = rng.standard_normal((32, 512)) * rng.uniform(0.01, 30, size=(32, 1)) + rng.uniform(-5, 5, size=(32, 1))
    for rotate in (False, True):
        res = O.quantize_act_group(x, 256, 128, rotate=rotate)
        q, s, z = res["q"], res["scale"], res["zero"]
        sg = np.repeat(s, 128, axis=1)
        err = np.abs(O.dequantize_act_group(q, s, z, 128) - res["y"])
        clamped = (q == 15) & (np.rint(res["y"] / sg) + np.repeat(z, 128, axis=1) > 15)
        assert np.all(err[~clamped] <= sg[~clamped] * (0.5 + 1e-9))
        assert np.all(err <= sg * (1 + 1e-9))
        yg = res["y"].reshape(32, 4, 128)
        qg = q.reshape(32, 4, 128)
        # The group minimum always lands on code 0; the maximum on 15 (14 only
        # when both ends sit on rounding ties of opposite parity).
        at_min = np.take_along_axis(qg, yg.argmin(axis=2)[..., None], axis=2)
        at_max = np.take_along_axis(qg, yg.argmax(axis=2)[..., None], axis=2)
        assert np.all(at_min == 0) and np.all(at_max >= 14)


def test_group_brute_force_small_groups():
    """Group of 4: each code is the index of the nearest point of the grid
    s (j - z), j = 0..15, ties to an even j - z."""
    rng = np.random.default_rng(43)
    j = np.arange(16)
    for trial in range(300):
        y = rng.standard_normal((1, 4)) * rng.uniform(0.01, 50) + rng.uniform(-20, 20)
        q, s, z = O.quantize_groups_asym(y, 4)
        for k in range(4):
            d = np.abs(y[0, k] - s[0, 0] * (j - z[0, 0]))
            best = j[d <= d.min() + 1e-12 * s[0, 0]]
            expect = best[0] if len(best) == 1 else best[(best - int(z[0, 0])) % 2 == 0][0]
            assert q[0, k] == expect


def test_group_constant_and_zero_groups():
    y = np.zeros((2, 256))
    y[1, 128:] = 3.25
    q, s, z = O.quantize_groups_asym(y, 128)
    assert np.all(s == 0) and np.all(z == 0) and np.all(q == 0)


def test_group_pack_roundtrip():
    rng = np.random.default_rng(44)
    q = rng.integers(0, 16, size=(3, 64))
    packed = O.pack_unsigned_codes(q)
    assert packed[0, 0] == (q[0, 0] | (q[0, 1] << 4))
    np.testing.assert_array_equal(O.unpack_act_codes(packed) + 8, q)


@pytest.mark.parametrize("rotate", [False, True])
def test_group_gemm_equals_dequantized_product(rotate):
    """s_w sum_j s_j (P_j - z_j R_j) is the product of the dequantized
    activations and weights, formed here by a plain float64 matmul."""
    rng = np.random.default_rng(45)
    T, K, N, g = 9, 512, 24, 256
    x = W.activations(T, K, seed=46, n_out=2, mult=80.0)
    w = rng.standard_normal((N, K)) * 0.02
    a = O.quantize_act_group(x, g, 128, rotate=rotate)
    wp = O.prepare_weight(w, g, rotate=rotate)
    R = O.weight_group_sums(wp["q"], 128)
    res = O.w4a4_linear_group(a["q"], a["scale"], a["zero"], wp["q"], wp["scale"], R, 128)
    xh = O.dequantize_act_group(a["q"], a["scale"], a["zero"], 128)
    wh = wp["q"] * wp["scale"][:, None]
    ref = xh @ wh.T
    np.testing.assert_allclose(res["y"], ref, rtol=1e-11, atol=1e-12 * np.abs(ref).max())
    # Each group's integer product, by the triple loop on a corner.
    np.testing.assert_array_equal(res["P"][1][:3, :4], O.int_gemm_loops(a["q"][:3, 128:256], wp["q"][:4, 128:256]))
    # And the group layer approximates the unquantized one.
    y32 = O.linear_reference(x, w)
    assert np.linalg.norm(res["y"] - y32) < 0.3 * np.linalg.norm(y32)


# --------------------------------------------------------------------------
# Key cache with a dense per-head rotation M = U3 P3 H3 (Sec. 3.3 Step 2 (3)).
# --------------------------------------------------------------------------

def _keys_with_outlier(T=96, H=2, hd=128, seed=50, mag=(20.0, 60.0)):
    rng = np.random.default_rng(seed)
    k = rng.standard_normal((T, H, hd))
    dirs = rng.standard_normal((H, hd))
    dirs /= np.linalg.norm(dirs, axis=1, keepdims=True)
    a = rng.uniform(*mag, size=(T, H))
    return k + a[:, :, None] * dirs[None], dirs, a


def test_householder_and_pca_direction():
    rng = np.random.default_rng(51)
    v = rng.standard_normal(128)
    U = O.householder_to_first(v)
    np.testing.assert_allclose(U, U.T, atol=1e-15)
    np.testing.assert_allclose(U @ U, np.eye(128), atol=1e-13)
    np.testing.assert_allclose(U[:, 0], v / np.linalg.norm(v), atol=1e-14)
    # Rank-one data plus tiny noise: the top-1 direction is the generating one.
    t = rng.uniform(1, 2, size=200)
    x = np.outer(t, v) + 1e-6 * rng.standard_normal((200, 128))
    np.testing.assert_allclose(O.top1_pca_direction(x), v / np.linalg.norm(v) * np.sign(v[np.argmax(np.abs(v))]),
                               atol=1e-6)


def test_key_rotation_is_orthonormal_and_keeps_scores():
    k, _, _ = _keys_with_outlier()
    q = np.random.default_rng(52).standard_normal(k.shape)
    perm = np.concatenate([[0], 1 + np.random.default_rng(53).permutation(127)])
    M = O.key_rotation(k, perm)
    for h in range(M.shape[0]):
        np.testing.assert_allclose(M[h] @ M[h].T, np.eye(128), atol=1e-13)
    qr, kr = O.rotate_heads(q, M), O.rotate_heads(k, M)
    for h in range(M.shape[0]):
        np.testing.assert_allclose(qr[:, h] @ kr[:, h].T, q[:, h] @ k[:, h].T, rtol=1e-11, atol=1e-9)


def test_dense_rotation_special_cases():
    """M = H/sqrt(hd) reproduces the per-head Hadamard quantizer; M = I the plain one."""
    k, _, _ = _keys_with_outlier(T=40)
    H = O.sylvester_hadamard(128).astype(np.float64) / math.sqrt(128)
    for rot, rotate in ((np.stack([H, H]), True), (np.stack([np.eye(128)] * 2), False)):
        a = O.kv4_quantize_dense(k, rot)
        b = O.kv4_quantize(k, rotate=rotate)
        np.testing.assert_allclose(a["scale"], b["scale"], rtol=1e-12)
        np.testing.assert_allclose(a["offset"], b["offset"], rtol=1e-12, atol=1e-12)
        t = b["residual"] / b["scale"][:, :, None]
        near = np.abs(np.abs(t) - np.floor(np.abs(t)) - 0.5) < 1e-9
        assert np.all((a["q"] == b["q"]) | near)


def test_u3_turns_the_outlier_into_an_offset():
    """k = n + a v: k U3 = n U3 + a e_1, and e_1 H3 / sqrt(hd) is constant, so
    the rotated outlier is the offset a / sqrt(hd) (Eq. 5) and the residual
    (hence scale and codes) does not depend on a."""
    rng = np.random.default_rng(54)
    T, hd = 32, 128
    n = rng.standard_normal((T, 1, hd))
    v = rng.standard_normal(hd)
    v /= np.linalg.norm(v)
    Hs = O.sylvester_hadamard(hd).astype(np.float64) / math.sqrt(hd)
    M = (O.householder_to_first(v) @ Hs)[None]
    base = O.kv4_quantize_dense(n, M)
    a = rng.uniform(100, 1000, size=(T, 1))
    spiked = O.kv4_quantize_dense(n + a[:, :, None] * v, M)
    np.testing.assert_allclose(spiked["offset"] - base["offset"], a / math.sqrt(hd), rtol=1e-12)
    np.testing.assert_allclose(spiked["scale"], base["scale"], rtol=1e-9)
    # The plain per-head Hadamard leaves the outlier in the residual.
    plain = O.kv4_quantize(n + a[:, :, None] * v, rotate=True)
    assert np.all(plain["scale"] > 5 * spiked["scale"])


def test_key_rotation_from_samples_offsets_the_outlier():
    """M built from key samples (U3 from their top-1 PCA, then P3, then H3)
    leaves the residual at the noise level; the outlier rides in the offset."""
    k, dirs, a = _keys_with_outlier(T=256, mag=(30.0, 90.0))
    perm = np.concatenate([[0], 1 + np.random.default_rng(55).permutation(127)])
    M = O.key_rotation(k, perm)
    with pytest.raises(ValueError):
        O.key_rotation(k, np.roll(np.arange(128), 1))
    rot = O.kv4_quantize_dense(k, M)
    noise = O.kv4_quantize_dense(k - a[:, :, None] * dirs[None], M)
    assert np.all(rot["scale"] < 1.5 * noise["scale"].max())
    assert np.all(np.abs(rot["offset"]) > 0.5 * a / math.sqrt(128))


# --------------------------------------------------------------------------
# Offline transform builder (Sec. 3.1 top-1 PCA, Sec. 3.2 sorted grouping,
# Sec. 3.3 Steps 1-2 fusion).
# --------------------------------------------------------------------------

def test_sorted_grouping_golden(golden_dir):
    d = _load(golden_dir, "sorted_grouping.json")
    vals = np.array(d["values"], dtype=np.float64)
    perm = O.sorted_grouping(vals, d["groups"])
    np.testing.assert_array_equal(vals[perm], d["sorted"])
    assert list(vals[perm]) != d["zigzag_not_used"]


def test_linf_selection_golden(golden_dir):
    d = _load(golden_dir, "linf_sphere.json")
    x = np.array([d["tokens"]])
    idx, rows = O.top1_tokens(x)
    assert idx[0] == d["selected"]
    np.testing.assert_allclose(np.max(np.abs(x[0]), axis=1), d["linf"])
    np.testing.assert_array_equal(rows[0], d["tokens"][d["selected"]])


def test_top1_pca_rank_one_and_power_iteration():
    """X = a v^T (+ tiny noise): the leading eigenvector is v (sign fixed) with
    eigenvalue mean(a^2); an independent power iteration agrees."""
    rng = np.random.default_rng(60)
    v = rng.standard_normal(256)
    v /= np.linalg.norm(v)
    a = rng.uniform(5, 10, size=64)
    X = np.outer(a, v)
    vv, lam1, lam2 = O.top1_pca(X)
    sign = 1.0 if v[np.argmax(np.abs(v))] > 0 else -1.0
    np.testing.assert_allclose(vv, sign * v, atol=1e-12)
    np.testing.assert_allclose(lam1, np.mean(a ** 2), rtol=1e-12)
    assert abs(lam2) < 1e-9
    Xn = X + 1e-3 * rng.standard_normal(X.shape)
    vv, _, _ = O.top1_pca(Xn)
    p = np.ones(256) / 16.0
    for _ in range(200):
        p = Xn.T @ (Xn @ p)
        p /= np.linalg.norm(p)
    assert abs(abs(p @ vv) - 1.0) < 1e-12


def test_offset_basis_orthonormal_and_fusion_exact():
    rng = np.random.default_rng(61)
    D, G = 256, 4
    v = rng.standard_normal(D)
    perm = O.sorted_grouping(rng.standard_normal(D), G)
    M = O.offset_basis(v, perm, D // G)
    np.testing.assert_allclose(M @ M.T, np.eye(D), atol=1e-12)
    x = rng.standard_normal((9, D))
    w = rng.standard_normal((7, D))
    np.testing.assert_allclose((x @ M) @ O.fuse_rotation(w, M).T, x @ w.T, rtol=1e-11, atol=1e-11)


def test_builder_turns_the_outlier_into_group_offsets():
    """Tokens n + a v (Sec. 3.1 structure): after M = U1 P1 H1 from the builder,
    v lands in the leading channel of a group and leaves as that group's
    constant offset a / sqrt(g) (Eq. 5); the residual no longer holds a."""
    rng = np.random.default_rng(62)
    S, L, D, G = 48, 16, 256, 4
    v = rng.standard_normal(D)
    v /= np.linalg.norm(v)
    x = rng.standard_normal((S, L, D))
    spikes = rng.integers(0, L, size=S)
    a = rng.uniform(80, 120, size=S)
    x[np.arange(S), spikes] += a[:, None] * v
    res = O.build_offset_transform(x, G)
    np.testing.assert_array_equal(res["index"], spikes)
    assert abs(abs(res["v"] @ v) - 1.0) < 1e-3
    g = D // G
    Xr = res["X"] @ res["M"]
    offs = Xr.reshape(S, G, g).mean(axis=2)
    gi = int(np.argmax(np.abs(offs).mean(axis=0)))
    np.testing.assert_allclose(np.abs(offs[:, gi]), (a + 0.0) / math.sqrt(g), rtol=0.05)
    # Statistical consequence (the exact one is the offset above): the 4-bit
    # step falls to the noise level.
    q_before = O.quantize_act(res["X"], g, rotate=False, offset=False)["scale"]
    q_after = O.quantize_act(Xr, g, rotate=False, offset=True)["scale"]
    assert np.all(q_after < 0.5 * q_before) and q_after.mean() < 0.25 * q_before.mean()


# --------------------------------------------------------------------------
# MXFP4 residuals with the offset as zero-point (Sec. 3.4, "Generality on
# Data Formats"; readings with quantize_mx_rows).
# --------------------------------------------------------------------------

def test_mx_rounding_fixture(golden_dir):
    d = _load(golden_dir, "mxfp4_blocks.json")
    v = np.array([e["v"] for e in d["rounding"]])
    np.testing.assert_array_equal(O.rne_e2m1(v), [e["code"] for e in d["rounding"]])
    for blk in d["blocks"]:
        res = O.quantize_mx_rows(np.array([blk["x"]]))
        assert res["X"][0, 0] == blk["X"]
        np.testing.assert_array_equal(res["code"][0], blk["code"])


def test_mx_grid_points_round_trip_and_error_bound():
    # Every E2M1 value comes back as its own code (-0 as +0).
    codes = np.arange(16)
    back = O.rne_e2m1(O.e2m1_value(codes))
    np.testing.assert_array_equal(back, np.where(codes == 8, 0, codes))
    # Monotone, and within half the local grid gap of the value (saturated values aside).
    v = np.linspace(-8, 8, 20001)
    q = O.e2m1_value(O.rne_e2m1(v))
    assert np.all(np.diff(q) >= 0)
    grid = np.concatenate([-O.E2M1_MAG[::-1], O.E2M1_MAG[1:]])
    inside = np.abs(v) <= 6
    gaps = np.diff(grid)
    idx = np.clip(np.searchsorted(grid, v[inside]) - 1, 0, len(gaps) - 1)
    assert np.all(np.abs(v[inside] - q[inside]) <= gaps[idx] / 2 + 1e-15)


def test_mx_block_exponent_places_the_largest_value_on_the_top_binades():
    rng = np.random.default_rng(45)
    r = rng.standard_normal((64, 256)) * np.exp(rng.uniform(-8, 8, size=(64, 1)))
    res = O.quantize_mx_rows(r)
    blk = np.abs(r.reshape(64, 8, 32)).max(axis=2)
    ratio = blk / np.ldexp(1.0, res["X"])
    unclamped = res["X"] > res["xmax"][:, None] - O.MX_SPAN
    assert np.all((ratio[unclamped] >= 4) & (ratio[unclamped] < 8))
    # The block maximum codes to magnitude 4 or 6 (or saturates at 6).
    mags = np.abs(O.e2m1_value(res["code"])).reshape(64, 8, 32).max(axis=2)
    assert np.all(np.isin(mags[unclamped], [4.0, 6.0]))
    # Reconstruction error: half a grid gap (at most 2^X) below saturation, 2 * 2^X at it.
    err = np.abs(res["value"] - r).reshape(64, 8, 32).max(axis=2)
    assert np.all(err <= 2 * np.ldexp(1.0, res["X"]) + 1e-300)


def test_mx_span_clamp_and_zero_blocks():
    r = np.zeros((1, 128))
    r[0, :32] = 1000.0 * np.linspace(-1, 1, 32)   # X = floor(log2 1000) - 2 = 7
    r[0, 32:64] = 1e-3                            # would be X = -12; clamped to 7 - 6 = 1
    res = O.quantize_mx_rows(r)
    np.testing.assert_array_equal(res["X"][0], [7, 1, 1, 1])
    np.testing.assert_array_equal(res["shift"][0], [6, 0, 0, 0])
    assert np.all(res["code"][0, 32:] == 0)       # 1e-3 / 2 rounds to 0
    assert res["row_scale"][0] == 2.0


def test_mx_offset_absorbs_the_outlier():
    """Eq. 5 through the MX residual: pairs [x1, x2] rotated by H_2 leave the constant
    offset x1 / sqrt 2 and residuals +-x2 / sqrt 2, so the codes and exponents do not
    depend on the outlier x1."""
    x2 = np.array([0.3, -1.7, 2.5, 0.9] * 8)
    base = np.stack([np.zeros(32), x2], axis=1).reshape(1, 64)
    for x1 in (0.0, 50.0, -400.0, 1e4):
        x = base.copy()
        x[0, 0::2] = x1
        res = O.quantize_act_mx(x, 2, rotate=True, offset=True)
        np.testing.assert_allclose(res["offset"][0], x1 / math.sqrt(2), rtol=1e-14)
        ref = O.quantize_act_mx(base, 2, rotate=True, offset=True)
        np.testing.assert_array_equal(res["code"], ref["code"])
        np.testing.assert_array_equal(res["X"], ref["X"])


def test_mx_linear_equals_the_dequantized_product():
    rng = np.random.default_rng(46)
    T, K, N, g = 12, 512, 40, 256
    x = rng.standard_normal((T, K))
    x[:, ::g] += 80.0
    w = rng.standard_normal((N, K)) * 0.02
    a = O.quantize_act_mx(x, g)
    wp = O.prepare_weight_mx(w, g)
    res = O.mx_linear(a, wp, g)
    xh = a["value"] + np.repeat(a["offset"], g, axis=1)
    ref = xh @ wp["value"].T
    np.testing.assert_allclose(res["y"], ref, rtol=1e-12, atol=1e-12 * np.abs(ref).max())
    np.testing.assert_allclose(res["y_factored"], ref, rtol=1e-12, atol=1e-12 * np.abs(ref).max())
    # The operand values are exact E4M3 numbers: multiples of 2^-1 up to 384.
    opv = np.abs(wp["operand"])
    assert opv.max() <= 384 and np.all(opv * 2 == np.round(opv * 2))
    # And the layer approximates the unquantized one (the rotation cancels).
    y32 = O.linear_reference(x, w)
    assert np.linalg.norm(res["y"] - y32) < 0.3 * np.linalg.norm(y32)


def test_mx_pack_and_shift_layouts():
    rng = np.random.default_rng(47)
    code = rng.integers(0, 16, size=(37, 256))
    p = O.pack_mx_codes(code)
    assert p[0, 0] == (code[0, 0] | (code[0, 1] << 4))
    np.testing.assert_array_equal(O.unpack_mx_codes(p), code)
    sh = rng.integers(0, 7, size=(37, 8))
    t = O.tile_mx_shifts(sh)
    # Row 33 (second 32-row block, row 1), block 5 (k-tile 1, position 1).
    assert t[((1 * 2 + 1) * 32 + 1) * 4 + 1] == sh[33, 5]
    np.testing.assert_array_equal(O.untile_mx_shifts(t, 37, 256), sh)
