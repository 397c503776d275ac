"""The FP8 (e4m3) oracle pinned to the format's definition, to torch's e4m3 cast inside the finite
range (a library routine), and to closed forms (CPU)."""
import numpy as np
import pytest
import torch

from oracle import fp8


def test_hand_checked_values():
    x = np.array([1.0625, 1.1875, 300.0, 500.0, -2.5, 2.0 ** -10, 3 * 2.0 ** -10, 2.0 ** -9, 447.9, 464.0,
                  1.96875, 0.0, 17.0, 0.0146484375])
    want = np.array([1.0,      # tie between 1 and 1.125: even mantissa
                     1.25,     # tie between 1.125 and 1.25: even mantissa
                     288.0,    # spacing 32 above 256
                     448.0,    # saturated
                     -2.5, 0.0,  # 2^-10: tie between 0 and 2^-9
                     2.0 ** -8,  # 1.5 subnormal steps: tie, even
                     2.0 ** -9, 448.0, 448.0, 2.0, 0.0,
                     16.0,     # tie between 16 and 18
                     0.015625])  # 0.0146484375 = 7.5 x 2^-9: tie between 7 and 8 subnormal steps
    assert np.array_equal(fp8.e4m3_round(x), want)
    assert np.isnan(fp8.e4m3_round(np.array([np.nan])))[0]


def test_code_table():
    codes = np.arange(256, dtype=np.uint8)
    v = fp8.e4m3_decode(codes)
    fin = np.isfinite(v)
    assert fin.sum() == 254 and set(codes[~fin].tolist()) == {0x7F, 0xFF}
    pos = v[fin & (v > 0)]
    assert pos.size == 126 and pos.max() == 448.0 and pos.min() == 2.0 ** -9
    assert np.array_equal(fp8.e4m3_encode(v[fin]), codes[fin])
    assert np.array_equal(fp8.e4m3_round(v[fin]), v[fin])  # every value is its own rounding


def test_matches_torch_cast_inside_range():
    g = np.random.default_rng(0)
    mag = np.exp(g.uniform(np.log(2.0 ** -12), np.log(448.0), 200_000))
    x = (mag * g.choice([-1.0, 1.0], mag.size)).astype(np.float32)
    ref = torch.from_numpy(x).to(torch.float8_e4m3fn).to(torch.float64).numpy()
    assert np.array_equal(fp8.e4m3_round(x.astype(np.float64)), ref)


def test_rounding_is_nearest_and_monotone():
    g = np.random.default_rng(1)
    x = np.sort(g.uniform(-460.0, 460.0, 50_000))
    r = fp8.e4m3_round(x)
    assert np.all(np.diff(r) >= 0)
    grid = np.unique(fp8.e4m3_decode(np.arange(256, dtype=np.uint8)))
    grid = grid[np.isfinite(grid)]
    inside = np.abs(x) <= 448.0
    nearest = np.abs(grid[None, :] - x[inside][:1000, None]).min(axis=1)
    assert np.allclose(np.abs(r[inside][:1000] - x[inside][:1000]), nearest, rtol=0, atol=0)


def test_quantize_rows_scale_and_extreme_code():
    g = np.random.default_rng(2)
    A = (g.standard_normal((40, 96)) * np.exp(g.uniform(-6, 6, (40, 1)))).astype(np.float32)
    A[3] = 0.0
    q, s = fp8.quantize_rows_fp8(A)
    m = np.abs(A).max(axis=1).astype(np.float32)
    assert np.array_equal(s, (m / np.float32(448.0)).astype(np.float32))
    live = m > 0
    assert np.all(np.abs(q[live]).max(axis=1) == 448.0) and not q[3].any() and s[3] == 0.0
    r = (np.float32(448.0) / m[live]).astype(np.float32)
    scaled = (A[live] * r[:, None]).astype(np.float32).astype(np.float64)
    err = np.abs(scaled - q[live])
    assert np.all(err <= np.maximum(np.abs(scaled) * 2.0 ** -4, 2.0 ** -10))  # half a spacing


def test_linear_on_the_grid_is_the_exact_matmul():
    """delta = 1, every row's absmax 448 and all values on the e4m3 grid: scales are 1, codes are the
    values, and y is the exact product (rounded to fp32 once, then bf16)."""
    g = np.random.default_rng(3)
    grid = fp8.e4m3_decode(np.arange(256, dtype=np.uint8))
    grid = grid[np.isfinite(grid)]
    X = g.choice(grid, (5, 64)).astype(np.float32)
    W = g.choice(grid, (7, 64)).astype(np.float32)
    X[:, 0] = 448.0
    W[:, 1] = -448.0
    prep = fp8.prepare_weights_fp8(W, None, smooth=False)
    r = fp8.fp8_linear(X, prep, out="f32")
    assert np.all(prep["s_w"] == 1.0) and np.all(r["s_x"] == 1.0)
    exact = X.astype(np.float64) @ W.astype(np.float64).T
    assert np.array_equal(r["acc"], exact)
    assert np.array_equal(r["y"], exact.astype(np.float32))


@pytest.mark.parametrize("smooth", [True, False])
def test_linear_error_bound(smooth):
    """|y - X W^T| <= (2^-4 + 2^-4 + 2^-8) sum_j |x_hat_j| |w_hat_ij| + the subnormal floor terms +
    fp32 slack: each e4m3 code is within half a spacing (2^-4 relative, or 2^-10 of the scale) of
    its scaled value, on both operands."""
    g = np.random.default_rng(4)
    K = 256
    X = g.standard_normal((6, K)).astype(np.float32)
    X[:, 5] *= 20.0  # an outlier channel
    W = (0.02 * g.standard_normal((9, K))).astype(np.float32)
    prep = fp8.prepare_weights_fp8(W, np.abs(X).max(axis=0), smooth=smooth)
    r = fp8.fp8_linear(X, prep, out="f32")
    xh = np.abs(X.astype(np.float64) * prep["inv_delta"].astype(np.float64))
    wh = np.abs(W.astype(np.float64) * prep["delta"].astype(np.float64))
    mag = xh @ wh.T
    s_x = r["s_x"].astype(np.float64)[:, None]
    s_w = prep["s_w"].astype(np.float64)[None, :]
    floor = 2.0 ** -10 * (s_x * wh.sum(axis=1)[None, :] + s_w * xh.sum(axis=1)[:, None]) * 1.1
    bound = (2 * 2.0 ** -4 + 2.0 ** -8) * mag + floor + 1e-5 * mag + 1e-30
    exact = X.astype(np.float64) @ W.astype(np.float64).T
    assert np.all(np.abs(r["y"] - exact) <= bound)
    # and the bound is not vacuous: the error is a visible fraction of it somewhere
    assert np.max(np.abs(r["y"] - exact) / bound) > 0.01


def test_fp8_ffn_block_stages_chain():
    """The FP8 block's stages chain: h is bf16(geglu(g, u)) of the fp32 gate/up outputs, down's
    codes are those of that h, and the block stays within the quantisation error of the bf16 block."""
    import synth
    from oracle import blocks, geglu
    from oracle import w8a8 as W
    c = synth.ffn_case(3, seed=0, hidden=64, inter=96, calib_rows=16)
    prep = blocks.prepare_ffn_fp8(c["wg32"], c["wu32"], c["wd32"], W.act_absmax(c["calib32"]), c["stat_h"])
    r = blocks.ffn_fp8(c["x32"], prep)
    assert np.array_equal(r["h"], W.round_to_bf16(geglu.geglu_f32(r["g"], r["u"])))
    xq, _ = fp8.quantize_rows_fp8(W.smooth_activations(r["h"], prep["down"]["inv_delta"]))
    assert np.array_equal(xq, r["down"]["xq"])
    ref = blocks.ffn_bf16(c["x32"], c["wg32"], c["wu32"], c["wd32"])
    assert np.abs(r["y"] - ref["y"]).max() < 0.1 * np.abs(ref["y"]).max()
