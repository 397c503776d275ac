"""Pins for oracle/w8a8.py against things other than the oracle itself: exact rational
arithmetic, the quantiser's invariants, the textbook special case, a closed-form error bound
and library conversions."""
from fractions import Fraction

import numpy as np
import pytest
import torch

from oracle import w8a8 as W

F32 = np.float32


def _rne_int(fr: Fraction) -> int:
    """Round a rational to the nearest integer, ties to even (exact)."""
    fl = fr.numerator // fr.denominator
    rem = fr - fl
    if rem > Fraction(1, 2) or (rem == Fraction(1, 2) and fl % 2 == 1):
        return fl + 1
    return fl


# ------------------------------------------------------------------------------ bf16 helpers
def test_bf16_rounding_matches_torch_conversion():
    g = np.random.default_rng(1)
    x = np.concatenate([
        g.standard_normal(20000).astype(F32) * F32(100),
        np.array([0.0, -0.0, 1.0, np.inf, -np.inf, 3.4e38, -3.4e38, 1e-40, -1e-40], F32),
        # exact ties between two bf16 neighbours: 1 + 2^-8 (tie, even -> 1), 1 + 3*2^-8 (tie -> up)
        np.array([1 + 2 ** -8, 1 + 3 * 2 ** -8, -(1 + 2 ** -8), 256 + 1, 256 + 3], F32),
    ])
    ours = W.f32_to_bf16_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(ours, ref)
    assert np.isnan(W.round_to_bf16(np.array([np.nan], F32)))[0]


# ------------------------------------------------------------------------------- quantiser
def test_quantize_rows_against_exact_rounding():
    """Every code equals round-half-even of the exact x * 127 / m, except where the exact value
    lies within a few fp32 ulps of a half-integer (the reciprocal is rounded once, the product
    once); codes never exceed 127; the scale is m / 127 rounded once."""
    g = np.random.default_rng(2)
    A = (g.standard_normal((7, 96)) * g.uniform(0.01, 50, size=(7, 1))).astype(F32)
    q, s = W.quantize_rows(A)
    assert q.dtype == np.int8 and np.abs(q.astype(int)).max() <= 127
    for i in range(A.shape[0]):
        m = Fraction(float(np.max(np.abs(A[i]))))
        assert float(s[i]) == float(np.float32(float(m / 127)))
        for j in range(A.shape[1]):
            exact = Fraction(float(A[i, j])) * 127 / m
            frac = abs(exact - (exact.numerator // exact.denominator)) if exact >= 0 else None
            near_tie = abs(abs(exact - int(exact)) - Fraction(1, 2)) < Fraction(1, 2 ** 16)
            if not near_tie:
                assert int(q[i, j]) == _rne_int(exact), (i, j, float(exact), frac)


def test_absmax_maps_to_127_with_sign():
    g = np.random.default_rng(3)
    A = g.standard_normal((50, 33)).astype(F32)
    q, _ = W.quantize_rows(A)
    for i in range(A.shape[0]):
        j = int(np.argmax(np.abs(A[i])))
        assert int(q[i, j]) == (127 if A[i, j] > 0 else -127)


def test_half_step_dequant_bound():
    """|a - s * q| <= s/2 (plus the rounding of the reciprocal and of s) for every element."""
    g = np.random.default_rng(4)
    A = (g.standard_normal((40, 200)) * 3).astype(F32)
    A[:, 7] *= 40
    q, s = W.quantize_rows(A)
    err = np.abs(A.astype(np.float64) - s[:, None].astype(np.float64) * q)
    bound = s[:, None].astype(np.float64) / 2 * (1 + 2 ** -20) + np.abs(A) * 2 ** -22
    assert np.all(err <= bound)


def test_round_half_to_even_on_exact_ties():
    """With row absmax 127 the reciprocal 127/m is exactly 1, so x = k + 1/2 is an exact tie."""
    A = np.array([[127.0, 2.5, 3.5, -2.5, -3.5, 0.5, 1.5, -0.5, 126.5]], F32)
    q, s = W.quantize_rows(A)
    assert s[0] == F32(1.0)
    assert q[0].tolist() == [127, 2, 4, -2, -4, 0, 2, 0, 126]


def test_zero_rows_and_zero_statistics():
    A = np.zeros((2, 16), F32)
    A[1, 3] = 5.0
    q, s = W.quantize_rows(A)
    assert s[0] == 0 and not q[0].any() and q[1, 3] == 127
    delta, inv = W.smoothing_factors(np.array([0, 4, 9], F32), np.array([1, 0, 4], F32))
    assert delta.tolist() == [1.0, 1.0, 1.5] and inv.tolist() == [1.0, 1.0, F32(1 / 1.5)]
    x = np.zeros((1, 8), F32)
    prep = W.prepare_weights(np.ones((3, 8), F32), np.ones(8, F32))
    bias = np.array([0.25, -1.0, 3.0], F32)
    r = W.w8a8_linear(x, prep, bias=bias, out="f32")
    assert r["s_x"][0] == 0 and not r["xq"].any() and np.array_equal(r["y"][0], bias)


# ---------------------------------------------------------------------- smoothing factors
def test_smoothing_factor_balances_maxima():
    """With alpha = 0.5 the smoothed activation and weight column maxima are equal:
    max|x_j / delta_j| = max|W_ij * delta_j| = sqrt(ax_j * aw_j) (SmoothQuant's migration);
    for general alpha they are ax^(1-a) aw^(1-a) and ax^a aw^a."""
    g = np.random.default_rng(5)
    ax = g.uniform(0.1, 40, 64).astype(F32)
    aw = g.uniform(0.001, 0.2, 64).astype(F32)
    for alpha in (0.5, 0.3, 0.8):
        delta, inv = W.smoothing_factors(ax, aw, alpha)
        d64 = ax.astype(np.float64) ** alpha / aw.astype(np.float64) ** (1 - alpha)
        assert np.all(np.abs(delta / d64 - 1) <= 3 * 2 ** -24)
        xs = ax / delta.astype(np.float64)
        ws = aw * delta.astype(np.float64)
        assert np.allclose(xs, ax.astype(np.float64) ** (1 - alpha) * aw.astype(np.float64) ** (1 - alpha), rtol=1e-6)
        assert np.allclose(ws, ax.astype(np.float64) ** alpha * aw.astype(np.float64) ** alpha, rtol=1e-6)
        assert np.array_equal(inv, (F32(1) / delta).astype(F32))


def test_smoothing_leaves_product_unchanged():
    """sum_j (x_j / delta_j)(W_ij delta_j) = sum_j x_j W_ij: exactly in rational arithmetic
    with the oracle's delta, and to K * 2^-23 relative with the oracle's fp32 x_hat and W_hat."""
    g = np.random.default_rng(6)
    M, K, N = 3, 32, 5
    X = g.standard_normal((M, K)).astype(F32)
    X[:, 4] *= 20
    Wt = (g.standard_normal((N, K)) * 0.02).astype(F32)
    delta, inv = W.smoothing_factors(W.act_absmax(X), W.weight_col_absmax(Wt))
    for t in range(M):
        for i in range(N):
            exact = sum(Fraction(float(X[t, j])) / Fraction(float(delta[j])) * Fraction(float(Wt[i, j])) *
                        Fraction(float(delta[j])) for j in range(K))
            plain = sum(Fraction(float(X[t, j])) * Fraction(float(Wt[i, j])) for j in range(K))
            assert exact == plain
    xh = W.smooth_activations(X, inv).astype(np.float64)
    wh = W.smooth_weights(Wt, delta).astype(np.float64)
    ref = X.astype(np.float64) @ Wt.astype(np.float64).T
    mag = np.abs(X).astype(np.float64) @ np.abs(Wt).astype(np.float64).T
    assert np.all(np.abs(xh @ wh.T - ref) <= K * 2 ** -22 * mag)


# ------------------------------------------------------------------------------ INT8 GEMM
def test_int_gemm_against_python_ints():
    g = np.random.default_rng(7)
    xq = g.integers(-127, 128, (3, 40)).astype(np.int8)
    wq = g.integers(-127, 128, (5, 40)).astype(np.int8)
    acc = W.int_gemm(xq, wq)
    for t in range(3):
        for i in range(5):
            assert acc[t, i] == sum(int(xq[t, j]) * int(wq[i, j]) for j in range(40))


def test_int_gemm_adversarial_extremes():
    """All-(+-127) operands at K = 6912 reach |acc| = 127^2 * 6912, far beyond 2^24."""
    K = 6912
    xq = np.full((2, K), 127, np.int8)
    xq[1, ::2] = -127
    wq = np.full((3, K), 127, np.int8)
    wq[1] = -127
    wq[2, 1::3] = -127
    acc = W.int_gemm(xq, wq)
    ref = xq.astype(np.int64) @ wq.astype(np.int64).T
    assert np.array_equal(acc, ref) and acc[0, 0] == 127 * 127 * K


def test_textbook_special_case_integer_grid():
    """delta = 1 and operands already on the integer grid with row absmax 127: every scale is 1,
    the codes are the operands and y is the exact integer matmul (rounded to bf16)."""
    g = np.random.default_rng(8)
    X = g.integers(-127, 128, (4, 64)).astype(F32)
    X[:, 0] = 127
    Wt = g.integers(-127, 128, (6, 64)).astype(F32)
    Wt[:, 5] = -127
    prep = W.prepare_weights(Wt, np.ones(64, F32), smooth=False)
    assert np.all(prep["s_w"] == 1) and np.array_equal(prep["wq"].astype(F32), Wt)
    r = W.w8a8_linear(X, prep, out="f32")
    exact = X.astype(np.int64) @ Wt.astype(np.int64).T
    assert np.all(r["s_x"] == 1) and np.array_equal(r["xq"].astype(F32), X)
    assert np.array_equal(r["y"].astype(np.float64), exact.astype(np.float32).astype(np.float64))
    rb = W.w8a8_linear(X, prep, out="bf16")
    assert np.array_equal(rb["y"], W.round_to_bf16(exact.astype(F32)))


def test_error_bound_closed_form():
    """|y - x W^T| <= (s_w/2) sum|x_hat| + (s_t/2) sum|W_hat| + K s_t s_w / 4 (+ fp32 slack),
    for every output of a smoothed linear with outlier channels."""
    g = np.random.default_rng(9)
    M, K, N = 8, 256, 48
    X = g.standard_normal((M, K)).astype(F32)
    X[:, [3, 100, 201]] *= 20
    X = W.round_to_bf16(X)
    Wt = W.round_to_bf16((g.standard_normal((N, K)) * 0.02).astype(F32))
    prep = W.prepare_weights(Wt, W.act_absmax(X))
    r = W.w8a8_linear(X, prep, out="f32")
    ref = X.astype(np.float64) @ Wt.astype(np.float64).T
    xh = np.abs(W.smooth_activations(X, prep["inv_delta"])).astype(np.float64)
    wh = np.abs(W.smooth_weights(Wt, prep["delta"])).astype(np.float64)
    st = r["s_x"].astype(np.float64)[:, None]
    sw = prep["s_w"].astype(np.float64)[None, :]
    bound = sw / 2 * xh.sum(1)[:, None] + st / 2 * wh.sum(1)[None, :] + K * st * sw / 4
    slack = 1e-5 * (np.abs(X).astype(np.float64) @ np.abs(Wt).astype(np.float64).T) + 1e-6
    assert np.all(np.abs(r["y"] - ref) <= bound + slack)
    # a dropped scale or a transposed smoothing factor would break the bound by orders of magnitude
    assert np.abs(r["y"] - ref).max() < 0.2 * np.abs(ref).max()


def test_bf16_linear_is_correctly_rounded_exact_sum():
    g = np.random.default_rng(10)
    X = W.round_to_bf16(g.standard_normal((2, 24)).astype(F32))
    Wt = W.round_to_bf16(g.standard_normal((3, 24)).astype(F32))
    y32 = W.bf16_linear(X, Wt, out="f32")
    for t in range(2):
        for i in range(3):
            exact = sum(Fraction(float(X[t, j])) * Fraction(float(Wt[i, j])) for j in range(24))
            assert abs(Fraction(float(y32[t, i])) - exact) <= abs(exact) * Fraction(1, 2 ** 24) + Fraction(1, 2 ** 120)


def test_top1_ties_lowest_index():
    z = np.array([[1.0, 3.0, 3.0, -1.0], [5.0, 5.0, 5.0, 5.0]], F32)
    assert W.top1(z).tolist() == [1, 0]
