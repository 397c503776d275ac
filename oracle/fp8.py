"""Oracle: the FP8 (e4m3) variant of the W8A8 linear (test infrastructure; no kernel yet).

The paper names the move from INT8 to FP8 on Blackwell as the next step (its Future Work list:
FP8 GEMMs ran the FFN 1.46x faster than INT8's 1.10x) but gives no scheme.  Reading used here:
the INT8 path's SmoothQuant structure unchanged, with the e4m3 grid in place of the integers:
  * weights: W_hat = W * delta (Eq. what-lmhead), s_i^W = max_j |W_hat_ij| / 448, codes
    e4m3(W_hat_ij * fl32(448 / max_j |W_hat_ij|));
  * activations: x_hat = x * (1 / delta) (Eq. xhat-lmhead), s_t^x = max_j |x_hat_tj| / 448, codes
    e4m3(x_hat_tj * fl32(448 / m_t)), per token;
  * acc_ti = sum_j xq_tj * wq_ij, exactly (fp64: every product of two e4m3 values has at most 8
    significant bits between 2^-18 and 448^2 < 2^18, and K <= 6912 adds 13 bits of growth, 49
    bits in all, inside fp64's 53);
  * y = fl32(fl32(s_t^x * s_i^W) * fl32(acc)) (+ bias), as Eq. gemm-final orders it for INT8.
e4m3 here is the OCP 8-bit float E4M3 ("fn"): 1 sign, 4 exponent bits with bias 7, 3 mantissa
bits, subnormals down to 2^-9, no infinities, the all-ones pattern NaN, largest finite value 448.
Rounding is to nearest, ties to even, saturating at +-448 (the conversion the GPU offers with
.satfinite).  Parity unpinned against the paper (it prints no FP8 numbers to match); pinned to
the format's definition, to torch's e4m3 cast inside the range, and to closed-form bounds.
"""
from __future__ import annotations

import numpy as np

from . import w8a8 as OW

E4M3_MAX = 448.0
E4M3_MIN_NORMAL = 2.0 ** -6
E4M3_MIN_SUBNORMAL = 2.0 ** -9


def e4m3_round(x: np.ndarray) -> np.ndarray:
    """Nearest e4m3 value of x (float64 result), ties to even, saturating at +-448; NaN stays NaN.
    The spacing is 2^(e-3) in the binade [2^e, 2^(e+1)) for e >= -6 and 2^-9 below 2^-6, so
    |x| / spacing is rounded half-to-even to an integer (exact: spacings are powers of two)."""
    x = np.asarray(x, dtype=np.float64)
    a = np.abs(x)
    _, e = np.frexp(np.where(a > 0, a, 1.0))  # a = f 2^e with f in [0.5, 1): floor(log2 a) = e - 1
    q = np.where(a >= E4M3_MIN_NORMAL, np.ldexp(1.0, (e - 1) - 3), E4M3_MIN_SUBNORMAL)
    r = np.minimum(np.rint(a / q) * q, E4M3_MAX)
    return np.where(np.isnan(x), np.nan, np.copysign(r, x))


def e4m3_decode(codes: np.ndarray) -> np.ndarray:
    """Value of 8-bit e4m3 codes (uint8): sign | 4 exponent bits | 3 mantissa bits."""
    c = np.asarray(codes, dtype=np.uint8).astype(np.int64)
    s = np.where(c & 0x80, -1.0, 1.0)
    ex, mt = (c >> 3) & 0xF, c & 0x7
    v = np.where(ex == 0, mt * 2.0 ** -9, (1.0 + mt / 8.0) * np.ldexp(1.0, ex - 7))
    return np.where((ex == 0xF) & (mt == 0x7), np.nan, s * v)


def e4m3_encode(x: np.ndarray) -> np.ndarray:
    """8-bit code of e4m3_round(x) (uint8); NaN becomes 0x7F, -0 the sign bit alone."""
    r = e4m3_round(x)
    a = np.abs(r)
    sign = np.where(np.signbit(r), 0x80, 0).astype(np.int64)
    _, e = np.frexp(np.where(a > 0, a, 1.0))
    ex = (e - 1) + 7
    normal = a >= E4M3_MIN_NORMAL
    mant = np.where(normal, np.rint((a / np.ldexp(1.0, e - 1) - 1.0) * 8.0), np.rint(a / E4M3_MIN_SUBNORMAL))
    code = sign | np.where(normal, (ex << 3) | mant.astype(np.int64), mant.astype(np.int64))
    return np.where(np.isnan(r), 0x7F, code).astype(np.uint8)


def quantize_rows_fp8(A: np.ndarray):
    """Per-row e4m3 quantisation with the INT8 rule's arithmetic and 448 in place of 127:
    m = max_j |A_j| (fp32), s = fl32(m / 448), codes = e4m3(fl32(A_j * fl32(448 / m)));
    a zero row has s = 0 and zero codes.  Returns (code values as float64, s as float32)."""
    A = np.asarray(A, dtype=np.float32)
    m = np.abs(A).max(axis=1).astype(np.float32)
    safe = np.where(m > 0, m, np.float32(1.0)).astype(np.float32)
    r = np.where(m > 0, np.float32(E4M3_MAX) / safe, np.float32(0.0)).astype(np.float32)
    scaled = (A * r[:, None]).astype(np.float32)
    s = (m / np.float32(E4M3_MAX)).astype(np.float32)
    return e4m3_round(scaled.astype(np.float64)), s


def prepare_weights_fp8(W: np.ndarray, act_stat, alpha: float = 0.5, smooth: bool = True):
    """Offline preparation of one linear for the FP8 variant: the INT8 path's smoothing factors
    (Eq. delta-lmhead; delta = 1 without smoothing), then per-output-channel e4m3 codes."""
    W = np.asarray(W, dtype=np.float32)
    if smooth:
        delta, inv_delta = OW.smoothing_factors(np.asarray(act_stat, np.float32), OW.weight_col_absmax(W), alpha)
    else:
        delta = np.ones(W.shape[1], np.float32)
        inv_delta = np.ones(W.shape[1], np.float32)
    wq, s_w = quantize_rows_fp8(OW.smooth_weights(W, delta))
    return {"wq": wq, "s_w": s_w, "delta": delta, "inv_delta": inv_delta}


def fp8_linear(X: np.ndarray, prep: dict, bias=None, out: str = "bf16"):
    """y = fl32(fl32(s_x s_w) * fl32(acc)) (+ bias) of the FP8 variant; acc exact in fp64.
    Returns dict with xq (code values), s_x, acc (fp64) and y (fp32 or rounded to bf16)."""
    xh = OW.smooth_activations(np.asarray(X, np.float32), prep["inv_delta"])
    xq, s_x = quantize_rows_fp8(xh)
    acc = xq @ prep["wq"].T
    scale = (s_x[:, None] * prep["s_w"][None, :]).astype(np.float32)
    y = (scale * acc.astype(np.float32)).astype(np.float32)
    if bias is not None:
        y = (y + np.asarray(bias, np.float32)[None, :]).astype(np.float32)
    if out == "bf16":
        y = OW.round_to_bf16(y)
    return {"xq": xq, "s_x": s_x, "acc": acc, "y": y}
