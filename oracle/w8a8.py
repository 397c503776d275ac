"""Oracle: the W8A8 SmoothQuant linear, one paper step per function (test infrastructure).

Each function restates one equation of the paper in plain numpy.  Wherever a floating-point
value decides an integer (an INT8 code, a scale that multiplies an exact INT32 sum), the
step is evaluated in IEEE fp32 with every operation rounded to nearest-even, because that is
the precision the GPU path decides in and both sides must decide identically.  Sums that
the paper defines exactly (the INT8 dot products, the bf16 pass-through) are evaluated
exactly or in fp64.

Readings of points the paper leaves open:
  * round() is round-half-to-even (np.rint); codes are clamped to [-127, 127]
    (2^(b-1) - 1 with b = 8, Eq. si), so -128 never occurs.
  * x / s with s = m / 127 is evaluated as x * (127 / m): one fp32 division per row or
    token, then one rounded multiply per element.
  * x_j / delta_j is evaluated as x_j * inv_delta_j with inv_delta_j = fl32(1 / delta_j).
  * An all-zero row or token gives scale 0 and codes 0; a zero calibration or weight
    statistic gives delta_j = 1.
  * The dequantising product of Eq. gemm-final is evaluated left to right:
    y = fl32(fl32(s_t^x * s_i^W) * fl32(acc)), then + bias (fl32), then the output rounding.
"""
from __future__ import annotations

import numpy as np

F32 = np.float32
QMAX = 127  # 2^(b-1) - 1 with b = 8 (Eq. si)


# --------------------------------------------------------------------------- bf16 helpers
def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """Exact widening of raw bf16 bit patterns (uint16) to fp32."""
    b = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return b.view(np.float32)


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """fp32 -> bf16 bit pattern, round to nearest, ties to even; NaN stays a quiet NaN."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    lsb = (u >> np.uint64(16)) & np.uint64(1)
    r = ((u + np.uint64(0x7FFF) + lsb) >> np.uint64(16)).astype(np.uint16)
    nan = np.isnan(x)
    if nan.any():
        r = r.copy()
        r[nan] = ((u[nan] >> np.uint64(16)).astype(np.uint16)) | np.uint16(0x0040)
    return r


def round_to_bf16(x: np.ndarray) -> np.ndarray:
    """Value of fp32 x after rounding to bf16 (returned as fp32)."""
    return bf16_bits_to_f32(f32_to_bf16_bits(x))


# ------------------------------------------------------------------ calibration statistics
def act_absmax(X: np.ndarray) -> np.ndarray:
    """max_t |X_{t,j}| per input channel j over the calibration tokens (Eq. delta-attn numerator;
    the LM Head section collects it with a forward hook over N calibration tokens)."""
    X = np.asarray(X, dtype=np.float32)
    if X.shape[0] == 0:
        return np.zeros(X.shape[1], dtype=np.float32)
    return np.max(np.abs(X), axis=0).astype(np.float32)


def weight_col_absmax(W: np.ndarray) -> np.ndarray:
    """max_i |W_{i,j}| per input channel j over all output rows (Eq. delta-attn denominator)."""
    return np.max(np.abs(np.asarray(W, dtype=np.float32)), axis=0).astype(np.float32)


# ------------------------------------------------------------------------- smoothing factor
def smoothing_factors(ax: np.ndarray, aw: np.ndarray, alpha: float = 0.5):
    """Eq. delta-attn / delta-lmhead: delta_j = max_t|X_tj|^alpha / max_i|W_ij|^(1-alpha).

    alpha = 0.5 (the paper's value) is evaluated as fl32(sqrt(ax)) / fl32(sqrt(aw)), each step
    correctly rounded.  Any other alpha is taken as an fp32 number (the precision in which it is
    specified), and the quotient is evaluated in fp64 and rounded once to fp32.
    A zero statistic on either side gives delta_j = 1.  Returns (delta, inv_delta) with
    inv_delta = fl32(1 / delta).
    """
    ax = np.asarray(ax, dtype=np.float32)
    aw = np.asarray(aw, dtype=np.float32)
    if alpha == 0.5:
        with np.errstate(divide="ignore", invalid="ignore"):
            delta = (np.sqrt(ax) / np.sqrt(aw)).astype(np.float32)
    else:
        a = float(np.float32(alpha))
        with np.errstate(divide="ignore", invalid="ignore"):
            d64 = np.power(ax.astype(np.float64), a) / np.power(aw.astype(np.float64), 1.0 - a)
        delta = d64.astype(np.float32)
    degenerate = (ax == 0) | (aw == 0) | ~np.isfinite(delta) | (delta == 0)
    delta = np.where(degenerate, F32(1.0), delta).astype(np.float32)
    inv_delta = (F32(1.0) / delta).astype(np.float32)
    return delta, inv_delta


def smooth_weights(W: np.ndarray, delta: np.ndarray) -> np.ndarray:
    """Eq. what-lmhead: W_hat_{i,j} = W_{i,j} * delta_j (fp32, rounded)."""
    return (np.asarray(W, dtype=np.float32) * delta[None, :]).astype(np.float32)


def smooth_activations(X: np.ndarray, inv_delta: np.ndarray) -> np.ndarray:
    """Eq. xhat-lmhead: x_hat_j = x_j / delta_j, evaluated as x_j * inv_delta_j (fp32)."""
    return (np.asarray(X, dtype=np.float32) * inv_delta[None, :]).astype(np.float32)


# ----------------------------------------------------------------------- symmetric quantiser
def quantize_rows(A: np.ndarray):
    """Symmetric per-row INT8 quantisation shared by Eq. si / what-ffn (weights, per output
    channel i) and Eq. stx / xint8 (activations, per token t).

    m = max_j |A_j|;  s = fl32(m / 127);  q_j = clamp(rint(fl32(A_j * fl32(127 / m))), -127, 127).
    A zero row gives s = 0 and q = 0.  Returns (q int8 [R, C], s fp32 [R]).
    """
    A = np.asarray(A, dtype=np.float32)
    m = np.max(np.abs(A), axis=1).astype(np.float32) if A.shape[1] else np.zeros(A.shape[0], np.float32)
    s = (m / F32(QMAX)).astype(np.float32)
    nz = m > 0
    r = np.zeros_like(m)
    r[nz] = (F32(QMAX) / m[nz]).astype(np.float32)
    prod = (A * r[:, None]).astype(np.float32)
    q = np.clip(np.rint(prod), -QMAX, QMAX).astype(np.int8)
    q[~nz] = 0
    return q, s


def prepare_weights(W: np.ndarray, act_stat: np.ndarray, alpha: float = 0.5, smooth: bool = True):
    """Offline weight preparation of one linear (LM Head section, Eq. delta-lmhead, what-lmhead,
    then Eq. si / what-ffn on the smoothed rows).

    W: fp32 values of the bf16 weight [N, K] (row i = output channel).  act_stat: max_t|X_tj|
    from calibration.  smooth=False gives delta = 1 (the paper's no-smoothing ablation).
    Returns dict(wq int8 [N,K], s_w fp32 [N], delta fp32 [K], inv_delta fp32 [K]).
    """
    W = np.asarray(W, dtype=np.float32)
    K = W.shape[1]
    if smooth:
        delta, inv_delta = smoothing_factors(act_stat, weight_col_absmax(W), alpha)
    else:
        delta = np.ones(K, np.float32)
        inv_delta = np.ones(K, np.float32)
    wq, s_w = quantize_rows(smooth_weights(W, delta))
    return {"wq": wq, "s_w": s_w, "delta": delta, "inv_delta": inv_delta}


def quantize_activations(X: np.ndarray, inv_delta: np.ndarray):
    """Dynamic per-token quantisation of the smoothed input (Eq. xhat-lmhead, stx, xint8).
    Returns (xq int8 [M,K], s_x fp32 [M])."""
    return quantize_rows(smooth_activations(X, inv_delta))


# ---------------------------------------------------------------------------- INT8 GEMM
def int_gemm(xq: np.ndarray, wq: np.ndarray) -> np.ndarray:
    """The integer sum of Eq. gemm-final: acc_{t,i} = sum_j xq_{t,j} * wq_{i,j}, exactly.

    Evaluated with a float64 matmul of the integer-valued operands: every partial sum is an
    integer of magnitude <= K * 127^2 < 2^53 for any K below 5.5e11, so each fp64 operation is
    exact whatever the summation order.  The result is checked to be integral and to fit int32.
    """
    xq = np.asarray(xq)
    wq = np.asarray(wq)
    K = xq.shape[1]
    assert K * QMAX * QMAX < 2**53
    acc = xq.astype(np.float64) @ wq.astype(np.float64).T
    acc_i = acc.astype(np.int64)
    assert np.array_equal(acc_i.astype(np.float64), acc)
    assert np.all(np.abs(acc_i) < 2**31)
    return acc_i


def dequantize(acc: np.ndarray, s_x: np.ndarray, s_w: np.ndarray, bias=None) -> np.ndarray:
    """Eq. gemm-final scale: y_{t,i} = (s_t^x * s_i^W) * acc_{t,i}, fp32, left to right,
    then + bias_i (fp32).  Returns fp32 [M, N]."""
    scale = (s_x.astype(np.float32)[:, None] * s_w.astype(np.float32)[None, :]).astype(np.float32)
    y = (scale * acc.astype(np.float32)).astype(np.float32)
    if bias is not None:
        y = (y + np.asarray(bias, dtype=np.float32)[None, :]).astype(np.float32)
    return y


def w8a8_linear(X: np.ndarray, prep: dict, bias=None, out: str = "bf16") -> dict:
    """One W8A8 SmoothQuant linear (LM Head section, Eq. xhat-lmhead .. gemm-final).

    X: fp32 values of the bf16 input [M, K].  out='bf16' rounds y to bf16 (a hidden-state
    linear); out='f32' keeps fp32 (the logits of lm_head).
    Returns dict(xq, s_x, acc, y) with every intermediate for element-wise comparison.
    """
    xq, s_x = quantize_activations(X, prep["inv_delta"])
    acc = int_gemm(xq, prep["wq"])
    y = dequantize(acc, s_x, prep["s_w"], bias)
    if out == "bf16":
        y = round_to_bf16(y)
    return {"xq": xq, "s_x": s_x, "acc": acc, "y": y}


def bf16_linear(X: np.ndarray, W: np.ndarray, bias=None, out: str = "bf16") -> np.ndarray:
    """The bf16 pass-through of an unselected layer (FFN section: layers outside Q_FFN keep the
    original precision): y = X W^T summed in fp64 (products of bf16 values are exact in fp64),
    rounded once to fp32, + bias, then rounded to bf16 unless out='f32'."""
    y = (np.asarray(X, np.float64) @ np.asarray(W, np.float64).T).astype(np.float32)
    if bias is not None:
        y = (y + np.asarray(bias, dtype=np.float32)[None, :]).astype(np.float32)
    return round_to_bf16(y) if out == "bf16" else y


def top1(logits: np.ndarray) -> np.ndarray:
    """Index of the largest logit per row; ties go to the lowest index."""
    return np.argmax(np.asarray(logits), axis=-1).astype(np.int32)
