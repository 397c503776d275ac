"""Oracle: the GeGLU activation of the FFN block (test infrastructure).

The FFN section describes the block as gate_proj, an activation, up_proj and down_proj; the
Gemma-3 FFN it studies gates with the tanh approximation of GELU (Hendrycks & Gimpel, 2016):

    gelu_tanh(g) = 0.5 * g * (1 + tanh(sqrt(2/pi) * (g + 0.044715 * g^3)))
                 = g / (1 + exp(-2 z)),   z = sqrt(2/pi) * (g + 0.044715 * g^3)

(the second line is the identity 0.5 * (1 + tanh z) = 1 / (1 + e^{-2z})).  h = gelu_tanh(g) * u.

Two evaluations are given:
  * ``gelu_tanh_f64``: the definition in fp64, the reference the fp32 recipe is pinned to.
  * ``gelu_tanh_f32``: a fixed fp32 recipe, every operation rounded to nearest-even and
    evaluated in the order written, with its own exponential: 2^w = 2^n * 2^f, n = rint(w),
    f = w - n in [-1/2, 1/2] (exact), and 2^f = e^{f ln 2} from the degree-7 Taylor series of
    the exponential (remainder < 1e-8 relative on that interval), evaluated by Horner's rule.
    Because the h it produces is quantised to INT8 for down_proj, the GPU implements the same
    recipe so that the INT8 codes of down_proj's input can be compared bit for bit.
    Its error against the fp64 definition is bounded in the tests.
"""
from __future__ import annotations

import math

import numpy as np

F32 = np.float32

C_SQRT_2_OVER_PI = F32(math.sqrt(2.0 / math.pi))     # 0.7978845608...
C_CUBIC = F32(0.044715)
C_NEG_2_LOG2E = F32(-2.0 / math.log(2.0))            # -2 * log2(e): e^{-2z} = 2^{w}, w = this * z
W_CLAMP = F32(126.0)                                  # keeps 2^n a normal fp32 number
# Taylor coefficients of 2^f = sum_k (ln 2)^k / k! * f^k, k = 0..7, each rounded to fp32.
EXP2_COEF = [F32(math.log(2.0) ** k / math.factorial(k)) for k in range(8)]


def gelu_tanh_f64(g: np.ndarray) -> np.ndarray:
    """The definition, evaluated in fp64 in its logistic form g / (1 + e^{-2z}), which has no
    cancellation in the negative tail (0.5 * (1 + tanh z) loses all digits there)."""
    g = np.asarray(g, dtype=np.float64)
    z = math.sqrt(2.0 / math.pi) * (g + 0.044715 * g ** 3)
    with np.errstate(over="ignore"):
        return g / (1.0 + np.exp(-2.0 * z))


def exp2_f32(w: np.ndarray) -> np.ndarray:
    """2^w for fp32 w in [-126, 126] by the recipe in the module docstring."""
    w = np.asarray(w, dtype=np.float32)
    n = np.rint(w).astype(np.float32)
    f = (w - n).astype(np.float32)                       # exact: |w| < 2^23
    p = np.full_like(f, EXP2_COEF[7])
    for k in range(6, -1, -1):
        p = (p * f).astype(np.float32)
        p = (p + EXP2_COEF[k]).astype(np.float32)
    scale = np.ldexp(np.ones_like(f), n.astype(np.int32)).astype(np.float32)  # exact power of two
    return (p * scale).astype(np.float32)


def gelu_tanh_f32(g: np.ndarray) -> np.ndarray:
    """The fp32 recipe: g2 = g*g; g3 = g2*g; t = g + C_CUBIC*g3; z = C_SQRT_2_OVER_PI*t;
    w = clamp(C_NEG_2_LOG2E*z, -126, 126); e = 2^w; gelu = g / (1 + e)."""
    g = np.asarray(g, dtype=np.float32)
    g2 = (g * g).astype(np.float32)
    g3 = (g2 * g).astype(np.float32)
    t = (g + (C_CUBIC * g3).astype(np.float32)).astype(np.float32)
    z = (C_SQRT_2_OVER_PI * t).astype(np.float32)
    w = np.clip((C_NEG_2_LOG2E * z).astype(np.float32), -W_CLAMP, W_CLAMP).astype(np.float32)
    e = exp2_f32(w)
    d = (F32(1.0) + e).astype(np.float32)
    return (g / d).astype(np.float32)


def geglu_f32(g: np.ndarray, u: np.ndarray) -> np.ndarray:
    """h = fl32(gelu_tanh_f32(g) * u)."""
    return (gelu_tanh_f32(g) * np.asarray(u, dtype=np.float32)).astype(np.float32)
