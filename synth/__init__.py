"""Seeded synthetic inputs shared by the tests, the bench and the oracle's callers.

This module draws random numbers and rounds them to the storage type; it holds none of the
W8A8 method's arithmetic (no smoothing, quantisation, GEMM or dequantisation), so both the
CUDA path and the oracle can take their inputs from it without sharing method code.

Generator: numpy PCG64 via ``np.random.default_rng([seed, *stream_keys])``; fp32 draws are
rounded to bf16 (round-to-nearest-even) with torch's conversion.  Every function returns
``(fp32 numpy array holding bf16 values, torch.bfloat16 CPU tensor)`` pairs or plain arrays.

Shapes and distributions follow the workloads the paper measures (Gemma-3-1B, batch 1
decode and short prefills), with synthetic data standing in for its trained weights,
prompt and held-out text, which are not available:
  * activations N(0, 1) with a few outlier input channels scaled x20 (SmoothQuant's regime);
  * weights N(0, 0.02) (random init);
  * lm_head inputs N(0, 1) rows normalised to unit RMS (the output of the final RMSNorm);
  * token ids uniform in [0, vocab).
"""
from __future__ import annotations

import numpy as np
import torch

HIDDEN, INTER, VOCAB = 1152, 6912, 262144


def rng(seed: int, *keys: int) -> np.random.Generator:
    return np.random.default_rng([int(seed), *[int(k) for k in keys]])


def to_bf16(x: np.ndarray):
    """Round fp32 draws to bf16.  Returns (fp32 array of the bf16 values, bf16 torch tensor)."""
    t = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).to(torch.bfloat16)
    return t.float().numpy(), t


def normal(shape, std: float, g: np.random.Generator) -> np.ndarray:
    return (g.standard_normal(size=shape, dtype=np.float32) * np.float32(std)).astype(np.float32)


def outlier_channels(K: int, n: int, g: np.random.Generator) -> np.ndarray:
    return np.sort(g.choice(K, size=n, replace=False))


def activations(M: int, K: int, n_outliers: int, seed: int, stream: int = 0,
                channels: np.ndarray | None = None, scale: float = 20.0):
    """X [M, K] ~ N(0, 1) with `n_outliers` channels (drawn without replacement unless given)
    multiplied by `scale`.  Returns (x32, x_bf16, channels)."""
    g = rng(seed, 1, stream)
    if channels is None:
        channels = outlier_channels(K, n_outliers, rng(seed, 2))
    x = g.standard_normal(size=(M, K), dtype=np.float32)
    x[:, channels] *= np.float32(scale)
    x32, xt = to_bf16(x)
    return x32, xt, channels


def weight(N: int, K: int, seed: int, stream: int = 0, std: float = 0.02):
    """W [N, K] (row = output channel) ~ N(0, std)."""
    return to_bf16(normal((N, K), std, rng(seed, 3, stream)))


def normed_rows(M: int, K: int, seed: int, stream: int = 0):
    """Rows of N(0, 1) divided by their RMS (the statistics of a final-RMSNorm output)."""
    x = rng(seed, 4, stream).standard_normal(size=(M, K)).astype(np.float64)
    if M:
        x = x / np.sqrt(np.mean(x * x, axis=1, keepdims=True))
    return to_bf16(x.astype(np.float32))


def positive_stat(K: int, lo: float, hi: float, seed: int, stream: int = 0) -> np.ndarray:
    """A synthetic per-channel calibration statistic (max |x_j|), uniform in [lo, hi], rounded
    to bf16 values (absmax of bf16 data is itself a bf16 value)."""
    return to_bf16(rng(seed, 5, stream).uniform(lo, hi, size=K).astype(np.float32))[0]


def tokens(n: int, vocab: int, seed: int, stream: int = 0) -> np.ndarray:
    return rng(seed, 6, stream).integers(0, vocab, size=n, dtype=np.int64).astype(np.int32)


# ----------------------------------------------------------------------- workload recipes
def linear_case(M: int = 16, K: int = HIDDEN, N: int = INTER, n_outliers: int = 8, seed: int = 0):
    """Single W8A8 linear, Gemma-3-1B gate_proj shape: X [M, K] N(0,1) with 8 outlier channels
    x20, W [N, K] N(0, 0.02); the calibration set is X itself."""
    x32, xt, ch = activations(M, K, n_outliers, seed)
    w32, wt = weight(N, K, seed)
    return {"x32": x32, "x": xt, "w32": w32, "w": wt, "calib32": x32, "calib": xt, "channels": ch}


def ffn_case(M: int, seed: int = 0, hidden: int = HIDDEN, inter: int = INTER, calib_rows: int = 512):
    """One FFN block: X [M, hidden] N(0,1) with 1% outlier channels x20; gate/up [inter, hidden]
    and down [hidden, inter] N(0, 0.02); calibration X (512 rows, same outlier channels);
    a synthetic statistic for down_proj's input h."""
    n_out = max(1, round(0.01 * hidden))
    x32, xt, ch = activations(M, hidden, n_out, seed)
    c32, ct, _ = activations(calib_rows, hidden, n_out, seed, stream=1, channels=ch)
    wg32, wg = weight(inter, hidden, seed, 10)
    wu32, wu = weight(inter, hidden, seed, 11)
    wd32, wd = weight(hidden, inter, seed, 12)
    stat_h = positive_stat(inter, 0.5, 8.0, seed, 13)
    return {"x32": x32, "x": xt, "calib32": c32, "calib": ct, "wg32": wg32, "wg": wg,
            "wu32": wu32, "wu": wu, "wd32": wd32, "wd": wd, "stat_h": stat_h, "channels": ch}


def lm_head_case(M: int, seed: int = 0, hidden: int = HIDDEN, vocab: int = VOCAB, calib_rows: int = 640):
    """lm_head: X [M, hidden] = unit-RMS rows; W [vocab, hidden] N(0, 0.02); calibration rows
    drawn the same way (a separate stream)."""
    x32, xt = normed_rows(M, hidden, seed)
    c32, ct = normed_rows(calib_rows, hidden, seed, stream=1)
    w32, wt = weight(vocab, hidden, seed, 20)
    return {"x32": x32, "x": xt, "calib32": c32, "calib": ct, "w32": w32, "w": wt}


def decoder_weights(layers: int = 26, hidden: int = HIDDEN, inter: int = INTER, vocab: int = VOCAB,
                    n_q: int = 4, n_kv: int = 1, head_dim: int = 256, seed: int = 0, std: float = 0.02,
                    want_f32: bool = True):
    """Random-init weights of the decoder: every matrix N(0, std), every norm multiplier 1.
    Returns (f32: dict of fp32 arrays or None, bf16: dict of torch bf16 tensors, norms: dict of
    fp32 arrays).  Per-layer matrices are lists indexed by layer."""
    qkv = (n_q + 2 * n_kv) * head_dim
    f32, bf = {}, {}
    names = [("wqkv", (qkv, hidden)), ("wo", (hidden, n_q * head_dim)), ("wg", (inter, hidden)),
             ("wu", (inter, hidden)), ("wd", (hidden, inter))]
    for s, (name, shape) in enumerate(names):
        f32[name], bf[name] = [], []
        for l in range(layers):
            a, t = to_bf16(normal(shape, std, rng(seed, 7, s, l)))
            f32[name].append(a if want_f32 else None)
            bf[name].append(t)
    a, t = to_bf16(normal((vocab, hidden), std, rng(seed, 8)))
    f32["embed"], bf["embed"] = (a if want_f32 else None), t
    norms = {}
    for name, n in [("ln_in", hidden), ("ln_post_attn", hidden), ("ln_pre_ffn", hidden),
                    ("ln_post_ffn", hidden), ("q_norm", head_dim), ("k_norm", head_dim)]:
        norms[name] = [np.ones(n, np.float32) for _ in range(layers)]
    norms["final_norm"] = np.ones(hidden, np.float32)
    return (f32 if want_f32 else None), bf, norms
