"""Oracle: the FFN block and lm_head built from the W8A8 linear (test infrastructure).

FFN block (FFN section): gate_proj and up_proj share their input, so the oracle quantises the
fused weight [gate; up] (2F rows) with one smoothing factor per input channel, computed over
all 2F rows; g and u leave the dequantising epilogue in fp32, h = gelu_tanh(g) * u is rounded
to bf16 (the activation between two linears), and down_proj is a second W8A8 linear on h.
Layers outside Q_FFN run the same block with bf16 linears (FFN section, "remain at the
original precision").

lm_head (LM Head section): logits = W8A8 linear of the final-norm hidden state with the tied
[V, d] table, kept in fp32, and the top-1 index (ties to the lowest index).

FP8 block (Future Work: e4m3 in place of INT8; the reading of oracle/fp8.py): the same block with
both linears in the e4m3 variant, g and u in fp32 out of its epilogue, h rounded to bf16.  Parity
against the paper unpinned (it prints no FP8 numbers).
"""
from __future__ import annotations

import numpy as np

from . import fp8 as _fp8
from . import geglu as _geglu
from . import w8a8 as _w


def prepare_ffn(w_gate, w_up, w_down, stat_in, stat_h, alpha: float = 0.5, smooth: bool = True):
    """Prepare the fused gate/up weight [2F, H] = [gate; up] against the calibration statistic
    of the block input, and down [H, F] against the statistic of h."""
    gu = np.concatenate([np.asarray(w_gate, np.float32), np.asarray(w_up, np.float32)], axis=0)
    return {
        "F": int(np.asarray(w_gate).shape[0]),
        "gu": _w.prepare_weights(gu, stat_in, alpha, smooth),
        "down": _w.prepare_weights(w_down, stat_h, alpha, smooth),
    }


def ffn_w8a8(X, prep) -> dict:
    """W8A8 FFN block.  Returns every stage: gate/up (xq, s_x, acc), g, u, h (bf16 values),
    down (xq, s_x, acc) and y (bf16 values)."""
    F = prep["F"]
    gu = _w.w8a8_linear(X, prep["gu"], out="f32")
    g, u = gu["y"][:, :F], gu["y"][:, F:]
    h = _w.round_to_bf16(_geglu.geglu_f32(g, u))
    dn = _w.w8a8_linear(h, prep["down"], out="bf16")
    return {"gu": gu, "g": g, "u": u, "h": h, "down": dn, "y": dn["y"]}


def ffn_bf16(X, w_gate, w_up, w_down) -> dict:
    """bf16 pass-through FFN block: g, u = X W^T (fp64 sums rounded to fp32), h = bf16(geglu),
    y = bf16(h W_down^T)."""
    g = _w.bf16_linear(X, w_gate, out="f32")
    u = _w.bf16_linear(X, w_up, out="f32")
    h = _w.round_to_bf16(_geglu.geglu_f32(g, u))
    y = _w.bf16_linear(h, w_down, out="bf16")
    return {"g": g, "u": u, "h": h, "y": y}


def lm_head_w8a8(X, prep) -> dict:
    """W8A8 lm_head: fp32 logits and top-1 (LM Head section, Eq. gemm-final)."""
    r = _w.w8a8_linear(X, prep, out="f32")
    r["logits"] = r["y"]
    r["top1"] = _w.top1(r["y"])
    return r


def lm_head_bf16(X, W) -> dict:
    """bf16 pass-through lm_head: fp32 logits (fp64 sums rounded once) and top-1."""
    logits = _w.bf16_linear(X, W, out="f32")
    return {"logits": logits, "top1": _w.top1(logits)}


def prepare_ffn_fp8(w_gate, w_up, w_down, stat_in, stat_h, alpha: float = 0.5, smooth: bool = True):
    """prepare_ffn with the e4m3 rule: one delta over the fused [gate; up] rows, then e4m3 codes."""
    gu = np.concatenate([np.asarray(w_gate, np.float32), np.asarray(w_up, np.float32)], axis=0)
    return {
        "F": int(np.asarray(w_gate).shape[0]),
        "gu": _fp8.prepare_weights_fp8(gu, stat_in, alpha, smooth),
        "down": _fp8.prepare_weights_fp8(w_down, stat_h, alpha, smooth),
    }


def ffn_fp8(X, prep) -> dict:
    """FP8 FFN block: g, u (fp32) from the e4m3 gate/up linear, h = bf16(geglu(g, u)), y from the
    e4m3 down linear (bf16)."""
    F = prep["F"]
    gu = _fp8.fp8_linear(X, prep["gu"], out="f32")
    g, u = gu["y"][:, :F], gu["y"][:, F:]
    h = _w.round_to_bf16(_geglu.geglu_f32(g, u))
    dn = _fp8.fp8_linear(h, prep["down"], out="bf16")
    return {"gu": gu, "g": g, "u": u, "h": h, "down": dn, "y": dn["y"]}
