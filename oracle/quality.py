"""Oracle: the quality measures used as the allocation's constraint (test infrastructure).

  * Top-1 agreement (LM Head section): the fraction of positions at which the quantised and
    the reference model choose the same next token (argmax of the logits).
  * Perplexity and its relative change (LM Head section): PPL = exp(mean negative
    log-likelihood of the next token); delta = PPL_q / PPL_ref - 1.
  * SQNR in dB of a layer output (Eq. sqnr-ffn) and of a decoder block output (Eq. sqnr-block).
  * Speedup and latency reduction (Combined Configurations table): speedup = tok/s ratio;
    the per-token latency reduction is 1 - 1/speedup.
"""
from __future__ import annotations

import numpy as np


def top1_agreement(top_q: np.ndarray, top_ref: np.ndarray) -> float:
    top_q = np.asarray(top_q).ravel()
    top_ref = np.asarray(top_ref).ravel()
    assert top_q.shape == top_ref.shape and top_q.size > 0
    return float(np.mean(top_q == top_ref))


def nll(logits: np.ndarray, targets: np.ndarray) -> np.ndarray:
    """Per-position negative log-likelihood of targets under softmax(logits), in fp64
    (log-sum-exp with the row maximum subtracted)."""
    z = np.asarray(logits, dtype=np.float64)
    m = np.max(z, axis=-1, keepdims=True)
    lse = m[..., 0] + np.log(np.sum(np.exp(z - m), axis=-1))
    picked = np.take_along_axis(z, np.asarray(targets)[..., None].astype(np.int64), axis=-1)[..., 0]
    return lse - picked


def perplexity(logits: np.ndarray, targets: np.ndarray) -> float:
    return float(np.exp(np.mean(nll(logits, targets))))


def ppl_from_nll(nll_values: np.ndarray) -> float:
    return float(np.exp(np.mean(np.asarray(nll_values, dtype=np.float64))))


def ppl_delta(ppl_q: float, ppl_ref: float) -> float:
    return ppl_q / ppl_ref - 1.0


def sqnr_db(y_clean: np.ndarray, y_dirty: np.ndarray) -> float:
    """Eq. sqnr-ffn: 10 log10(||y_clean||^2 / ||y_clean - y_dirty||^2); +inf when the two are
    equal (the noiseless limit)."""
    c = np.asarray(y_clean, np.float64)
    d = c - np.asarray(y_dirty, np.float64)
    e = np.sum(d * d)
    return float("inf") if e == 0 else float(10.0 * np.log10(np.sum(c * c) / e))


def sqnr_block_db(h_ref: np.ndarray, h_q: np.ndarray) -> float:
    """Eq. sqnr-block: 10 log10(E[h_ref^2] / E[(h_ref - h_q)^2]); +inf when the two are equal."""
    r = np.asarray(h_ref, np.float64)
    d = r - np.asarray(h_q, np.float64)
    e = np.mean(d * d)
    return float("inf") if e == 0 else float(10.0 * np.log10(np.mean(r * r) / e))


def speedup(toks_per_s: float, toks_per_s_base: float) -> float:
    return toks_per_s / toks_per_s_base


def latency_reduction(speedup_value: float) -> float:
    return 1.0 - 1.0 / speedup_value
