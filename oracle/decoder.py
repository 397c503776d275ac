"""Oracle: a Gemma-3-1B-shaped decoder under a precision mask (test infrastructure).

Parity unpinned: the paper prints no number a random-init decoder can reproduce.  The parts
are pinned by textbook identities in the tests (RMSNorm of a constant row, RoPE as a
rotation, softmax weights summing to one, a one-key attention returning its value).

Architecture (Problem Statement and Attention / LM Head sections; Gemma-3 layer order with
the pre/post "sandwich" norms the LM Head section mentions): 26 layers, hidden 1152,
4 query heads sharing 1 KV head of dim 256 (GQA), FFN 6912, vocab 262144 with the lm_head
tied to the embedding table, sliding-window attention of 1024 on local layers and full
attention on the global layers 0, 6, 12, 18.

Dataflow, with the points where values are rounded to bf16 (the GPU rounds at the same
points; everything else is fp64 here and fp32 on the GPU):
    r = embed[token] * sqrt(hidden)                                      (residual stream)
    per layer l:
      a   = bf16(rmsnorm(r) * w_in)
      qkv = Linear_ATT[l](a)                                              -> bf16
      q_h = rope(rmsnorm(q_h) * w_qn), k = rope(rmsnorm(k) * w_kn)        (qk-norm, RoPE)
      K/V cache <- bf16(k), v
      o   = bf16(softmax((q_h . K) / sqrt(256)) V) over the allowed keys
      r   = r + rmsnorm(Linear_ATT[l](o)) * w_post_attn
      a2  = bf16(rmsnorm(r) * w_pre_ffn)
      r   = r + rmsnorm(FFN_FFN[l](a2)) * w_post_ffn
    logits = lm_head_LM(bf16(rmsnorm(r) * w_final))                      (fp32), top-1
Linear_S[l] is the W8A8 linear when layer l is in the set S of the mask, else bf16.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

from . import blocks as _b
from . import w8a8 as _w


@dataclass
class DecoderConfig:
    hidden: int = 1152
    inter: int = 6912
    layers: int = 26
    n_q: int = 4
    n_kv: int = 1
    head_dim: int = 256
    vocab: int = 262144
    eps: float = 1e-6
    rope_local: float = 10000.0
    rope_global: float = 1000000.0
    window: int = 1024
    global_layers: tuple = (0, 6, 12, 18)
    qk_norm: bool = True
    alpha: float = 0.5

    @property
    def q_dim(self):
        return self.n_q * self.head_dim

    @property
    def kv_dim(self):
        return self.n_kv * self.head_dim

    @property
    def qkv_dim(self):
        return self.q_dim + 2 * self.kv_dim

    @property
    def attn_scale(self):
        return 1.0 / math.sqrt(self.head_dim)

    @property
    def embed_scale(self):
        return float(np.float32(math.sqrt(self.hidden)))


def rmsnorm(x, w, eps):
    x = np.asarray(x, np.float64)
    inv = 1.0 / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps)
    return x * inv * np.asarray(w, np.float64)


def rope(x, pos, base, head_dim):
    """Rotate-half RoPE: pairs (i, i + d/2) rotated by pos * base^(-2i/d)."""
    half = head_dim // 2
    inv_freq = base ** (-(2.0 * np.arange(half)) / head_dim)
    ang = np.asarray(pos, np.float64)[:, None] * inv_freq[None, :]
    c, s = np.cos(ang), np.sin(ang)
    x = np.asarray(x, np.float64)
    x1, x2 = x[..., :half], x[..., half:]
    if x.ndim == 3:  # [T, heads, d]
        c, s = c[:, None, :], s[:, None, :]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


class OracleDecoder:
    """Holds fp64 copies of the bf16 weights, the prepared W8A8 weights and a KV cache."""

    def __init__(self, cfg: DecoderConfig, weights: dict, batch: int, max_len: int):
        self.cfg = cfg
        self.w = weights
        self.B = batch
        self.max_len = max_len
        self.prep = None
        self.stats = None
        self.reset()

    def reset(self):
        c = self.cfg
        self.kc = np.zeros((c.layers, self.B, self.max_len, c.kv_dim), np.float64)
        self.vc = np.zeros((c.layers, self.B, self.max_len, c.kv_dim), np.float64)

    # ------------------------------------------------------------------ calibration / prep
    def calibrate(self, token_batches):
        """Run the bf16 model over calibration sequences and record max_t |x_tj| at each
        linear's input (the forward-hook statistic of the LM Head section)."""
        c = self.cfg
        stats = {"qkv": [np.zeros(c.hidden, np.float32) for _ in range(c.layers)],
                 "o": [np.zeros(c.q_dim, np.float32) for _ in range(c.layers)],
                 "gu": [np.zeros(c.hidden, np.float32) for _ in range(c.layers)],
                 "down": [np.zeros(c.inter, np.float32) for _ in range(c.layers)],
                 "lm": np.zeros(c.hidden, np.float32)}
        for toks in token_batches:
            toks = np.asarray(toks).reshape(self.B, -1)
            self.reset()
            self.forward(toks, 0, mask=None, stats=stats, want_logits=False)
        self.stats = stats
        self.reset()
        return stats

    def prepare(self, stats=None, smooth=True):
        c = self.cfg
        st = stats if stats is not None else self.stats
        a = c.alpha
        self.prep = {
            "qkv": [_w.prepare_weights(self.w["wqkv"][l], st["qkv"][l], a, smooth) for l in range(c.layers)],
            "o": [_w.prepare_weights(self.w["wo"][l], st["o"][l], a, smooth) for l in range(c.layers)],
            "ffn": [_b.prepare_ffn(self.w["wg"][l], self.w["wu"][l], self.w["wd"][l],
                                   st["gu"][l], st["down"][l], a, smooth) for l in range(c.layers)],
            "lm": _w.prepare_weights(self.w["embed"], st["lm"], a, smooth),
        }

    # ---------------------------------------------------------------------------- forward
    def _linear(self, x, name, l, int8, stats):
        if stats is not None:
            key = {"wqkv": "qkv", "wo": "o"}[name]
            stats[key][l] = np.maximum(stats[key][l], _w.act_absmax(x))
        if int8:
            key = {"wqkv": "qkv", "wo": "o"}[name]
            return _w.w8a8_linear(x, self.prep[key][l], out="bf16")["y"]
        return _w.bf16_linear(x, self.w[name][l], out="bf16")

    def _ffn(self, x, l, int8, stats):
        if stats is not None:
            stats["gu"][l] = np.maximum(stats["gu"][l], _w.act_absmax(x))
        if int8:
            return _b.ffn_w8a8(x, self.prep["ffn"][l])["y"]
        r = _b.ffn_bf16(x, self.w["wg"][l], self.w["wu"][l], self.w["wd"][l])
        if stats is not None:
            stats["down"][l] = np.maximum(stats["down"][l], _w.act_absmax(r["h"]))
        return r["y"]

    def _attention(self, l, q, pos0, T):
        """q: [B, T, n_q, d] (fp64).  Keys/values from the cache positions allowed for each
        query position p: all j <= p on global layers, p - window < j <= p on local ones."""
        c = self.cfg
        glob = l in c.global_layers
        out = np.zeros((self.B, T, c.n_q, c.head_dim), np.float64)
        group = c.n_q // c.n_kv
        for b in range(self.B):
            for t in range(T):
                p = pos0 + t
                lo = 0 if glob else max(0, p - c.window + 1)
                for h in range(c.n_q):
                    kvh = h // group
                    K = self.kc[l, b, lo:p + 1, kvh * c.head_dim:(kvh + 1) * c.head_dim]
                    V = self.vc[l, b, lo:p + 1, kvh * c.head_dim:(kvh + 1) * c.head_dim]
                    s = (K @ q[b, t, h]) * c.attn_scale
                    s = np.exp(s - np.max(s))
                    pr = s / np.sum(s)
                    out[b, t, h] = pr @ V
        return out

    def forward(self, tokens, pos0, mask=None, stats=None, want_logits=True, want_layers=False):
        """tokens [B, T] at positions pos0 .. pos0+T-1; mask an oracle.masks.Mask or None
        (all bf16).  Returns dict(logits fp32 [B, T, V], top1 [B, T], final bf16 hidden, and with
        want_layers every layer's output: the residual stream after its post-FFN step, [L][M, H])."""
        c, w = self.cfg, self.w
        toks = np.asarray(tokens).reshape(self.B, -1)
        T = toks.shape[1]
        M = self.B * T
        ffn_set = mask.ffn if mask is not None else frozenset()
        att_set = mask.att if mask is not None else frozenset()
        lm8 = bool(mask.lm) if mask is not None else False
        es = np.float32(c.embed_scale)
        r = (w["embed"][toks.reshape(-1)].astype(np.float32) * es).astype(np.float64)
        pos = np.arange(pos0, pos0 + T)
        layers = []
        for l in range(c.layers):
            base = c.rope_global if l in c.global_layers else c.rope_local
            a = _w.round_to_bf16(rmsnorm(r, w["ln_in"][l], c.eps).astype(np.float32))
            qkv = self._linear(a, "wqkv", l, l in att_set, stats).astype(np.float64)
            q = qkv[:, :c.q_dim].reshape(self.B, T, c.n_q, c.head_dim)
            k = qkv[:, c.q_dim:c.q_dim + c.kv_dim].reshape(self.B, T, c.n_kv, c.head_dim)
            v = qkv[:, c.q_dim + c.kv_dim:].reshape(self.B, T, c.kv_dim)
            if c.qk_norm:
                q = rmsnorm(q, w["q_norm"][l], c.eps)
                k = rmsnorm(k, w["k_norm"][l], c.eps)
            for b in range(self.B):
                q[b] = rope(q[b], pos, base, c.head_dim)
                k[b] = rope(k[b], pos, base, c.head_dim)
            kb = _w.round_to_bf16(k.reshape(self.B, T, c.kv_dim).astype(np.float32))
            self.kc[l, :, pos0:pos0 + T] = kb
            self.vc[l, :, pos0:pos0 + T] = v
            o = self._attention(l, q, pos0, T).reshape(M, c.q_dim)
            o = _w.round_to_bf16(o.astype(np.float32))
            y = self._linear(o, "wo", l, l in att_set, stats).astype(np.float64)
            r = r + rmsnorm(y, w["ln_post_attn"][l], c.eps)
            a2 = _w.round_to_bf16(rmsnorm(r, w["ln_pre_ffn"][l], c.eps).astype(np.float32))
            f = self._ffn(a2, l, l in ffn_set, stats).astype(np.float64)
            r = r + rmsnorm(f, w["ln_post_ffn"][l], c.eps)
            if want_layers:
                layers.append(r.copy())
        fin = _w.round_to_bf16(rmsnorm(r, w["final_norm"], c.eps).astype(np.float32))
        if stats is not None:
            stats["lm"] = np.maximum(stats["lm"], _w.act_absmax(fin))
        if not want_logits:
            return {"final": fin, "layers": layers}
        if lm8:
            head = _b.lm_head_w8a8(fin, self.prep["lm"])
        else:
            head = _b.lm_head_bf16(fin, w["embed"])
        return {"logits": head["logits"].reshape(self.B, T, -1),
                "top1": head["top1"].reshape(self.B, T), "final": fin, "layers": layers}

    def sqnr_profile(self, tokens, mask, isolated: bool):
        """SQNR of every layer's output (Eq. sqnr-block) and of the logits (Eq. sqnr-ffn) under
        mask against the all-bf16 model, over a prefill from position 0 (Combined Configurations):
        propagated, one pass under the whole mask; isolated, a pass per layer with only that
        layer's sublayers of the mask quantised (it then takes the reference input; +inf where the
        mask quantises nothing in the layer), and the lm_head alone likewise."""
        from . import masks as _m
        from . import quality as _q
        L = self.cfg.layers
        self.reset()
        ref = self.forward(tokens, 0, None, want_layers=True)
        if not isolated:
            self.reset()
            q = self.forward(tokens, 0, mask, want_layers=True)
            self.reset()
            return ([_q.sqnr_block_db(ref["layers"][l], q["layers"][l]) for l in range(L)],
                    _q.sqnr_db(ref["logits"].astype(np.float64), q["logits"].astype(np.float64)))
        out = []
        for l in range(L):
            f = frozenset({l}) & mask.ffn
            a = frozenset({l}) & mask.att
            if not f and not a:
                out.append(float("inf"))
                continue
            self.reset()
            q = self.forward(tokens, 0, _m.Mask(f, a, False), want_layers=True, want_logits=False)
            out.append(_q.sqnr_block_db(ref["layers"][l], q["layers"][l]))
        lm = float("inf")
        if mask.lm:
            self.reset()
            q = self.forward(tokens, 0, _m.Mask(frozenset(), frozenset(), True))
            lm = _q.sqnr_db(ref["logits"].astype(np.float64), q["logits"].astype(np.float64))
        self.reset()
        return out, lm
