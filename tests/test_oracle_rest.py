"""Pins for the rest of the oracle: GeGLU (closed forms, the fp64 definition, a library
routine), the masks (the paper's equations and tables), the quality measures (the paper's
printed ratios, closed forms), the allocation rule (the paper's combined table) and the
decoder's parts (textbook identities, prefill/decode consistency)."""
import json
import math
import os

import numpy as np
import pytest
import torch

from oracle import allocator, blocks, decoder, geglu, masks, quality
from oracle import w8a8 as W

F32 = np.float32


# ---------------------------------------------------------------------------------- GeGLU
def test_gelu_definition_matches_library_tanh_gelu():
    g = np.linspace(-12, 12, 4001)
    ref = torch.nn.functional.gelu(torch.from_numpy(g), approximate="tanh").numpy()
    # torch evaluates 0.5 g (1 + tanh z), which cancels to ~1e-16 |g| absolute in the tail
    assert np.allclose(geglu.gelu_tanh_f64(g), ref, rtol=1e-13, atol=4e-16 * 12)
    pos = g > -1
    assert np.allclose(geglu.gelu_tanh_f64(g[pos]), ref[pos], rtol=1e-13, atol=1e-300)


def test_logistic_identity_used_by_recipe():
    mpmath = pytest.importorskip("mpmath")
    mpmath.mp.dps = 60
    for z in np.linspace(-40, 40, 321):
        zz = mpmath.mpf(float(z))
        lhs = (1 + mpmath.tanh(zz)) / 2
        rhs = 1 / (1 + mpmath.exp(-2 * zz))
        assert abs(lhs / rhs - 1) < mpmath.mpf(10) ** -20  # 60 digits minus the tail cancellation


def test_exp2_recipe_relative_error():
    w = np.concatenate([np.linspace(-126, 126, 200001), np.arange(-126, 127)]).astype(F32)
    ours = geglu.exp2_f32(w).astype(np.float64)
    ref = np.exp2(w.astype(np.float64))
    assert np.max(np.abs(ours / ref - 1)) < 4 * 2 ** -24
    assert np.all(geglu.exp2_f32(np.arange(-20, 21).astype(F32)) == np.exp2(np.arange(-20, 21)).astype(F32))


def test_gelu_recipe_against_fp64_definition():
    g = np.concatenate([np.linspace(-9, 12, 300001), np.array([1e-6, -1e-6, 1e-20, 0.5, -0.5])]).astype(F32)
    ours = geglu.gelu_tanh_f32(g).astype(np.float64)
    ref = geglu.gelu_tanh_f64(g.astype(np.float64))
    # fp32 rounding of the exponent w = -2 log2(e) z is amplified by 2^w into a relative error
    # of about |w| * 2^-24 * ln 2; elsewhere the recipe is within a few ulps.
    w = np.abs(2.0 / math.log(2.0) * math.sqrt(2 / math.pi) * (g.astype(np.float64) + 0.044715 * g.astype(np.float64) ** 3))
    big = np.abs(ref) > 1e-36
    rel = np.abs(ours[big] / ref[big] - 1)
    assert np.all(rel <= 4.8e-7 + np.minimum(w[big], 126) * 2 ** -21)
    assert np.max(np.abs(ours - ref)) < 1e-6


def test_gelu_closed_forms():
    assert geglu.gelu_tanh_f32(np.array([0.0], F32))[0] == 0
    big = np.array([10.0, 20.0, 1e4], F32)
    assert np.array_equal(geglu.gelu_tanh_f32(big), big)
    gneg = np.array([-10.0, -20.0, -1e4], F32)
    neg = geglu.gelu_tanh_f32(gneg)
    # the clamp of the exponent at 126 bounds the tail by |g| * 2^-126 (true value ~ |g| e^{-2|z|})
    assert np.all(neg <= 0) and np.all(np.abs(neg) <= np.abs(gneg) * 2.0 ** -125)
    h = geglu.geglu_f32(np.array([1.0, -1.0], F32), np.array([2.0, 2.0], F32))
    assert np.allclose(h, 2 * geglu.gelu_tanh_f64(np.array([1.0, -1.0])), rtol=1e-6)


# ----------------------------------------------------------------------------------- masks
def test_masks_equal_paper_sets(golden_dir):
    assert masks.GROUPS["5+5"] == {0, 1, 2, 3, 4, 21, 22, 23, 24, 25}
    assert masks.GROUPS["10+10"] == {0, 1, 2, 3, 4, 5, 6, 7, 8, 9, 16, 17, 18, 19, 20, 21, 22, 23, 24, 25}
    assert masks.GROUPS["all26"] == set(range(26))
    gold = json.load(open(os.path.join(golden_dir, "table1_weight_mb.json")))
    for k, v in gold["ffn_bench_int8_layers"].items():
        if not k.startswith("_"):
            assert len(masks.GROUPS[k]) == v
    assert len(masks.PAPER_CONFIGS) == 14
    m = masks.PAPER_CONFIGS["attn_ffn 10+10 + lm_head"]
    assert m.ffn == masks.GROUPS["10+10"] and m.att == masks.L and m.lm
    ffn_bits, att_bits, lm = masks.PAPER_CONFIGS["FFN 5+5 + lm_head"].bits()
    assert ffn_bits == 0b11111_0000000000000000_11111 and att_bits == 0 and lm == 1
    cands = masks.candidate_masks()
    assert len(cands) == 16 and set(masks.PAPER_CONFIGS.values()) <= set(cands.values())


def test_weight_sizes_match_table1(golden_dir):
    gold = json.load(open(os.path.join(golden_dir, "table1_weight_mb.json")))["weights_mb"]
    for name, mb in gold.items():
        # printed to 2 decimals (3.375 appears as 3.37, 30.375 as 30.38): within half a unit
        assert abs(masks.weight_mib(name) - mb) <= 0.005 + 1e-12, name


# --------------------------------------------------------------------------------- quality
def test_quality_definitions_reproduce_paper_numbers(golden_dir):
    gold = json.load(open(os.path.join(golden_dir, "lm_head_quality.json")))
    n, agree = gold["positions"], gold["agree"]
    top_ref = np.arange(n)
    top_q = top_ref.copy()
    top_q[: n - agree] += 1
    assert round(100 * quality.top1_agreement(top_q, top_ref), 2) == gold["agree_pct_printed"]
    assert round(100 * quality.ppl_delta(gold["ppl_q"], gold["ppl_ref"]), 2) == gold["ppl_delta_pct_printed"]
    for name, (sp, pct) in gold["speedups"].items():
        assert round(100 * (sp - 1), 1) == pct
    assert round(100 * quality.latency_reduction(1.110), 1) == 9.9
    assert round(100 * quality.latency_reduction(1.191), 1) == 16.0


def test_perplexity_closed_forms():
    V = 1000
    z = np.zeros((7, V))
    assert quality.perplexity(z, np.arange(7)) == pytest.approx(V, rel=1e-12)
    z[np.arange(7), np.arange(7)] = 1e4
    assert quality.perplexity(z, np.arange(7)) == pytest.approx(1.0, abs=1e-12)
    # two-way logits: NLL = log(1 + e^-d)
    z2 = np.array([[0.0, 2.0]])
    assert quality.nll(z2, np.array([1]))[0] == pytest.approx(math.log1p(math.exp(-2.0)), rel=1e-12)


def test_sqnr_closed_form():
    g = np.random.default_rng(0).standard_normal(1000)
    assert quality.sqnr_db(g, g * (1 + 1e-3)) == pytest.approx(60.0, abs=1e-9)
    assert quality.sqnr_block_db(g, g * (1 - 1e-2)) == pytest.approx(40.0, abs=1e-9)


# ------------------------------------------------------------------------------- allocator
def _paper_candidates(golden_dir):
    gold = json.load(open(os.path.join(golden_dir, "paper_combined_table.json")))
    rows = gold["rows"]
    cands = []
    for r in rows:
        ok = r["quality"] in ("reference", "good", "excellent")
        m = masks.PAPER_CONFIGS[r["name"]]
        cands.append({"name": r["name"], "latency": 1.0 / r["speedup"], "top1": 1.0 if ok else 0.5,
                      "ppl_delta": 0.0 if ok else 1.0, "n_int8": m.n_int8_sublayers()})
    return gold, cands


def test_allocator_reproduces_paper_choice(golden_dir):
    gold, cands = _paper_candidates(golden_dir)
    assert cands[allocator.choose(cands)]["name"] == gold["chosen_quality_preserved"]
    assert cands[allocator.choose(cands, min_top1=0.0, max_ppl_delta=math.inf)]["name"] == gold["fastest_any_quality"]
    # by tok/s instead of the printed speedup column the choice is the same
    rows = gold["rows"]
    for c, r in zip(cands, rows):
        c["latency"] = 1.0 / r["tok_s"]
    assert cands[allocator.choose(cands)]["name"] == gold["chosen_quality_preserved"]


def test_allocator_tie_break_and_infeasible():
    c = [{"latency": 1.0, "top1": 1.0, "ppl_delta": 0.0, "n_int8": 0},
         {"latency": 0.8, "top1": 0.99, "ppl_delta": 0.0, "n_int8": 11},
         {"latency": 0.8, "top1": 0.995, "ppl_delta": 0.001, "n_int8": 10},
         {"latency": 0.5, "top1": 0.90, "ppl_delta": 0.0, "n_int8": 1}]
    assert allocator.choose(c) == 2
    assert allocator.choose(c, min_top1=0.999) == 0
    assert allocator.choose([{"latency": 1, "top1": 0.1, "ppl_delta": 0, "n_int8": 0}]) is None


# --------------------------------------------------------------------------------- decoder
def test_rmsnorm_constant_row_and_rope_rotation():
    x = np.full((1, 64), 3.0)
    assert np.allclose(decoder.rmsnorm(x, np.ones(64), 0.0), 1.0)
    g = np.random.default_rng(1)
    v = g.standard_normal((5, 2, 16))
    pos = np.array([0, 1, 7, 100, 2047])
    r = decoder.rope(v, pos, 10000.0, 16)
    assert np.allclose(r[0], v[0])
    pair = lambda a: a[..., :8] ** 2 + a[..., 8:] ** 2
    assert np.allclose(pair(r), pair(v))
    # rotation composition: rope(rope(x, a), b) == rope(x, a + b)
    a = decoder.rope(decoder.rope(v, pos, 10000.0, 16), pos, 10000.0, 16)
    assert np.allclose(a, decoder.rope(v, 2 * pos, 10000.0, 16))


def _tiny_decoder(layers=3, window=3, seed=0):
    cfg = decoder.DecoderConfig(hidden=32, inter=48, layers=layers, n_q=4, n_kv=1, head_dim=8, vocab=64,
                                window=window, global_layers=(0,))
    import synth
    f32, _, norms = synth.decoder_weights(layers, 32, 48, 64, 4, 1, 8, seed=seed, std=0.2)
    w = dict(f32)
    w.update(norms)
    return cfg, w


def test_decoder_prefill_equals_incremental_decode():
    """Prefill of T tokens in one call gives the same logits as T one-token decode steps with the
    KV cache (the cache and the causal / sliding-window masks are consistent), for the bf16
    mask and for a mixed W8A8 mask."""
    cfg, w = _tiny_decoder()
    toks = np.random.default_rng(3).integers(0, cfg.vocab, (1, 9))
    dec = decoder.OracleDecoder(cfg, w, batch=1, max_len=16)
    dec.calibrate([np.random.default_rng(4).integers(0, cfg.vocab, (1, 12))])
    dec.prepare()
    mask = masks.Mask(frozenset({0, 2}), frozenset({1}), True)
    for mk in (None, mask):
        dec.reset()
        full = dec.forward(toks, 0, mk)["logits"][0]
        dec.reset()
        steps = [dec.forward(toks[:, t:t + 1], t, mk)["logits"][0, 0] for t in range(toks.shape[1])]
        # bf16 roundings see identical inputs both ways, so only fp64 reassociation differs
        assert np.allclose(full, np.stack(steps), rtol=1e-6, atol=1e-6)


def test_sliding_window_hides_old_keys():
    """On a local layer a query at position p sees keys p-window+1 .. p only: changing the
    token at position 0 cannot change a local-only model's output at position >= window."""
    cfg, w = _tiny_decoder(layers=2, window=3)
    cfg.global_layers = ()
    dec = decoder.OracleDecoder(cfg, w, batch=1, max_len=16)
    a = np.array([[5, 9, 13, 17, 21, 25, 29]])
    b = a.copy()
    b[0, 0] = 40
    la = dec.forward(a, 0)["logits"][0]
    dec.reset()
    lb = dec.forward(b, 0)["logits"][0]
    # position t depends on positions >= t - 2*(window-1) through two local layers
    assert not np.allclose(la[1], lb[1])
    assert np.allclose(la[5:], lb[5:], rtol=0, atol=0)


def test_single_key_attention_returns_value():
    cfg, w = _tiny_decoder(layers=1)
    dec = decoder.OracleDecoder(cfg, w, batch=1, max_len=4)
    dec.vc[0, 0, 0] = np.arange(8.0)
    dec.kc[0, 0, 0] = np.ones(8)
    q = np.random.default_rng(0).standard_normal((1, 1, 4, 8))
    o = dec._attention(0, q, 0, 1)
    assert np.allclose(o[0, 0], np.arange(8.0)[None, :])


def test_ffn_block_stages_consistent():
    """The W8A8 block's stages chain: h is bf16(geglu(g, u)) of the fp32 gate/up outputs, and
    down consumes exactly that h."""
    import synth
    c = synth.ffn_case(3, seed=0, hidden=64, inter=96, calib_rows=16)
    prep = blocks.prepare_ffn(c["wg32"], c["wu32"], c["wd32"], W.act_absmax(c["calib32"]), c["stat_h"])
    r = blocks.ffn_w8a8(c["x32"], prep)
    assert np.array_equal(r["h"], W.round_to_bf16(geglu.geglu_f32(r["g"], r["u"])))
    xq, _ = W.quantize_activations(r["h"], prep["down"]["inv_delta"])
    assert np.array_equal(xq, r["down"]["xq"])
    ref = blocks.ffn_bf16(c["x32"], c["wg32"], c["wu32"], c["wd32"])
    assert np.abs(r["y"] - ref["y"]).max() < 0.1 * np.abs(ref["y"]).max()


def test_decoder_sqnr_profile_structure():
    """The oracle's SQNR profile: nothing quantised gives +inf everywhere; in the propagated regime
    the layers before the first quantised one are untouched (+inf: errors do not flow backwards),
    and the first quantised layer has the same SQNR in both regimes (it sees the reference input
    either way); in the isolated regime a layer the mask leaves in bf16 is +inf."""
    cfg, w = _tiny_decoder(layers=4)
    dec = decoder.OracleDecoder(cfg, w, batch=1, max_len=16)
    dec.calibrate([np.random.default_rng(4).integers(0, cfg.vocab, (1, 12))])
    dec.prepare()
    toks = np.random.default_rng(5).integers(0, cfg.vocab, (1, 10))
    none, none_lm = dec.sqnr_profile(toks, masks.Mask(frozenset(), frozenset(), False), isolated=False)
    assert all(v == float("inf") for v in none) and none_lm == float("inf")
    mask = masks.Mask(frozenset({1, 3}), frozenset({2}), True)
    pro, pro_lm = dec.sqnr_profile(toks, mask, isolated=False)
    iso, iso_lm = dec.sqnr_profile(toks, mask, isolated=True)
    assert pro[0] == float("inf") and all(np.isfinite(pro[1:])) and np.isfinite(pro_lm)
    assert iso[0] == float("inf") and all(np.isfinite(iso[1:])) and np.isfinite(iso_lm)
    assert iso[1] == pro[1]


def test_rope_frequencies_by_hand_and_relative_position():
    """Rotate-half RoPE with angle pos * base^(-2i/d) for pair (i, i + d/2): checked element by
    element at d = 4 (pair 0 turns by pos radians, pair 1 by pos / 100 with base 10^4), and the
    defining property: the score of a rotated query and key depends on their positions' difference
    only."""
    x = np.array([[1.0, 2.0, 3.0, 4.0]])
    r = decoder.rope(x, np.array([3]), 10000.0, 4)[0]
    a0, a1 = 3.0, 3.0 / 100.0
    want = [1 * np.cos(a0) - 3 * np.sin(a0), 2 * np.cos(a1) - 4 * np.sin(a1),
            3 * np.cos(a0) + 1 * np.sin(a0), 4 * np.cos(a1) + 2 * np.sin(a1)]
    assert np.allclose(r, want, rtol=0, atol=1e-12)
    g = np.random.default_rng(6)
    q, k = g.standard_normal((1, 256)), g.standard_normal((1, 256))
    for base in (1e4, 1e6):
        def score(m, n):
            return (decoder.rope(q, np.array([m]), base, 256) @ decoder.rope(k, np.array([n]), base, 256).T).item()
        for m, n, s in ((5, 2, 11), (100, 99, 1900), (0, 7, 1024)):
            assert score(m, n) == pytest.approx(score(m + s, n + s), rel=1e-9, abs=1e-9)


def test_rmsnorm_against_torch_and_scale_invariance():
    g = np.random.default_rng(7)
    x = g.standard_normal((9, 1152)) * 3.0
    w = g.uniform(0.5, 1.5, 1152)
    ref = torch.nn.functional.rms_norm(torch.from_numpy(x), (1152,), torch.from_numpy(w), eps=1e-6).numpy()
    assert np.allclose(decoder.rmsnorm(x, w, 1e-6), ref, rtol=1e-12, atol=1e-12)
    assert np.allclose(decoder.rmsnorm(5.0 * x, w, 0.0), decoder.rmsnorm(x, w, 0.0), rtol=1e-12, atol=0)


@pytest.mark.parametrize("glob", [True, False])
def test_attention_against_torch_sdpa(glob):
    """The oracle's attention (scores q.k / sqrt(d), softmax over the allowed keys, 4 query heads
    sharing one key/value head) against torch's scaled_dot_product_attention in fp64 with the causal
    (global layer) or causal sliding-window (local layer) mask written out."""
    cfg, w = _tiny_decoder(layers=1, window=3)
    cfg.global_layers = (0,) if glob else ()
    dec = decoder.OracleDecoder(cfg, w, batch=1, max_len=16)
    g = np.random.default_rng(8)
    T, d = 7, cfg.head_dim
    dec.kc[0, 0, :T] = g.standard_normal((T, cfg.kv_dim))
    dec.vc[0, 0, :T] = g.standard_normal((T, cfg.kv_dim))
    q = g.standard_normal((1, T, cfg.n_q, d))
    got = dec._attention(0, q, 0, T)[0]  # [T, n_q, d]
    K = torch.from_numpy(dec.kc[0, 0, :T].copy()).view(1, 1, T, d).expand(1, cfg.n_q, T, d)
    V = torch.from_numpy(dec.vc[0, 0, :T].copy()).view(1, 1, T, d).expand(1, cfg.n_q, T, d)
    Q = torch.from_numpy(q.copy()).permute(0, 2, 1, 3)  # [1, n_q, T, d]
    i = torch.arange(T)
    allowed = (i[None, :] <= i[:, None]) & (glob | (i[None, :] > i[:, None] - cfg.window))
    ref = torch.nn.functional.scaled_dot_product_attention(Q, K, V, attn_mask=allowed)[0].permute(1, 0, 2).numpy()
    assert np.allclose(got, ref, rtol=1e-12, atol=1e-12)


# ------------------------------------------------------------------- decoder composition
def _composition_decoder(seed=11):
    """One layer, every matrix N(0, 0.2), the final norm's multiplier non-uniform."""
    cfg = decoder.DecoderConfig(hidden=32, inter=48, layers=1, n_q=4, n_kv=1, head_dim=8, vocab=64,
                                window=16, global_layers=(0,))
    import synth
    f32, _, norms = synth.decoder_weights(1, 32, 48, 64, 4, 1, 8, seed=seed, std=0.2)
    w = dict(f32)
    w.update(norms)
    w["final_norm"] = np.linspace(0.5, 1.5, 32).astype(F32)
    return cfg, w


def _logits(cfg, w, toks):
    dec = decoder.OracleDecoder(cfg, w, batch=1, max_len=8)
    return dec.forward(toks, 0)["logits"][0].astype(np.float64)


def test_decoder_closed_form_with_zero_post_norms():
    """With the post-attention and post-FFN norm multipliers zero, a sublayer's output cannot reach
    the residual stream whatever its weights (it enters only through those norms and the residual
    adds), so the residual stream stays at the scaled embedding row.  For a row c * s (s_j = +-1)
    the logits are then the closed form
        logits_v = sum_j E_vj * bf16(s_j * kappa * f_j),  kappa = c S / sqrt(c^2 S^2 + eps),
    S = fl32(sqrt(H)) the embedding scale and f the final norm's multiplier.  c^2 H is chosen
    comparable to eps, where dropping the embedding scale moves kappa from 0.81 to 0.24."""
    cfg, w = _composition_decoder()
    H, eps = cfg.hidden, cfg.eps
    c = 2.0 ** -12
    signs = np.where(np.random.default_rng(12).random((2, H)) < 0.5, -1.0, 1.0)
    w["embed"] = w["embed"].copy()
    w["embed"][[3, 7]] = (c * signs).astype(F32)  # exactly representable in bf16
    w["ln_post_attn"] = [np.zeros(H, F32)]
    w["ln_post_ffn"] = [np.zeros(H, F32)]
    got = _logits(cfg, w, np.array([[3, 7]]))
    S = float(F32(math.sqrt(H)))
    kappa = c * S / math.sqrt(c * c * S * S + eps)
    assert 0.8 < kappa < 0.82 and abs(c / math.sqrt(c * c + eps) - 0.24) < 0.01
    fin = W.round_to_bf16((signs * kappa * w["final_norm"].astype(np.float64)).astype(F32))
    want = fin.astype(np.float64) @ w["embed"].astype(np.float64).T
    assert np.allclose(got, want, rtol=1e-6, atol=1e-7)


def test_decoder_sublayers_enter_through_their_post_norms():
    """Each sublayer's output passes an RMSNorm before the residual add (the sandwich norms), and q
    and k are RMS-normalised before the scores.  Scaling the value rows of W_qkv, W_o, W_up or
    W_down by 4 scales that sublayer's output by exactly 4 (bf16 rounding commutes with powers of
    two), and scaling the query or key rows by 2 leaves the normalised q and k unchanged, so the
    logits move only through eps; doubling a post-norm multiplier or the gate rows does move them.
    A composition that skipped a post-norm, normed the residual sum or left out the QK-norm fails."""
    cfg, w = _composition_decoder()
    toks = np.array([[5, 9, 33, 2]])
    base = _logits(cfg, w, toks)
    qd, kd = cfg.q_dim, cfg.kv_dim
    rows = {"q": slice(0, qd), "k": slice(qd, qd + kd), "v": slice(qd + kd, qd + 2 * kd)}

    def scaled(name, factor, part=None):
        v = {k: (list(x) if isinstance(x, list) else x) for k, x in w.items()}
        m = v[name][0].copy()
        if part is None:
            m = m * F32(factor)
        else:
            m[rows[part]] = m[rows[part]] * F32(factor)
        v[name] = [m]
        return _logits(cfg, v, toks)

    scale = np.abs(base).max()
    for name, factor, part in (("wqkv", 4, "v"), ("wo", 4, None), ("wu", 4, None), ("wd", 4, None),
                               ("wqkv", 2, "q"), ("wqkv", 2, "k")):
        assert np.abs(scaled(name, factor, part) - base).max() < 1e-3 * scale, (name, part)
    for name, factor in (("ln_post_attn", 2), ("ln_post_ffn", 2), ("wg", 2)):
        assert np.abs(scaled(name, factor) - base).max() > 0.05 * scale, name


def test_qk_norm_precedes_rope():
    """QK-norm, then RoPE: a rotation keeps each (i, i + d/2) pair's length, so the cached key of
    one token stays the same length at every position even when the norm's multipliers differ
    between the two dims of a pair.  Normalising after the rotation would weight the rotated
    coordinates, and the length would then depend on the position, as the direct check of the two
    orders on a random vector shows.  The same token at positions 0..5 of one sequence reaches
    layer 0 with the same input, so its raw key row is the same at each position."""
    cfg, w = _composition_decoder()
    d, half = cfg.head_dim, cfg.head_dim // 2
    kn = np.array([0.25, 1.0, 4.0, 0.5, 3.0, 0.5, 1.0, 2.0], F32)  # pair (i, i + 4): unequal weights
    w["k_norm"] = [kn]
    dec = decoder.OracleDecoder(cfg, w, batch=1, max_len=8)
    dec.forward(np.full((1, 6), 9), 0, want_logits=False)
    keys = dec.kc[0, 0, :6, :d]
    lengths = np.linalg.norm(keys, axis=-1)
    assert np.all(np.abs(lengths / lengths[0] - 1.0) < 2.0 ** -6), lengths  # bf16 rounding of the cache
    # the other order on a random row: the length moves with the position by far more than that
    x = np.random.default_rng(3).standard_normal((1, d))
    pos = np.arange(6)
    other = np.stack([decoder.rmsnorm(decoder.rope(x, pos[i:i + 1], cfg.rope_global, d), kn, cfg.eps)[0]
                      for i in range(6)])
    ol = np.linalg.norm(other, axis=-1)
    assert np.abs(ol / ol[0] - 1.0).max() > 0.05, ol
    this = decoder.rope(np.repeat(decoder.rmsnorm(x, kn, cfg.eps), 6, axis=0), pos, cfg.rope_global, d)
    assert np.allclose(np.linalg.norm(this, axis=-1), np.linalg.norm(decoder.rmsnorm(x, kn, cfg.eps)))
    assert half * 2 == d
