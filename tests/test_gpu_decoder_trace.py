"""Teacher-forced, per-step parity of the full 26-layer Gemma-3-1B-shaped decoder (hidden 1152,
FFN 6912, 4 query heads / 1 key-value head of 256, vocab 262144) against the oracle.

The end-to-end decoder test compares logits after every layer's rounding has compounded; here each
step of each layer is checked on the GPU's own inputs, captured by the library's trace
(w8a8_model_set_trace), so no error is amplified by the layers before it:
  * W8A8 linears (q/k/v and o of the mask's attention layers, gate/up + GeGLU and down of its FFN
    layers, the lm_head): outputs bit-exact, given the GPU's bf16 input of that linear;
  * bf16 linears: within 1 bf16 ulp + K 2^-24 sum |x w| of the oracle's fp64 sum;
  * RMSNorm outputs (the q/k/v, FFN and lm_head inputs): within 1 bf16 ulp, almost all equal;
  * attention (QK-norm, RoPE, the bf16 key cache, softmax over the causal / sliding window):
    within 2 bf16 ulps of the oracle's fp64 attention over the GPU's q/k/v rows, plus eta max_k |v_kj|
    for output j: eta = 2^-12 at decode (fp32 throughout), 2^-7 at prefill, whose tensor-core
    attention rounds the scaled query and the probabilities to fp16 (2^-11 relative; a score of
    |q| |k| / 16 = 16 after the QK-norm moves by up to 2^-7, every weight by up to 1.6 %);
  * the residual stream (fp32): within 4e-6 relative of the oracle's fp64 update.
Workload: a 2048-token prefill (tensor-core GEMMs, CTA-pair GeGLU epilogue, prefill attention over
the 1024-position sliding window and the full context of the global layers), sampled at positions
on tile boundaries, then two one-token decode steps (the row-owning decode GEMV with its fused K1,
decode attention), all rows.  Mask: FFN 5+5, attention W8A8 on layers 0, 1, 6, 12 and 25, lm_head
W8A8; the other sublayers run the bf16 pass-through.
"""
import numpy as np
import pytest
import torch

import synth
from oracle import blocks as OB
from oracle import decoder as OD
from oracle import w8a8 as OW

pytestmark = pytest.mark.gpu

L, H, F, V, T = 26, 1152, 6912, 262144, 2048
QD, KVD = 1024, 256
FFN_LAYERS = (0, 1, 2, 3, 4, 21, 22, 23, 24, 25)
ATT_LAYERS = (0, 1, 6, 12, 25)
POS = np.array([0, 1, 5, 127, 128, 1023, 1024, 1500, 2046, 2047])


def bits(layers):
    return sum(1 << l for l in layers)


def ulp_bf16(x):
    return np.spacing(np.abs(x).astype(np.float32)).astype(np.float64) * 2.0 ** 16


@pytest.fixture(scope="module")
def B():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2608_28003_gb300 import build
    build.build()
    from paper_2608_28003_gb300 import binding
    return binding


@pytest.fixture(scope="module")
def run(B):
    f32, bf, norms = synth.decoder_weights(L, seed=0)
    w = {k: [t.cuda() for t in v] if isinstance(v, list) else v.cuda() for k, v in bf.items()}
    n = {k: [torch.from_numpy(a).cuda() for a in v] if isinstance(v, list) else torch.from_numpy(v).cuda()
         for k, v in norms.items()}
    cfg = B.DecoderConfig(max_batch=4, max_seq=T + 16, max_tokens=T)
    dec = B.Decoder(cfg, w, n)
    dec.calibrate(torch.from_numpy(synth.tokens(4 * 128, V, seed=1).reshape(4, 128)).cuda())
    dec.prepare()
    stats = dec.get_stats()
    dec.set_mask(bits(FFN_LAYERS), bits(ATT_LAYERS), 1)
    toks = synth.tokens(T + 2, V, seed=2)
    tt = torch.from_numpy(toks).cuda()
    tr = dec.set_trace(T)
    logits, top1 = dec.forward(tt[:T].view(1, T), 0)
    pre = {k: v.cpu() for k, v in tr.items()}
    pre_logits = logits.view(T, V)[torch.from_numpy(POS).cuda()].cpu().numpy()
    pre_top1 = top1.view(T).cpu().numpy()
    steps = []
    for s in range(2):
        tr = dec.set_trace(1)
        lg, tp = dec.decode_step(tt[T + s:T + s + 1].contiguous(), T + s,
                                 logits=torch.empty(1, V, dtype=torch.float32, device="cuda"))
        steps.append(({k: v.cpu() for k, v in tr.items()}, lg.cpu().numpy(), tp.cpu().numpy()))
    dec.set_trace(None)
    dec.close()
    ow = dict(f32)
    ow.update(norms)
    return {"w": ow, "stats": stats, "toks": toks, "pre": pre, "pre_logits": pre_logits, "pre_top1": pre_top1,
            "steps": steps, "cfg": OD.DecoderConfig()}


@pytest.fixture(scope="module")
def prep(run):
    """The oracle's preparation from the GPU's calibration statistics (the GPU prepares from the
    same statistics with the same rule; that preparation is bit-exact, tested elsewhere)."""
    w, st = run["w"], run["stats"]
    stride = 2 * H + QD + F
    p = {"qkv": {}, "o": {}, "ffn": {}}
    for l in range(L):
        s = st[l * stride:(l + 1) * stride]
        if l in ATT_LAYERS:
            p["qkv"][l] = OW.prepare_weights(w["wqkv"][l], s[:H])
            p["o"][l] = OW.prepare_weights(w["wo"][l], s[H:H + QD])
        if l in FFN_LAYERS:
            p["ffn"][l] = OB.prepare_ffn(w["wg"][l], w["wu"][l], w["wd"][l], s[H + QD:2 * H + QD], s[2 * H + QD:])
    p["lm"] = OW.prepare_weights(w["embed"], st[L * stride:])
    return p


def f32(t):
    return t.float().numpy().astype(np.float64) if t.dtype != torch.float32 else t.numpy().astype(np.float64)


def check_norm(got, want, what="", in_err=0.0):
    """bf16 RMSNorm outputs: fp32 (GPU) against fp64 (oracle) sums, one rounding apart at most;
    in_err bounds what an error of the norm's input (absolute, per element) contributes."""
    want = OW.round_to_bf16(want.astype(np.float32)).astype(np.float64)
    bad = np.abs(got - want) > ulp_bf16(want) + in_err + 1e-30
    assert not bad.any(), (what, np.argwhere(bad)[:5].tolist(), got[bad][:5].tolist(), want[bad][:5].tolist())
    assert np.mean(got == want) > 0.99, what


def check_linear(x, got, int8, prep_q, W32):
    """One linear on the GPU's input rows x (bf16 values)."""
    if int8:
        ref = OW.w8a8_linear(x, prep_q, out="bf16")["y"]
        assert np.array_equal(got, ref)
        return
    ref = OW.bf16_linear(x, W32, out="bf16").astype(np.float64)
    mag = np.abs(x) @ np.abs(W32).astype(np.float64).T
    assert np.all(np.abs(got - ref) <= ulp_bf16(ref) + x.shape[1] * 2.0 ** -24 * mag)


def check_ffn(x, h, y, int8, prep_f, w, l):
    if int8:
        r = OB.ffn_w8a8(x, prep_f)
        assert np.array_equal(h, r["h"]) and np.array_equal(y, r["y"])
        return
    r = OB.ffn_bf16(x, w["wg"][l], w["wu"][l], w["wd"][l])
    assert np.max(np.abs(h - r["h"]) / np.maximum(np.abs(r["h"]), 1e-3)) < 2 ** -6
    check_linear(h, y, False, None, w["wd"][l])


def attention_ref(cfg, w, l, qkv_rows, p):
    """The oracle's attention for the query at position p of layer l, from the GPU's q/k/v rows of
    positions 0..p (qkv_rows[i] is position i)."""
    od = OD.OracleDecoder(OD.DecoderConfig(layers=1, global_layers=(0,) if l in cfg.global_layers else (),
                                           window=cfg.window), {}, batch=1, max_len=p + 1)
    glob = l in cfg.global_layers
    base = cfg.rope_global if glob else cfg.rope_local
    lo = 0 if glob else max(0, p - cfg.window + 1)
    k = OD.rmsnorm(qkv_rows[lo:p + 1, QD:QD + KVD], w["k_norm"][l], cfg.eps)
    k = OD.rope(k, np.arange(lo, p + 1), base, cfg.head_dim)
    od.kc[0, 0, lo:p + 1] = OW.round_to_bf16(k.astype(np.float32))
    od.vc[0, 0, lo:p + 1] = qkv_rows[lo:p + 1, QD + KVD:]
    q = OD.rmsnorm(qkv_rows[p, :QD].reshape(1, cfg.n_q, cfg.head_dim), w["q_norm"][l], cfg.eps)
    q = OD.rope(q, np.array([p]), base, cfg.head_dim)
    o = od._attention(0, q[None], p, 1).reshape(QD)
    vmax = np.abs(qkv_rows[lo:p + 1, QD + KVD:]).max(axis=0)  # max_k |v_kj| per dim of the shared head
    return OW.round_to_bf16(o.astype(np.float32)).astype(np.float64), np.tile(vmax, cfg.n_q)


def check_layers(run, prep, tr, rows, positions, qkv_all, eta):
    """Every layer's steps at the given trace rows (query positions `positions`); qkv_all(l) gives
    the GPU's q/k/v rows of positions 0..max for the attention reference."""
    w, cfg, toks = run["w"], run["cfg"], run["toks"]
    for l in range(L):
        att8, ffn8 = l in ATT_LAYERS, l in FFN_LAYERS
        a_in = f32(tr["a_in"][l, rows])
        if l == 0:
            r_prev = (w["embed"][toks[positions]].astype(np.float32) * np.float32(cfg.embed_scale)).astype(np.float64)
        else:
            r_prev = f32(tr["r"][l - 1, rows])
        check_norm(a_in, OD.rmsnorm(r_prev, w["ln_in"][l], cfg.eps), ("a_in", l))
        qkv = f32(tr["qkv"][l, rows])
        check_linear(a_in, qkv, att8, prep["qkv"].get(l), w["wqkv"][l])
        attn = f32(tr["attn"][l, rows])
        allq = qkv_all(l)
        for i, p in enumerate(positions):
            ref, vmax = attention_ref(cfg, w, l, allq, int(p))
            assert np.all(np.abs(attn[i] - ref) <= 2 * ulp_bf16(ref) + eta * vmax), (l, int(p))
        y_o = f32(tr["y_o"][l, rows])
        check_linear(attn, y_o, att8, prep["o"].get(l), w["wo"][l])
        n_o = OD.rmsnorm(y_o, w["ln_post_attn"][l], cfg.eps)
        r_mid = r_prev + n_o
        a_ffn = f32(tr["a_ffn"][l, rows])
        # the GPU forms r_mid in fp32 (not traced): a few roundings of |r_prev| + |n_o| at 2^-24 each,
        # scaled by the pre-FFN norm (1 / rms(r_mid) times its weight)
        inv = 1.0 / np.sqrt(np.mean(r_mid ** 2, axis=1, keepdims=True) + cfg.eps)
        mid_err = 4 * 2.0 ** -24 * (np.abs(r_prev) + np.abs(n_o)) * inv * np.abs(w["ln_pre_ffn"][l])
        check_norm(a_ffn, OD.rmsnorm(r_mid, w["ln_pre_ffn"][l], cfg.eps), ("a_ffn", l), mid_err)
        h, y_f = f32(tr["h"][l, rows]), f32(tr["y_f"][l, rows])
        check_ffn(a_ffn, h, y_f, ffn8, prep["ffn"].get(l), w, l)
        r = f32(tr["r"][l, rows])
        r_ref = r_mid + OD.rmsnorm(y_f, w["ln_post_ffn"][l], cfg.eps)
        assert np.all(np.abs(r - r_ref) <= 4e-6 * np.max(np.abs(r_ref), axis=1, keepdims=True)), l
    a_fin = f32(tr["a_fin"][rows])
    check_norm(a_fin, OD.rmsnorm(f32(tr["r"][L - 1, rows]), w["final_norm"], cfg.eps), "a_fin")
    return a_fin


def test_prefill_2048_every_layer_teacher_forced(run, prep):
    pre = run["pre"]
    a_fin = check_layers(run, prep, pre, POS, POS, lambda l: f32(pre["qkv"][l]), 2.0 ** -7)
    head = OB.lm_head_w8a8(a_fin, prep["lm"])
    assert np.array_equal(run["pre_logits"].view(np.uint32), head["logits"].view(np.uint32))
    assert np.array_equal(run["pre_top1"][POS], head["top1"])


@pytest.mark.parametrize("step", [0, 1])
def test_decode_steps_every_layer_teacher_forced(run, prep, step):
    pre = run["pre"]
    prev = [s[0] for s in run["steps"][:step + 1]]
    pos = T + step

    def qkv_all(l):  # the prefill's rows, then the decode steps' rows so far
        return np.concatenate([f32(pre["qkv"][l])] + [f32(t["qkv"][l, :1]) for t in prev])

    tr, lg, tp = run["steps"][step]
    a_fin = check_layers(run, prep, tr, np.array([0]), np.array([pos]), qkv_all, 2.0 ** -12)
    head = OB.lm_head_w8a8(a_fin, prep["lm"])
    assert np.array_equal(lg.view(np.uint32), head["logits"].view(np.uint32))
    assert np.array_equal(tp, head["top1"])
