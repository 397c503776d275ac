"""GPU parity of the FFN block and lm_head against the oracle, through the C ABI.

W8A8 paths are bit-exact (h, Y, logits, top-1).  bf16 paths are within 1 bf16 ulp plus the
fp32 accumulation bound; their top-1 must equal the oracle's wherever the oracle's margin
between the two best logits exceeds that bound.
"""
import numpy as np
import pytest
import torch

import synth
from oracle import blocks as OB
from oracle import w8a8 as OW

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def B():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2608_28003_gb300 import build
    build.build()
    from paper_2608_28003_gb300 import binding
    return binding


def cu(t):
    return t.contiguous().cuda()


def f32_of_bf16(t):
    return t.detach().cpu().float().numpy()


@pytest.fixture(scope="module")
def ffn(B):
    c = synth.ffn_case(2048, seed=0)  # rows 0..M-1 of this draw are the M-token inputs
    stat_in = OW.act_absmax(c["calib32"])
    # fp16 code copies too: 64 tokens take the tensor-core GEMM
    gu = B.prepare_gate_up(cu(c["wg"]), cu(c["wu"]), cu(torch.from_numpy(stat_in)), want_f16=True)
    dn = B.prepare_weights(cu(c["wd"]), cu(torch.from_numpy(c["stat_h"])), want_f16=True)
    f = B.FfnWeights(1152, 6912, gu, dn, B.interleave_gate_up(cu(c["wg"]), cu(c["wu"])), cu(c["wd"]))
    prep = OB.prepare_ffn(c["wg32"], c["wu32"], c["wd32"], stat_in, c["stat_h"])
    return c, f, prep


@pytest.mark.parametrize("M", [1, 3, 5, 8, 9, 13, 16, 24, 32, 64])
def test_ffn_w8a8_bit_exact(B, ffn, M):
    c, f, prep = ffn
    x = c["x"][:M]
    Y, h = B.ffn_block(f, B.W8A8_PREC_W8A8, cu(x), want_h=True)
    r = OB.ffn_w8a8(c["x32"][:M], prep)
    assert np.array_equal(f32_of_bf16(h), r["h"])
    assert np.array_equal(f32_of_bf16(Y), r["y"])


def _sample_rows(M):
    """Rows on tile and pair-tile boundaries (128 / 256 tokens), the ragged tail and a few drawn at
    random: the FFN is row-independent (per-token scales), so the oracle computes just these."""
    idx = {0, 1, 127, 128, 255, 256, M // 2, M - 2, M - 1}
    idx |= set(np.random.default_rng(M).integers(0, M, 7).tolist())
    return np.array(sorted(i for i in idx if 0 <= i < M))


@pytest.mark.parametrize("M", [300, 512, 2048])
def test_ffn_w8a8_large_m_sampled_bit_exact(B, ffn, M):
    """Prefill sizes: gate/up on the CTA-pair tensor-core GEMM with the GeGLU epilogue (16-column
    gate/up blocks, swizzled staging, TMA stores of half-width rows), down on the tensor-core GEMM;
    h and Y of sampled rows bit-exact, every column."""
    c, f, prep = ffn
    Y, h = B.ffn_block(f, B.W8A8_PREC_W8A8, cu(c["x"][:M]), want_h=True)
    idx = _sample_rows(M)
    r = OB.ffn_w8a8(c["x32"][idx], prep)
    assert np.array_equal(f32_of_bf16(h)[idx], r["h"])
    assert np.array_equal(f32_of_bf16(Y)[idx], r["y"])


def _bf16_ffn_check(c, h, Y, rows):
    """h within a few ulps of the oracle's; Y within 1 ulp + the fp32 bound of the oracle's down
    projection fed the GPU's own h."""
    r = OB.ffn_bf16(c["x32"][rows], c["wg32"], c["wu32"], c["wd32"])
    hg, hr = f32_of_bf16(h)[rows], r["h"]
    scale = np.maximum(np.abs(hr), 1e-3)
    assert np.max(np.abs(hg - hr) / scale) < 2 ** -6
    yref = OW.bf16_linear(hg, c["wd32"], out="bf16")
    mag = np.abs(hg).astype(np.float64) @ np.abs(c["wd32"]).astype(np.float64).T
    ulp = np.spacing(np.abs(yref).astype(np.float32)) * 2 ** 16
    assert np.all(np.abs(f32_of_bf16(Y)[rows] - yref) <= ulp + 6912 * 2.0 ** -24 * mag)


@pytest.mark.parametrize("M", [300, 512, 2048])
def test_ffn_bf16_large_m_sampled(B, ffn, M):
    c, f, _ = ffn
    Y, h = B.ffn_block(f, B.W8A8_PREC_BF16, cu(c["x"][:M]), want_h=True)
    _bf16_ffn_check(c, h, Y, _sample_rows(M))


@pytest.mark.parametrize("M", [1, 5, 8, 64])
def test_ffn_bf16_within_tolerance(B, ffn, M):
    c, f, _ = ffn
    Y, h = B.ffn_block(f, B.W8A8_PREC_BF16, cu(c["x"][:M]), want_h=True)
    # h: g and u carry fp32 accumulation error before the activation (a few ulps); down consumes
    # the GPU's own h and is checked against the oracle fed the same h
    _bf16_ffn_check(c, h, Y, np.arange(M))


@pytest.fixture(scope="module")
def head(B):
    c = synth.lm_head_case(16, seed=0)
    stat = OW.act_absmax(c["calib32"])
    q = B.prepare_weights(cu(c["w"]), cu(torch.from_numpy(stat)))
    hd = B.HeadWeights(262144, 1152, q, cu(c["w"]))
    prep = OW.prepare_weights(c["w32"], stat)
    return c, hd, prep


@pytest.mark.parametrize("M", [1, 16])
def test_lm_head_w8a8_bit_exact(B, head, M):
    c, hd, prep = head
    logits, top1 = B.lm_head(hd, B.W8A8_PREC_W8A8, cu(c["x"][:M]))
    r = OB.lm_head_w8a8(c["x32"][:M], prep)
    assert np.array_equal(logits.cpu().numpy().view(np.uint32), r["logits"].view(np.uint32))
    assert np.array_equal(top1.cpu().numpy(), r["top1"])
    # top-1 alone (no logits written) gives the same index
    _, t2 = B.lm_head(hd, B.W8A8_PREC_W8A8, cu(c["x"][:M]), want_logits=False)
    assert np.array_equal(t2.cpu().numpy(), r["top1"])


def test_lm_head_top1_ties_pick_lowest_index(B):
    """Rows 5, 900 and 70000 of the table are identical, so their logits tie exactly."""
    V, D = 131072, 128
    w32, w = synth.weight(V, D, seed=9, std=0.02)
    w[900] = w[5]
    w[70000] = w[5]
    w32 = w.float().numpy()
    x = (w[5].float() * 40).to(torch.bfloat16)[None, :]
    q = B.prepare_weights(cu(w), None, 0.5, False)
    hd = B.HeadWeights(V, D, q, cu(w))
    for prec in (B.W8A8_PREC_W8A8, B.W8A8_PREC_BF16):
        logits, top1 = B.lm_head(hd, prec, cu(x))
        lg = logits.cpu().numpy()[0]
        assert lg[5] == lg[900] == lg[70000] == lg.max()
        assert int(top1.cpu()[0]) == 5


@pytest.mark.parametrize("M", [1, 16])
def test_lm_head_bf16_within_tolerance(B, head, M):
    c, hd, _ = head
    logits, top1 = B.lm_head(hd, B.W8A8_PREC_BF16, cu(c["x"][:M]))
    r = OB.lm_head_bf16(c["x32"][:M], c["w32"])
    x = c["x32"][:M].astype(np.float64)
    mag = np.abs(x) @ np.abs(c["w32"]).astype(np.float64).T
    bound = 1152 * 2.0 ** -24 * mag + 1e-30
    lg = logits.cpu().numpy()
    assert np.all(np.abs(lg - r["logits"]) <= bound)
    srt = np.sort(r["logits"], axis=1)
    clear = (srt[:, -1] - srt[:, -2]) > 2 * bound.max(axis=1)
    t = top1.cpu().numpy()
    assert np.array_equal(t[clear], r["top1"][clear])
    assert np.all(lg[np.arange(M), t] == lg.max(axis=1))


@pytest.fixture(scope="module")
def head16(B, head):
    """The same lm_head with the fp16 copy of the codes (the tensor-core GEMM's operand)."""
    c, hd, prep = head
    q = hd.q
    q16 = B.prepare_weights(cu(c["w"]), q.delta.new_tensor(OW.act_absmax(c["calib32"])), want_f16=True)
    assert torch.equal(q16.wq, q.wq)
    return c, B.HeadWeights(262144, 1152, q16, hd.bf16), prep


@pytest.mark.parametrize("M", [128, 512])
def test_lm_head_w8a8_tensor_core_sampled(B, head16, M):
    c, hd, prep = head16
    x32, x = synth.normed_rows(M, 1152, seed=M + 7)
    logits, top1 = B.lm_head(hd, B.W8A8_PREC_W8A8, cu(x))
    idx = np.array([0, 1, 77, M // 2, M - 1])
    r = OB.lm_head_w8a8(x32[idx], prep)
    assert np.array_equal(logits.cpu().numpy()[idx].view(np.uint32), r["logits"].view(np.uint32))
    assert np.array_equal(top1.cpu().numpy()[idx], r["top1"])
    lg = logits.cpu().numpy()
    assert np.array_equal(top1.cpu().numpy(), np.argmax(lg, axis=1))


def test_lm_head_bf16_tensor_core_sampled(B, head):
    c, hd, _ = head
    M = 128
    x32, x = synth.normed_rows(M, 1152, seed=3)
    logits, top1 = B.lm_head(hd, B.W8A8_PREC_BF16, cu(x))
    idx = np.array([0, 5, 64, 127])
    r = OB.lm_head_bf16(x32[idx], c["w32"])
    mag = np.abs(x32[idx]).astype(np.float64) @ np.abs(c["w32"]).astype(np.float64).T
    lg = logits.cpu().numpy()
    assert np.all(np.abs(lg[idx] - r["logits"]) <= 1152 * 2.0 ** -24 * mag + 1e-30)
    t = top1.cpu().numpy()
    assert np.all(lg[np.arange(M), t] == lg.max(axis=1))


@pytest.mark.parametrize("M", [128, 512])
def test_lm_head_w8a8_large_m_sampled(B, head, M):
    """Large token counts (several token groups per launch): sampled tokens against the oracle
    computing just those rows."""
    c, hd, prep = head
    x32, x = synth.normed_rows(M, 1152, seed=M)
    logits, top1 = B.lm_head(hd, B.W8A8_PREC_W8A8, cu(x))
    idx = np.array([0, 1, M // 2, M - 1])
    r = OB.lm_head_w8a8(x32[idx], prep)
    assert np.array_equal(logits.cpu().numpy()[idx].view(np.uint32), r["logits"].view(np.uint32))
    assert np.array_equal(top1.cpu().numpy()[idx], r["top1"])
