"""GPU parity of the FP8 (e4m3) variant against the oracle, through the C ABI.

Codes and scales are decided in fp32 on both sides with the same operations and the hardware's
e4m3 conversion (nearest even, saturating), so they must match bit for bit: the weight codes and
s_w of the preparation, the activation codes and s_x of K1.  The GEMM sums e4m3 products in fp32
in the kernel's order, which is not exact (the exact sum can need 49 bits), so its outputs are held
to the bound of fp32 summation: for output (t, i)
    |Y - Y_oracle| <= ulp_bf16(Y_oracle) + s_x s_w (K 2^-23 sum_j |xq_tj wq_ij|) + 2^-22 |Y_oracle|
(the oracle sums exactly; the last term covers the scale products' own rounding).
"""
import numpy as np
import pytest
import torch

import synth
from oracle import blocks as OB
from oracle import fp8 as OF
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


def codes_equal(gpu_bytes, oracle_values):
    """Bytes decode to the oracle's values, and equal the oracle's encoding wherever it is not 0."""
    g = gpu_bytes.cpu().numpy()
    v = OF.e4m3_decode(g)
    assert np.array_equal(v, oracle_values)
    nz = oracle_values != 0
    assert np.array_equal(g[nz], OF.e4m3_encode(oracle_values[nz]))


def within_fp32_sum_bound(Y, ref, K):
    """Y (GPU, bf16 tensor) against the oracle's fp8_linear result `ref` (exact sums)."""
    y = Y.float().cpu().numpy().astype(np.float64)
    yr = ref["y"].astype(np.float64)
    mag = np.abs(ref["xq"]) @ np.abs(ref["wq_used"]).T
    scale = ref["s_x"].astype(np.float64)[:, None] * ref["s_w_used"].astype(np.float64)[None, :]
    ulp = np.spacing(np.abs(yr).astype(np.float32)).astype(np.float64) * 2 ** 16
    bound = ulp + scale * K * 2.0 ** -23 * mag + 2.0 ** -22 * np.abs(yr)
    err = np.abs(y - yr)
    assert np.all(err <= bound), float(np.max(err - bound))
    return float(np.mean(err == 0))


@pytest.fixture(scope="module")
def lin(B):
    c = synth.linear_case(300)  # the single-linear workload's distribution, 300 tokens
    stat = OW.act_absmax(c["calib32"])
    q = B.fp8_prepare_weights(cu(c["w"]), cu(torch.from_numpy(stat)))
    prep = OF.prepare_weights_fp8(c["w32"], stat)
    return c, q, prep


def test_fp8_weight_codes_and_scales_bit_exact(B, lin):
    c, q, prep = lin
    codes_equal(q.wq, prep["wq"])
    assert np.array_equal(q.s_w.cpu().numpy().view(np.uint32), prep["s_w"].view(np.uint32))
    assert np.array_equal(q.inv_delta.cpu().numpy().view(np.uint32), prep["inv_delta"].view(np.uint32))
    # the rule's invariants: every non-zero row reaches +-448 exactly
    assert np.all(np.abs(prep["wq"]).max(axis=1) == 448.0)


def test_fp8_zero_row_and_saturation(B):
    K = 64
    w = torch.zeros(32, K, dtype=torch.bfloat16)
    w[1] = torch.linspace(-3, 3, K).to(torch.bfloat16)
    w[2, 5] = 1e-30  # a row whose only non-zero element is its maximum
    q = B.fp8_prepare_weights(cu(w), None, 0.5, False)
    prep = OF.prepare_weights_fp8(w.float().numpy(), None, smooth=False)
    codes_equal(q.wq, prep["wq"])
    assert float(q.s_w[0]) == 0.0 and np.all(q.wq[0].cpu().numpy() == 0)


@pytest.mark.parametrize("M", [1, 5, 300])
def test_fp8_activation_codes_bit_exact(B, lin, M):
    c, q, prep = lin
    xq, s_x = B.fp8_quantize_activations(cu(c["x"][:M]), q.inv_delta)
    xh = OW.smooth_activations(c["x32"][:M], prep["inv_delta"])
    rq, rs = OF.quantize_rows_fp8(xh)
    codes_equal(xq, rq)
    assert np.array_equal(s_x.cpu().numpy().view(np.uint32), rs.view(np.uint32))


def _oracle_linear(x32, prep):
    r = OF.fp8_linear(x32, prep, out="bf16")
    r["wq_used"], r["s_w_used"] = prep["wq"], prep["s_w"]
    return r


@pytest.mark.parametrize("M", [1, 2, 3, 8, 16, 64, 300])
def test_fp8_linear_within_fp32_sum_bound(B, lin, M):
    """1-2 tokens: the decode GEMV with the codes widened to fp32 for FMAs; 3-16: the decode GEMV
    on the tensor cores (e4m3 widened to fp16, mma.sync); K1 fused in both; more: K1 then the
    tcgen05 kind::f8f6f4 GEMM (single-CTA tiles, split-K at decode sizes)."""
    c, q, prep = lin
    Y, dbg = B.fp8_linear(q, cu(c["x"][:M]), debug=True)
    r = _oracle_linear(c["x32"][:M], prep)
    codes_equal(dbg["xq"], r["xq"])
    assert np.array_equal(dbg["s_x"].cpu().numpy().view(np.uint32), r["s_x"].view(np.uint32))
    exact = within_fp32_sum_bound(Y, r, 1152)
    assert exact > 0.9  # most outputs round to the same bf16 value


@pytest.fixture(scope="module")
def ffn8(B):
    c = synth.ffn_case(2048, seed=0)
    stat_in = OW.act_absmax(c["calib32"])
    gu = B.fp8_prepare_gate_up(cu(c["wg"]), cu(c["wu"]), cu(torch.from_numpy(stat_in)))
    dn = B.fp8_prepare_weights(cu(c["wd"]), cu(torch.from_numpy(c["stat_h"])))
    f = B.Fp8FfnWeights(1152, 6912, gu, dn)
    prep = OB.prepare_ffn_fp8(c["wg32"], c["wu32"], c["wd32"], stat_in, c["stat_h"])
    return c, f, prep


@pytest.mark.parametrize("M", [1, 2, 8, 64, 512, 2048])
def test_fp8_ffn_block(B, ffn8, M):
    """The block at the FFN workload's token counts: h within a few ulps of the oracle's (g and u
    carry the fp32 summation error before the activation), Y within the bound of the oracle's down
    projection fed the GPU's own h; sampled rows at prefill sizes (the block is row-independent)."""
    c, f, prep = ffn8
    Y, h = B.fp8_ffn_block(f, cu(c["x"][:M]), want_h=True)
    rows = np.arange(M) if M <= 64 else np.array(sorted({0, 1, 127, 128, 255, 256, M // 2, M - 1}))
    r = OB.ffn_fp8(c["x32"][rows], prep)
    hg = h.float().cpu().numpy()[rows]
    rel = np.abs(hg - r["h"]) / np.maximum(np.abs(r["h"]), 1e-2)
    assert np.max(rel) < 2 ** -5 and np.mean(hg == r["h"]) > 0.9
    dn = _oracle_linear(hg, prep["down"])
    within_fp32_sum_bound(Y[torch.from_numpy(rows).cuda()], dn, 6912)
