"""GPU parity of the W8A8 linear path against the oracle, through the C ABI.

Bar: INT8 codes, INT32 accumulators, fp32 scales, bf16/fp32 outputs of the W8A8 path are
bit-exact; the bf16 pass-through is within 1 bf16 ulp plus the fp32 accumulation bound
(K * 2^-24 * sum |x w|) of the oracle's fp64 sum.
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


def bits16(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def f32_of_bf16(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().float().numpy()


def _case(M, N, K, seed, n_out=4):
    x32, x, ch = synth.activations(M, K, min(n_out, K), seed)
    w32, w = synth.weight(N, K, seed)
    c32, c, _ = synth.activations(max(M, 8), K, min(n_out, K), seed, stream=1, channels=ch)
    return x32, x, w32, w, c32, c


# ------------------------------------------------------------------ K1 activation quantiser
@pytest.mark.parametrize("M,K", [(1, 1152), (16, 1152), (3, 16), (37, 6912), (5, 9216), (130, 1040)])
def test_quantize_activations_bit_exact(B, M, K):
    x32, x, _ = synth.activations(M, K, min(8, K), seed=M + K)
    inv = np.random.default_rng(K).uniform(0.05, 20.0, K).astype(np.float32)
    if M > 2:
        x32[2] = 0.0
        x[2] = 0
    xq, xf, sx = B.quantize_activations(cu(x), cu(torch.from_numpy(inv)))
    oq, os_ = OW.quantize_activations(x32, inv)
    assert np.array_equal(xq.cpu().numpy(), oq)
    assert np.array_equal(sx.cpu().numpy().view(np.uint32), os_.view(np.uint32))
    assert np.array_equal(xf.cpu().float().numpy(), oq.astype(np.float32))


def test_act_absmax_bit_exact(B):
    x32, x, _ = synth.activations(300, 1152, 12, seed=5)
    am = B.act_absmax(cu(x))
    am = B.act_absmax(cu(x[:7] * 3), am)
    ref = np.maximum(OW.act_absmax(x32), OW.act_absmax((x[:7] * 3).float().numpy()))
    assert np.array_equal(am.cpu().numpy(), ref)


# ------------------------------------------------------------------------- weight prep
@pytest.mark.parametrize("N,K,alpha,smooth", [(6912, 1152, 0.5, True), (100, 64, 0.5, False), (40, 6912, 0.5, True),
                                              (33, 1040, 0.3, True)])
def test_prepare_weights(B, N, K, alpha, smooth):
    _, _, w32, w, c32, c = _case(8, N, K, seed=N)
    stat = OW.act_absmax(c32)
    stat[5] = 0.0
    q = B.prepare_weights(cu(w), cu(torch.from_numpy(stat)), alpha, smooth, want_f16=True)
    ref = OW.prepare_weights(w32, stat, alpha, smooth)
    if alpha == 0.5:
        assert np.array_equal(q.delta.cpu().numpy(), ref["delta"])
        assert np.array_equal(q.inv_delta.cpu().numpy(), ref["inv_delta"])
        assert np.array_equal(q.wq.cpu().numpy(), ref["wq"])
        assert np.array_equal(q.s_w.cpu().numpy(), ref["s_w"])
    else:  # fp64 pow on both sides, one rounding to fp32: at most 1 ulp apart
        d = q.delta.cpu().numpy()
        assert np.all(np.abs(d.view(np.int32) - ref["delta"].view(np.int32)) <= 1)
        same = d == ref["delta"]
        assert same.mean() > 0.99
        assert np.array_equal(q.wq.cpu().numpy()[:, same], ref["wq"][:, same])
    assert np.array_equal(q.wq_f16.cpu().float().numpy(), q.wq.cpu().numpy().astype(np.float32))


def deinterleave_rows(a: np.ndarray, F: int) -> np.ndarray:
    """Inverse of the 8-row gate/up interleave: fused row p -> [gate; up] row."""
    p = np.arange(2 * F)
    q, r = p // 16, p % 16
    dst = np.where(r < 8, 8 * q + r, F + 8 * q + r - 8)
    out = np.empty_like(a)
    out[dst] = a
    return out


def test_prepare_gate_up_and_interleave(B):
    F, H = 6912, 1152
    c = synth.ffn_case(4, seed=3, calib_rows=64)
    stat = OW.act_absmax(c["calib32"])
    q = B.prepare_gate_up(cu(c["wg"]), cu(c["wu"]), cu(torch.from_numpy(stat)))
    ref = OW.prepare_weights(np.concatenate([c["wg32"], c["wu32"]]), stat)
    assert np.array_equal(q.delta.cpu().numpy(), ref["delta"])
    assert np.array_equal(deinterleave_rows(q.wq.cpu().numpy(), F), ref["wq"])
    assert np.array_equal(deinterleave_rows(q.s_w.cpu().numpy(), F), ref["s_w"])
    il = B.interleave_gate_up(cu(c["wg"]), cu(c["wu"]))
    assert np.array_equal(deinterleave_rows(bits16(il), F), np.concatenate([bits16(c["wg"]), bits16(c["wu"])]))


# ------------------------------------------------------------------------- W8A8 linear
LINEAR_SHAPES = [
    (16, 6912, 1152),   # the single-linear workload (gate_proj shape, M = 16)
    (1, 1000, 1152),    # ragged N
    (3, 24, 64),
    (2, 700, 2048),     # dp4a GEMV with two token slots
    (9, 4112, 1040),    # ragged K (not a multiple of 64)
    (17, 200, 6912),    # K-split across CTAs
    (33, 520, 1152),
    (64, 1152, 6912),   # down_proj shape
    (130, 300, 256),    # several token groups with a ragged tail
    (5, 1536, 1152),    # row-owning decode GEMV, 8 token slots (qkv shape)
    (8, 1152, 6912),    # row-owning decode GEMV, K past one stage ring (down_proj shape)
    (4, 1152, 1024),    # o_proj shape
    (7, 9, 16),         # fewer rows than one CTA's eight, K of one vector
    (2, 64, 9216),      # K too long for the fused quantiser: K1 + streaming kernel
    (13, 1536, 1152),   # row-owning decode GEMV, 16 token slots (both halves of the MMA's A tile)
    (11, 1000, 1152),   # 16 slots, ragged N and tokens
    (16, 1152, 1024),   # 16 slots, o_proj shape
]


@pytest.mark.parametrize("M,N,K", LINEAR_SHAPES)
def test_w8a8_linear_bit_exact(B, M, N, K):
    x32, x, w32, w, c32, c = _case(M, N, K, seed=M * 7 + N)
    stat = OW.act_absmax(np.concatenate([c32, x32]))
    q = B.prepare_weights(cu(w), cu(torch.from_numpy(stat)))
    bias = None
    if N == 1000:
        bias = np.random.default_rng(1).standard_normal(N).astype(np.float32)
    Y, dbg = B.linear(q, cu(x), bias=cu(torch.from_numpy(bias)) if bias is not None else None, debug=True)
    prep = OW.prepare_weights(w32, stat)
    r = OW.w8a8_linear(x32, prep, bias=bias, out="bf16")
    assert np.array_equal(dbg["xq"].cpu().numpy(), r["xq"])
    assert np.array_equal(dbg["s_x"].cpu().numpy(), r["s_x"])
    assert np.array_equal(dbg["acc"].cpu().numpy().astype(np.int64), r["acc"])
    assert np.array_equal(f32_of_bf16(Y), r["y"])


TC_SHAPES = [
    (16, 6912, 1152),    # the single-linear workload: 128 x 64 tiles, 15/16 of each tile padding
    (9, 1536, 1152),     # fewest tokens the tensor-core path takes
    (40, 1152, 6912),    # ragged M, seven k chunks
    (64, 1152, 6912),    # seven 1024-k chunks folded into INT32
    (32, 1152, 6912),    # split-K: 18 tiles of 128 x 64, k cut into 8 parts on 144 CTAs
    (200, 1152, 6912),   # split-K over two row blocks of a ragged M, parts of 27 stages
    (24, 1040, 4096),    # split-K with a bias added once, after the parts are summed
    (130, 4112, 1040),   # ragged M, K not a multiple of the 64-wide stage
    (256, 1536, 1152),
    (200, 13824, 1152),  # gate/up shape, ragged M: CTA pairs on 256 x 192 tiles
    (300, 4608, 2176),   # ragged M, three k chunks
    (512, 13824, 1152),  # CTA pairs on 256 x 192 tiles, two k chunks
    (1024, 13824, 1152), # CTA pairs on 256 x 256 tiles
]


@pytest.mark.parametrize("M,N,K", TC_SHAPES)
def test_w8a8_linear_tensor_core_bit_exact(B, M, N, K):
    """Prefill-sized calls with the fp16 code copy take the tcgen05 GEMM: codes, scales and INT32
    sums bit for bit, bf16 outputs bit for bit."""
    x32, x, w32, w, c32, c = _case(M, N, K, seed=M * 3 + K)
    stat = OW.act_absmax(np.concatenate([c32, x32]))
    q = B.prepare_weights(cu(w), cu(torch.from_numpy(stat)), want_f16=True)
    bias = np.random.default_rng(2).standard_normal(N).astype(np.float32) if N == 1040 else None
    Y, dbg = B.linear(q, cu(x), bias=cu(torch.from_numpy(bias)) if bias is not None else None, debug=True)
    r = OW.w8a8_linear(x32, OW.prepare_weights(w32, stat), bias=bias, out="bf16")
    assert np.array_equal(dbg["xq"].cpu().numpy(), r["xq"])
    assert np.array_equal(dbg["s_x"].cpu().numpy(), r["s_x"])
    assert np.array_equal(dbg["acc"].cpu().numpy().astype(np.int64), r["acc"])
    assert np.array_equal(f32_of_bf16(Y), r["y"])


def test_single_linear_workload_calibrated_on_its_input(B):
    """M = 16, K = 1152, N = 6912, 8 outlier channels x20, delta from X itself (seed 0)."""
    c = synth.linear_case()
    stat = OW.act_absmax(c["calib32"])
    q = B.prepare_weights(cu(c["w"]), cu(torch.from_numpy(stat)))
    Y, dbg = B.linear(q, cu(c["x"]), debug=True)
    r = OW.w8a8_linear(c["x32"], OW.prepare_weights(c["w32"], stat), out="bf16")
    assert np.array_equal(dbg["acc"].cpu().numpy().astype(np.int64), r["acc"])
    assert np.array_equal(f32_of_bf16(Y), r["y"])
    # every token row has an outlier channel mapped to +-127
    assert np.all(np.abs(r["xq"].astype(int)).max(axis=1) == 127)


@pytest.mark.parametrize("K", [1024, 1152, 6912])
def test_w8a8_accumulator_exact_at_extremes(B, K):
    """All codes +-127 (delta = 1, constant-magnitude rows), |acc| up to 127^2 K > 2^24: the fp32
    MMA accumulation is folded into INT32 before it can round."""
    M, N = 8, 48
    g = np.random.default_rng(K)
    x = np.where(g.random((M, K)) < 0.5, -1.0, 1.0).astype(np.float32)
    x[0] = 1.0
    w = np.where(g.random((N, K)) < 0.5, -0.5, 0.5).astype(np.float32)
    w[0] = 0.5
    w[1] = -0.5
    w[2, : K // 2] = 0.5
    w[2, K // 2:] = -0.5
    xt = torch.from_numpy(x).to(torch.bfloat16)
    wt = torch.from_numpy(w).to(torch.bfloat16)
    q = B.prepare_weights(cu(wt), None, 0.5, False)
    assert np.all(np.abs(q.wq.cpu().numpy()) == 127)
    Y, dbg = B.linear(q, cu(xt), debug=True)
    r = OW.w8a8_linear(x, OW.prepare_weights(w, None, smooth=False), out="bf16")
    acc = dbg["acc"].cpu().numpy().astype(np.int64)
    assert np.array_equal(acc, r["acc"]) and acc[0, 0] == 127 * 127 * K
    assert np.array_equal(f32_of_bf16(Y), r["y"])


@pytest.mark.parametrize("M,N,K,bad", [(640, 4608, 1152, (256, 512)),   # CTA pairs, 256-token row tiles
                                       (1024, 1152, 6912, (128, 256))])  # single CTAs, 128-token row tiles
def test_tc_exactness_bound_mixed_tiles(B, M, N, K, bad):
    """The tensor-core GEMM keeps one fp32 accumulator per tile when every token of the row tile
    has 127 sum_k |q| <= 2^24, and folds every 1024 k otherwise.  Here the rows of one tile are all
    +-1 (every code +-127: sum 127 K, past the bound; acc up to 127^2 K > 2^24, which only the folds
    keep exact) and the other tiles are small values with one spike per row (sums far below it), so
    both paths run in one call; every INT32 sum and output is compared bit for bit."""
    g = np.random.default_rng(M + K)
    x = (0.05 * g.standard_normal((M, K))).astype(np.float32)
    x[np.arange(M), g.integers(0, K, M)] = 1.0
    lo, hi = bad
    x[lo:hi] = np.where(g.random((hi - lo, K)) < 0.5, -1.0, 1.0)
    w = np.where(g.random((N, K)) < 0.5, -0.5, 0.5).astype(np.float32)
    w[0] = np.sign(x[lo]) * 0.5  # acc[lo, 0] = 127^2 K
    xt, wt = torch.from_numpy(x).to(torch.bfloat16), torch.from_numpy(w).to(torch.bfloat16)
    x = xt.float().numpy()
    q = B.prepare_weights(cu(wt), None, 0.5, False, want_f16=True)
    Y, dbg = B.linear(q, cu(xt), debug=True)
    r = OW.w8a8_linear(x, OW.prepare_weights(wt.float().numpy(), None, smooth=False), out="bf16")
    sums = np.abs(r["xq"].astype(np.int64)).sum(axis=1)
    assert np.all(127 * sums[lo:hi] > 2 ** 24) and np.all(127 * np.delete(sums, np.s_[lo:hi]) <= 2 ** 24)
    acc = dbg["acc"].cpu().numpy().astype(np.int64)
    assert acc[lo, 0] == 127 * 127 * K
    assert np.array_equal(acc, r["acc"])
    assert np.array_equal(f32_of_bf16(Y), r["y"])


WIDE_FEW_SHAPES = [
    (7, 8208, 1040),     # ragged N (8208 = 64 x 128 + 16) and K (an odd number of 64-k steps)
    (20, 8192, 1152),    # with a bias
    (32, 13824, 1152),   # the gate/up shape at a decode batch of 32
]


@pytest.mark.parametrize("M,N,K", WIDE_FEW_SHAPES)
def test_w8a8_wide_output_few_tokens_bit_exact(B, M, N, K):
    """5-32 tokens on wide outputs with the INT8 codes only (no fp16 copy): the streaming kernel;
    codes, scales, INT32 sums and outputs bit for bit."""
    x32, x, w32, w, c32, c = _case(M, N, K, seed=M * 11 + N)
    stat = OW.act_absmax(np.concatenate([c32, x32]))
    q = B.prepare_weights(cu(w), cu(torch.from_numpy(stat)))  # INT8 codes only: no fp16 copy
    bias = np.random.default_rng(3).standard_normal(N).astype(np.float32) if M == 20 else None
    Y, dbg = B.linear(q, cu(x), bias=cu(torch.from_numpy(bias)) if bias is not None else None, debug=True)
    r = OW.w8a8_linear(x32, OW.prepare_weights(w32, stat), bias=bias, out="bf16")
    assert np.array_equal(dbg["xq"].cpu().numpy(), r["xq"])
    assert np.array_equal(dbg["s_x"].cpu().numpy(), r["s_x"])
    assert np.array_equal(dbg["acc"].cpu().numpy().astype(np.int64), r["acc"])
    assert np.array_equal(f32_of_bf16(Y), r["y"])


def test_w8a8_wide_output_few_tokens_at_extremes(B):
    """Rows of +-1 (every code +-127) at 12 tokens on a wide output, K = 2048: acc[0, 0] = 127^2 K
    exceeds 2^24, so the fp32 MMA sums of the streaming kernel must be folded into INT32 to come
    out exact."""
    M, N, K = 12, 8192, 2048
    g = np.random.default_rng(5)
    x = np.where(g.random((M, K)) < 0.5, -1.0, 1.0).astype(np.float32)
    w = np.where(g.random((N, K)) < 0.5, -0.5, 0.5).astype(np.float32)
    w[0] = np.sign(x[0]) * 0.5
    xt, wt = torch.from_numpy(x).to(torch.bfloat16), torch.from_numpy(w).to(torch.bfloat16)
    q = B.prepare_weights(cu(wt), None, 0.5, False)
    Y, dbg = B.linear(q, cu(xt), debug=True)
    r = OW.w8a8_linear(xt.float().numpy(), OW.prepare_weights(wt.float().numpy(), None, smooth=False), out="bf16")
    acc = dbg["acc"].cpu().numpy().astype(np.int64)
    assert acc[0, 0] == 127 * 127 * K > 2 ** 24
    assert np.array_equal(acc, r["acc"])
    assert np.array_equal(f32_of_bf16(Y), r["y"])


# ---------------------------------------------------------------------- bf16 pass-through
def _bf16_close(y_gpu: np.ndarray, X: np.ndarray, W: np.ndarray, y_ref: np.ndarray):
    K = X.shape[1]
    mag = np.abs(X).astype(np.float64) @ np.abs(W).astype(np.float64).T
    ulp = np.spacing(np.abs(y_ref).astype(np.float32)) * 2 ** 16  # bf16 ulp = 2^16 fp32 ulps
    bound = ulp + K * 2.0 ** -24 * mag + 1e-30
    assert np.all(np.abs(y_gpu.astype(np.float64) - y_ref) <= bound)


@pytest.mark.parametrize("M,N,K", [(1, 6912, 1152), (16, 6912, 1152), (5, 1152, 6912), (40, 300, 1040),
                                   (1, 1536, 1152), (8, 1152, 6912), (3, 40, 64), (2, 13824, 1152),
                                   (128, 6912, 1152), (70, 1152, 6912), (300, 256, 64),
                                   (6, 1536, 1152),      # 8 token slots on the tensor cores, with a bias
                                   (13, 1536, 1152),     # 16 token slots on the tensor cores
                                   (7, 200, 64),         # the same, ragged rows, one 64-column box of K
                                   (8, 13824, 1152),     # the same, 48 rows per CTA
                                   (32, 1152, 4608),     # split-K: 18 tiles, k cut into 8 parts
                                   (200, 1152, 6912),    # split-K over two row blocks
                                   (300, 19472, 1152),   # CTA pairs on 256 x 192 tiles, ragged M and N
                                   (1024, 13824, 1152)])  # CTA pairs on 256 x 256 tiles
def test_bf16_linear_within_tolerance(B, M, N, K):
    x32, x, w32, w, _, _ = _case(M, N, K, seed=11 + M)
    bias = np.random.default_rng(3).standard_normal(N).astype(np.float32) if M in (6, 32) else None
    Y = B.linear_bf16(cu(w), cu(x), bias=cu(torch.from_numpy(bias)) if bias is not None else None)
    ref = OW.bf16_linear(x32, w32, bias=bias, out="bf16")
    _bf16_close(f32_of_bf16(Y), x32, w32, ref)
