"""CPU checks of the decode GEMV's launch plan (host logic, no GPU): for every decoder linear at 1-16
tokens, in every weight kind, a plan that takes the shape covers it, fits the shared memory of the
CTAs it puts on an SM, keeps its weight ring double-buffered (or holds the whole stream) and picks
16 consumer warps only where its rules allow; the decoder's own shapes land where the kernel
design puts them."""
import pytest

SMEM_PER_SM = 227 * 1024   # shared memory a CTA may use on GB300
STATIC_SMEM = 2048         # the kernel's static shared memory (reduction slots, scales) and slack
SMS = 152

# the Gemma-3-1B-shaped decoder's linears: (N, K, GeGLU epilogue, residual step fusable)
SHAPES = {
    "qkv": (1536, 1152, False, True),
    "o": (1152, 1024, False, False),
    "gate_up": (13824, 1152, True, True),
    "down": (1152, 6912, False, False),
}


@pytest.fixture(scope="module")
def B():
    from paper_2608_28003_gb300 import build
    build.build()
    from paper_2608_28003_gb300 import binding
    return binding


def plans(B):
    for kind in ("bf16", "int8", "fp8"):
        for name, (N, K, geglu, fusable) in SHAPES.items():
            for M in range(1, 17):
                for fused in ((False, True) if fusable else (False,)):
                    yield kind, name, M, N, K, geglu, fused, B.decode_gemv_plan(kind, M, N, K, geglu, fused, SMS)


def test_every_plan_covers_its_shape_and_fits(B):
    taken = 0
    for kind, name, M, N, K, geglu, fused, p in plans(B):
        what = (kind, name, M, fused)
        if not p["taken"]:
            assert all(v == 0 for v in p.values()), what
            continue
        taken += 1
        assert p["slots"] in (1, 2, 4, 8, 16) and p["slots"] >= M, what
        assert p["slots"] == 1 or p["slots"] // 2 < M or (kind == "fp8" and p["slots"] == 8), what
        R = 8 * p["rows_per_warp"]
        assert p["ctas"] == -(-N // R), what                       # every output row, once
        assert p["ctas_per_sm"] == (2 if p["ctas"] > SMS else 1), what
        sub = 256 if kind == "bf16" else 512                      # k elements per 512-byte row slice
        assert p["subslices"] == -(-K // sub) and p["kpad"] == p["subslices"] * sub >= K, what
        assert p["subslices_per_stage"] in (1, 2, 4), what
        assert p["steps"] == -(-p["subslices"] // p["subslices_per_stage"]), what
        assert p["stage_bytes"] == p["subslices_per_stage"] * R * 512, what
        assert min(p["steps"], 2) <= p["stages"] <= min(16, p["steps"]), what
        assert p["smem_bytes"] == (1024 + p["stages"] * p["stage_bytes"] + p["x_bytes"] + p["resid_bytes"]
                                   + p["partial_bytes"] + 16 * p["stages"]), what
        assert p["ctas_per_sm"] * (p["smem_bytes"] + STATIC_SMEM) <= SMEM_PER_SM, what
        if geglu:
            assert p["rows_per_warp"] % 2 == 0, what                # gate and up rows in pairs
        if fused:
            assert M <= 8 and K <= 2048, what                       # one 8-channel vector per thread
        mma = p["slots"] >= 8
        assert (p["partial_bytes"] > 0) == mma, what
        sixteen = mma and p["rows_per_warp"] == 1 and p["ctas"] <= SMS and not fused
        assert p["consumer_warps"] == (16 if sixteen else 8), what
        if mma:
            assert p["partial_bytes"] == p["consumer_warps"] * R * p["slots"] * 4, what
    assert taken > 150  # of the 288 shape, token-count and fusion combinations


def test_decoder_shapes_route_as_designed(B):
    P = lambda *a, **k: B.decode_gemv_plan(*a, sms=SMS, **k)  # noqa: E731
    # one token: q/k/v with the residual step fused, 8 rows per CTA on 192 CTAs
    p = P("bf16", 1, 1536, 1152, fused_norm=True)
    assert (p["taken"], p["slots"], p["rows_per_warp"], p["ctas"], p["consumer_warps"]) == (1, 1, 1, 192, 8)
    # gate/up + GeGLU: 48 rows per CTA (three gate/up pairs per warp), two CTAs per SM
    for kind in ("bf16", "int8"):
        p = P(kind, 1, 13824, 1152, geglu=True, fused_norm=True)
        assert (p["rows_per_warp"], p["ctas"], p["ctas_per_sm"]) == (6, 288, 2)
    # down and o: one CTA per SM; 16 consumer warps on the tensor-core paths (5-8 tokens)
    for M, warps in ((1, 8), (4, 8), (8, 16)):
        p = P("int8", M, 1152, 6912)
        assert (p["taken"], p["ctas"], p["consumer_warps"]) == (1, 144, warps), M
    # the residual step is fused at 1-8 tokens only; K = 6912 rows of 16 token slots do not fit
    assert not P("bf16", 9, 1536, 1152, fused_norm=True)["taken"]
    assert P("bf16", 9, 1536, 1152)["taken"]
    assert not P("bf16", 16, 1152, 6912)["taken"]
    assert not P("int8", 16, 1152, 6912)["taken"]
    # e4m3 codes: fp32 FMAs at 1-2 tokens, the 8-slot tensor-core path from 3
    assert P("fp8", 2, 1152, 1024)["slots"] == 2
    assert P("fp8", 3, 1152, 1024)["slots"] == 8


def test_plan_rejects_bad_arguments(B):
    with pytest.raises(B.W8A8Error):
        B.decode_gemv_plan("bf16", 1, 1152, 1024, sms=0)
    out = (B.ctypes.c_int32 * len(B.PLAN_FIELDS))()
    assert B.lib().w8a8_decode_gemv_plan(3, 1, 1152, 1024, 0, 0, SMS, out) != 0  # weight kind out of range
    assert B.lib().w8a8_decode_gemv_plan(0, 1, 1152, 1024, 0, 0, SMS, None) != 0


STREAM_STATIC = 8192  # the streaming kernel's static shared memory (barrier flags, top-1 keys)


def test_stream_plan_covers_its_shape_and_fits(B):
    """The persistent weight-streaming kernel (lm_head-sized outputs, 1-63 tokens): its token
    groups, 128-row groups and k chunks cover the call, every CTA has a unit, the grid holds at
    most its CTAs per SM on every SM, the ring fits beside them, and whole row groups per CTA
    (no partial tiles) use the widest k chunk."""
    for int8 in (True, False):
        for N in (262144, 13824, 1152):
            for K in (1152, 6912):
                for M in range(1, 64):
                    p = B.stream_gemm_plan(int8, M, N, K, SMS)
                    what = (int8, N, K, M)
                    dp4a = int8 and M <= 4 and 4 * K <= 32768
                    assert p["dp4a"] == int(dp4a), what
                    if dp4a:
                        assert p["slots"] in (1, 2, 4) and p["slots"] >= M and p["slots"] // 2 < M, what
                        assert p["tokens_per_group"] == p["slots"] and p["token_groups"] == 1, what
                        assert p["ctas_per_sm"] == 2, what
                    else:
                        nb = 1 if M <= 8 else 2 if M <= 16 else 4 if M <= 32 else 8
                        assert p["blocks"] == nb and p["tokens_per_group"] == 8 * nb, what
                        assert p["token_groups"] == -(-M // (8 * nb)), what
                        assert p["ctas_per_sm"] == (2 if nb <= 4 else 1), what
                    assert p["row_groups"] == -(-N // 128), what
                    assert p["k_chunks"] == -(-K // p["kc"]) and p["k_chunks"] * p["kc"] >= K, what
                    units = p["token_groups"] * p["row_groups"] * p["k_chunks"]
                    assert 1 <= p["ctas"] <= min(units, p["ctas_per_sm"] * SMS, 8192), what
                    assert p["whole"] == int(p["token_groups"] * p["row_groups"] >= p["ctas"]), what
                    if p["whole"]:
                        assert p["kc"] == (256 if int8 else 128), what
                    assert 2 <= p["stages"] <= 8, what
                    assert p["ctas_per_sm"] * (p["smem_bytes"] + STREAM_STATIC) <= SMEM_PER_SM, what
                    assert p["partial_bytes"] == p["ctas"] * 2 * 128 * p["tokens_per_group"] * 4, what


def test_lm_head_routes_as_designed(B):
    # one token: the dp4a GEMV, two CTAs per SM over 2048 whole 128-row groups
    p = B.stream_gemm_plan(True, 1, 262144, 1152, SMS)
    assert (p["dp4a"], p["ctas"], p["ctas_per_sm"], p["whole"]) == (1, 2 * SMS, 2, 1)
    # 5-32 tokens: the MMA streaming kernel with two CTAs per SM; from 33, one
    for M, cps in ((5, 2), (16, 2), (32, 2), (33, 1), (63, 1)):
        p = B.stream_gemm_plan(True, M, 262144, 1152, SMS)
        assert (p["dp4a"], p["ctas_per_sm"], p["ctas"]) == (0, cps, cps * SMS), M
    with pytest.raises(B.W8A8Error):
        B.stream_gemm_plan(True, 0, 262144, 1152, SMS)


def test_tc_gemm_choice_rules(B):
    """The tcgen05 GEMM's tile choice over a grid of shapes: a k split only on single-CTA tiles of a
    bf16-output call that has its partials, at least four parts, one unit per SM at most, and each
    part at least two stages of k; pairs only on 256-token tiles."""
    for mode in ("bf16", "int8", "fp8"):
        for kind in ("bf16", "geglu", "f32"):
            for split_ok in (False, True):
                for M in (1, 8, 16, 32, 64, 128, 256, 300, 512, 2048):
                    for N in (1152, 1536, 6912, 13824, 262144):
                        for K in (1024, 1152, 6912):
                            pair, bn, ks = B.tc_gemm_plan(mode, M, N, K, kind, split_ok, SMS)
                            what = (mode, kind, split_ok, M, N, K)
                            assert (pair, bn) in ((1, 256), (1, 192), (1, 128), (0, 128), (0, 64)), what
                            if pair == 1 and bn == 128:
                                assert mode == "int8", what      # the narrow pair tile is W8A8's
                            if ks > 1:
                                assert not pair and kind == "bf16" and split_ok, what
                                tiles = -(-N // bn) * -(-M // 128)
                                bk = 128 if mode == "fp8" else 64  # k elements per 128-byte stage row
                                assert ks >= 4 and ks * tiles <= SMS and 2 * ks <= -(-K // bk), what
                                assert 2 * tiles <= SMS, what
                            else:
                                assert ks == 1, what


def test_tc_gemm_routes_decoder_shapes_as_designed(B):
    P = lambda *a, **k: B.tc_gemm_plan(*a, sms=SMS, **k)  # noqa: E731
    # 2048-token prefill: gate/up on 256 x 256 pair tiles in every mode; W8A8 down on 256 x 128 pairs
    for mode in ("bf16", "int8", "fp8"):
        assert P(mode, 2048, 13824, 1152, "geglu") == (1, 256, 1)
    assert P("int8", 2048, 1152, 6912) == (1, 128, 1)
    assert P("bf16", 2048, 1152, 6912) == (0, 128, 1)
    # 512 tokens: the down projection on split 128-column tiles (four parts), bf16 and W8A8
    assert P("bf16", 512, 1152, 6912) == (0, 128, 4) == P("int8", 512, 1152, 6912)
    # decode batches: q/k/v, o and down at 32 tokens split over 6-8 parts of 64-column tiles
    assert P("bf16", 32, 1536, 1152) == (0, 64, 6)
    assert P("bf16", 32, 1152, 1024) == (0, 64, 8)
    assert P("bf16", 32, 1152, 6912) == (0, 64, 8)
    # without the partials' workspace, no split
    assert P("bf16", 32, 1152, 6912, split_ok=False) == (0, 64, 1)
    # fp32 logits (lm_head) never split
    assert P("bf16", 64, 262144, 1152, "f32")[2] == 1
    with pytest.raises(B.W8A8Error):
        P("bf16", 32, 1152, 1000)  # K not a multiple of 16


RESERVED = 65536  # W8A8_WS_RESERVED: the split-K and top-1 counters at the start of a workspace


def _ceil(x, a=256):
    return -(-x // a) * a


def test_workspace_sizes_cover_every_region(B):
    """The workspace a caller allocates from the size queries holds the reserved counters, the
    activation codes and scales, and the larger of the two kernels' partial sums (the streaming
    kernel's plan, the tcgen05 GEMM's k split: one unit per SM at most); the FFN block's holds h and
    both linears' regions and the row-maxima hand-off.  Sizes grow with the token count."""
    for N, K in ((1536, 1152), (1152, 1024), (13824, 1152), (1152, 6912), (262144, 1152)):
        prev = prev_bf = 0
        for M in (1, 2, 4, 5, 8, 9, 16, 33, 64, 128, 300, 512, 2048):
            total = B._size("w8a8_linear_workspace_size", M, N, K)
            rows = M if M >= 128 else -(-M // 8) * 8
            parts = max(B.stream_gemm_plan(True, M, N, K, SMS)["partial_bytes"], SMS * 128 * min(rows, 128) * 4)
            assert total == RESERVED + _ceil(2 * M * K) + _ceil(8 * M) + _ceil(parts), (M, N, K)
            assert total % 256 == 0 and total >= prev
            prev = total
            bf = B._size("w8a8_linear_bf16_workspace_size", M, N, K)
            parts_bf = max(B.stream_gemm_plan(False, M, N, K, SMS)["partial_bytes"], SMS * 128 * min(rows, 128) * 4)
            assert bf == RESERVED + _ceil(parts_bf) and bf >= prev_bf, (M, N, K)
            prev_bf = bf
    for M in (1, 8, 16, 64, 512, 2048):
        H, F = 1152, 6912
        ffn = B._size("w8a8_ffn_workspace_size", M, H, F)
        gu = B._size("w8a8_linear_workspace_size", M, 2 * F, H) - RESERVED
        dn = B._size("w8a8_linear_workspace_size", M, H, F) - RESERVED
        assert ffn == RESERVED + _ceil(2 * M * F) + gu + dn + _ceil(2 * SMS * 16 * 4), M
        assert B._size("w8a8_lm_head_workspace_size", M, 262144, H) == B._size("w8a8_linear_workspace_size", M, 262144, H)
