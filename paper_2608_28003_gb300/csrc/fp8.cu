// The FP8 (e4m3) variant of the W8A8 linear and of the FFN block (the paper's Future Work: FP8 in
// place of INT8 on Blackwell).  The SmoothQuant structure of the INT8 path is kept (Eq. delta-attn,
// what-lmhead, xhat-lmhead), with e4m3 codes in place of the integers: s_w = max|W_hat| / 448,
// s_x = max|x_hat| / 448, codes = e4m3(v * fl32(448 / max)), nearest even, saturating; the GEMM sums
// the code products in fp32 (not exact: a sum of e4m3 products needs up to 49 bits) and the
// epilogue dequantises y = fl32(fl32(s_x s_w) * acc) (+ bias), the order of Eq. gemm-final.
//
// Routing: 1-8 tokens run the row-owning decode GEMV on its tensor-core path (e4m3 weights and
// codes widened to fp16, K1 fused); more tokens run the per-token quantiser, then the tcgen05 GEMM
// with kind::f8f6f4 on the one-byte codes (no wider copy of the weights exists or is needed).
#include "common.cuh"
#include "gemm_tc.cuh"
#include "gemv_small.cuh"
#include "ops.cuh"
#include "stream_gemm.cuh"

namespace w8a8 {

namespace {

w8a8_status check_fp8_weight(const char* who, const w8a8_fp8_weight* w) {
  W8A8_CHECK_ARG(w != nullptr, W8A8_ERR_INVALID_ARG, "%s: null weight descriptor", who);
  W8A8_CHECK_ARG(w->n > 0 && w->k > 0, W8A8_ERR_SHAPE, "%s: weight shape [%d, %d] must be positive", who, w->n, w->k);
  W8A8_CHECK_ARG(w->k % 16 == 0 && w->k <= W8A8_MAX_K && w->n % 16 == 0, W8A8_ERR_SHAPE,
                 "%s: N=%d and K=%d must be multiples of 16 (K <= %d)", who, w->n, w->k, W8A8_MAX_K);
  W8A8_CHECK_ARG(w->wq && w->s_w && w->inv_delta, W8A8_ERR_INVALID_ARG, "%s: null weight pointer", who);
  W8A8_CHECK_ARG(aligned16(w->wq) && aligned16(w->s_w) && aligned16(w->inv_delta), W8A8_ERR_ALIGN,
                 "%s: weight pointers must be 16-byte aligned", who);
  return W8A8_OK;
}

// One FP8 linear.  `ws` holds the reserved counters and error word; `scratch` is where the
// linear's scratch regions start (LinearWs offsets minus the reserved bytes).
w8a8_status run_fp8_linear(const w8a8_fp8_weight* w, const uint16_t* X, int M, const float* bias, int kind,
                           uint16_t* Y, uint8_t* xq_dbg, float* s_x_dbg, void* ws, char* scratch, int sms,
                           cudaStream_t st) {
  const int N = w->n, K = w->k;
  SmallArgs s{};
  s.p = make_small_plan(SMALL_FP8, M, N, K, kind, sms, false);
  if (s.p.ok) {
    s.W = w->wq;
    s.X = X;
    s.M = M;
    s.N = N;
    s.K = K;
    s.kind = kind;
    s.inv_delta = w->inv_delta;
    s.s_w = w->s_w;
    s.bias = bias;
    s.y = Y;
    s.xq_dbg = reinterpret_cast<int8_t*>(xq_dbg);
    s.s_x_dbg = s_x_dbg;
    s.err = reinterpret_cast<unsigned int*>(reinterpret_cast<char*>(ws) + kErrWordOffset);
    return launch_small_gemv(SMALL_FP8, s, st);
  }
  W8A8_CHECK_ARG(tc_gemm_supported(M, N, K, kind, false, 0), W8A8_ERR_SHAPE,
                 "fp8 linear: no kernel takes M=%d N=%d K=%d", M, N, K);
  const LinearWs L = linear_ws(M, N, K, true, sms);
  uint8_t* codes = reinterpret_cast<uint8_t*>(scratch + (L.xf16 - W8A8_WS_RESERVED));
  float* s_x = reinterpret_cast<float*>(scratch + (L.sx - W8A8_WS_RESERVED));
  W8A8_TRY(launch_quantize_rows_fp8(X, M, K, w->inv_delta, codes, s_x, st));
  if (xq_dbg) W8A8_CUDA(cudaMemcpyAsync(xq_dbg, codes, (size_t)M * K, cudaMemcpyDeviceToDevice, st));
  if (s_x_dbg) W8A8_CUDA(cudaMemcpyAsync(s_x_dbg, s_x, sizeof(float) * M, cudaMemcpyDeviceToDevice, st));
  TcArgs a{};
  a.A = codes;
  a.B = w->wq;
  a.M = M;
  a.N = N;
  a.K = K;
  a.kind = kind;
  a.s_x = s_x;
  a.s_w = w->s_w;
  a.bias = bias;
  a.y = Y;
  StreamArgs r{};
  attach_reserved(r, ws);
  a.grid_counter = r.grid_counter;
  a.top_keys = r.top_keys;
  a.err = r.err;
  a.partials = scratch + (L.part - W8A8_WS_RESERVED);
  a.tile_counters = r.tile_counters;
  return launch_tc_gemm(TC_FP8, a, st);
}

w8a8_status check_ws_fp8(const char* who, void* ws, size_t have, size_t need) {
  W8A8_CHECK_ARG(ws != nullptr && have >= need, W8A8_ERR_WORKSPACE, "%s: workspace %zu bytes, need %zu", who,
                 ws ? have : 0, need);
  W8A8_CHECK_ARG(aligned16(ws), W8A8_ERR_ALIGN, "%s: workspace must be 16-byte aligned", who);
  return W8A8_OK;
}

}  // namespace

}  // namespace w8a8

using namespace w8a8;

extern "C" w8a8_status w8a8_fp8_linear(const w8a8_fp8_weight* w, const uint16_t* X, int M, const float* bias,
                                       uint16_t* Y, uint8_t* xq_dbg, float* s_x_dbg, void* workspace, size_t ws_bytes,
                                       void* stream) {
  W8A8_TRY(check_fp8_weight("w8a8_fp8_linear", w));
  W8A8_CHECK_ARG(M >= 0, W8A8_ERR_INVALID_ARG, "w8a8_fp8_linear: M=%d is negative", M);
  if (M == 0) return W8A8_OK;
  W8A8_CHECK_ARG(X && Y, W8A8_ERR_INVALID_ARG, "w8a8_fp8_linear: null X or Y");
  W8A8_CHECK_ARG(aligned16(X) && aligned16(Y) && (!bias || aligned16(bias)) && (!xq_dbg || aligned16(xq_dbg)) &&
                     (!s_x_dbg || aligned16(s_x_dbg)),
                 W8A8_ERR_ALIGN, "w8a8_fp8_linear: pointers must be 16-byte aligned");
  DevInfo d;
  W8A8_TRY(dev_info(&d));
  W8A8_TRY(check_ws_fp8("w8a8_fp8_linear", workspace, ws_bytes, linear_ws(M, w->n, w->k, true, d.sms).total));
  return run_fp8_linear(w, X, M, bias, EPI_BF16, Y, xq_dbg, s_x_dbg, workspace,
                        reinterpret_cast<char*>(workspace) + W8A8_WS_RESERVED, d.sms, as_stream(stream));
}

extern "C" w8a8_status w8a8_fp8_ffn_block(const w8a8_fp8_ffn_weights* f, const uint16_t* X, int M, uint16_t* Y,
                                          uint16_t* h_dbg, void* workspace, size_t ws_bytes, void* stream) {
  W8A8_CHECK_ARG(f != nullptr, W8A8_ERR_INVALID_ARG, "w8a8_fp8_ffn_block: null FFN descriptor");
  const int H = f->hidden, F = f->inter;
  W8A8_CHECK_ARG(H > 0 && F > 0 && H % 16 == 0 && F % 16 == 0 && H <= W8A8_MAX_K && F <= W8A8_MAX_K, W8A8_ERR_SHAPE,
                 "w8a8_fp8_ffn_block: hidden=%d inter=%d must be positive multiples of 16", H, F);
  W8A8_TRY(check_fp8_weight("w8a8_fp8_ffn_block(gate_up)", &f->gate_up));
  W8A8_TRY(check_fp8_weight("w8a8_fp8_ffn_block(down)", &f->down));
  W8A8_CHECK_ARG(f->gate_up.n == 2 * F && f->gate_up.k == H && f->down.n == H && f->down.k == F, W8A8_ERR_SHAPE,
                 "w8a8_fp8_ffn_block: weight shapes do not match hidden=%d inter=%d", H, F);
  W8A8_CHECK_ARG(M >= 0, W8A8_ERR_INVALID_ARG, "w8a8_fp8_ffn_block: M=%d is negative", M);
  if (M == 0) return W8A8_OK;
  W8A8_CHECK_ARG(X && Y, W8A8_ERR_INVALID_ARG, "w8a8_fp8_ffn_block: null X or Y");
  W8A8_CHECK_ARG(aligned16(X) && aligned16(Y) && (!h_dbg || aligned16(h_dbg)), W8A8_ERR_ALIGN,
                 "w8a8_fp8_ffn_block: X, Y, h must be 16-byte aligned");
  DevInfo d;
  W8A8_TRY(dev_info(&d));
  const FfnWs L = ffn_ws(M, H, F, d.sms);
  W8A8_TRY(check_ws_fp8("w8a8_fp8_ffn_block", workspace, ws_bytes, L.total));
  char* base = reinterpret_cast<char*>(workspace);
  uint16_t* h = h_dbg ? h_dbg : reinterpret_cast<uint16_t*>(base + L.h);
  cudaStream_t st = as_stream(stream);
  // gate/up with the GeGLU epilogue into h, then down; disjoint scratch, shared reserved counters
  W8A8_TRY(run_fp8_linear(&f->gate_up, X, M, nullptr, EPI_GEGLU, h, nullptr, nullptr, workspace, base + L.gu, d.sms,
                          st));
  return run_fp8_linear(&f->down, h, M, nullptr, EPI_BF16, Y, nullptr, nullptr, workspace, base + L.dn, d.sms, st);
}
