// C-ABI entry points of libw8a8: argument checks, workspace carve-up and kernel dispatch for the
// W8A8 linear, the bf16 pass-through linear, the FFN block and lm_head.
#include <cstdarg>
#include <cstdio>
#include <mutex>

#include "common.cuh"
#include "gemm_tc.cuh"
#include "gemv_small.cuh"
#include "ops.cuh"
#include "stream_gemm.cuh"

namespace w8a8 {

static thread_local char g_err[512] = "";

void set_error(const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
}
const char* get_error() { return g_err; }

static DevInfo g_dev[64];
static std::mutex g_dev_mu;

w8a8_status dev_info(DevInfo* out) {
  int dev = 0;
  W8A8_CUDA(cudaGetDevice(&dev));
  W8A8_CHECK_ARG(dev >= 0 && dev < 64, W8A8_ERR_UNSUPPORTED, "device ordinal %d out of range", dev);
  std::lock_guard<std::mutex> lk(g_dev_mu);
  DevInfo& d = g_dev[dev];
  if (d.ok < 0) {
    int major = 0, minor = 0, sms = 0;
    W8A8_CUDA(cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev));
    W8A8_CUDA(cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev));
    W8A8_CUDA(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
    d.ok = (major == 10 && minor == 3) ? 1 : 0;
    d.sms = sms;
  }
  W8A8_CHECK_ARG(d.ok == 1, W8A8_ERR_UNSUPPORTED, "libw8a8 is built for sm_103 (GB300) only");
  *out = d;
  return W8A8_OK;
}

w8a8_status check_device() {
  DevInfo d;
  return dev_info(&d);
}

int device_sms() {
  DevInfo d;
  return dev_info(&d) == W8A8_OK ? d.sms : 152;
}

// ------------------------------------------------------------------------ workspace plans
// Layout: [reserved counters | x codes [M,K] | s_x [M], sums of |codes| [M] | partials]

LinearWs linear_ws(int M, int N, int K, bool int8_path, int sms) {
  LinearWs w{};
  size_t off = W8A8_WS_RESERVED;
  w.xf16 = off;
  if (int8_path) off += round_up((size_t)M * K * 2, 256);
  w.sx = off;
  if (int8_path) off += round_up((size_t)M * 8, 256);
  w.part = off;
  off += round_up(std::max(make_stream_plan(int8_path, M, N, K, sms).partial_bytes, tc_split_partial_bytes(M, sms)), 256);
  w.total = off;
  return w;
}

static w8a8_status check_qweight(const char* who, const w8a8_qweight* w) {
  W8A8_CHECK_ARG(w != nullptr, W8A8_ERR_INVALID_ARG, "%s: null weight descriptor", who);
  W8A8_CHECK_ARG(w->n > 0 && w->k > 0, W8A8_ERR_SHAPE, "%s: weight shape [%d, %d] must be positive", who, w->n, w->k);
  W8A8_CHECK_ARG(w->k % 16 == 0 && w->k <= W8A8_MAX_K, W8A8_ERR_SHAPE, "%s: K=%d must be a multiple of 16 and <= %d",
                 who, w->k, W8A8_MAX_K);
  W8A8_CHECK_ARG(w->wq && w->s_w && w->inv_delta, W8A8_ERR_INVALID_ARG, "%s: null weight pointer", who);
  W8A8_CHECK_ARG(aligned16(w->wq) && aligned16(w->s_w) && aligned16(w->inv_delta) && (!w->wq_f16 || aligned16(w->wq_f16)),
                 W8A8_ERR_ALIGN, "%s: weight pointers must be 16-byte aligned", who);
  return W8A8_OK;
}

static w8a8_status check_ws(const char* who, void* ws, size_t have, size_t need) {
  W8A8_CHECK_ARG(ws != nullptr && have >= need, W8A8_ERR_WORKSPACE, "%s: workspace %zu bytes, need %zu", who,
                 ws ? have : 0, need);
  W8A8_CHECK_ARG(aligned16(ws), W8A8_ERR_ALIGN, "%s: workspace must be 16-byte aligned", who);
  return W8A8_OK;
}


// Per-token quantiser for a W8A8 GEMM plan: INT8 codes for the dp4a GEMV, fp16 codes for the MMA
// kernel, written to `codes` (workspace); `xq_dbg` (nullable) also receives the INT8 codes.
static w8a8_status quantize_for(const StreamPlan& p, const uint16_t* X, int M, int K, const float* inv_delta,
                                void* codes, int8_t* xq_dbg, float* s_x, cudaStream_t st) {
  if (p.dp4a) {
    W8A8_TRY(launch_quantize_rows(X, M, K, inv_delta, reinterpret_cast<int8_t*>(codes), nullptr, s_x, st));
    if (xq_dbg) W8A8_CUDA(cudaMemcpyAsync(xq_dbg, codes, (size_t)M * K, cudaMemcpyDeviceToDevice, st));
    return W8A8_OK;
  }
  return launch_quantize_rows(X, M, K, inv_delta, xq_dbg, reinterpret_cast<uint16_t*>(codes), s_x, st);
}

static unsigned int* err_word(void* ws) {
  return reinterpret_cast<unsigned int*>(reinterpret_cast<char*>(ws) + kErrWordOffset);
}

// Decode-sized calls whose CTAs can own whole weight rows go to the row-owning GEMV (K1 fused
// into it on the W8A8 path); returns false when the shape is left to the streaming kernel.
// Partial row maxima passed from the FFN's gate/up launch to its down launch (see SmallArgs).
struct RowMax {
  float* out;                   // gate/up: [P][MT]
  const float* next_inv_delta;  // gate/up: down's 1 / delta
  const float* in;              // down: gate/up's rows
  int n;                        // down: gate/up's CTA count
};

static bool small_gemv(bool int8, const void* W, const float* inv_delta, const float* s_w, const uint16_t* X, int M,
                       int N, int K, const float* bias, int kind, uint16_t* Y, const w8a8_debug* dbg, void* ws,
                       const ResNorm* rn, int sms, cudaStream_t st, w8a8_status* status, const RowMax* rm = nullptr) {
  if (kind != EPI_BF16 && kind != EPI_GEGLU) return false;
  SmallArgs a{};
  a.p = make_small_plan(int8, M, N, K, kind, sms, rn != nullptr);
  if (!a.p.ok) return false;
  if (rm) {
    a.rowmax_out = rm->out;
    a.next_inv_delta = rm->next_inv_delta;
    a.rowmax_in = rm->in;
    a.rowmax_n = rm->n;
  }
  if (rn) {
    a.has_rn = 1;
    a.rn = *rn;
  }
  a.W = W;
  a.X = X;
  a.M = M;
  a.N = N;
  a.K = K;
  a.kind = kind;
  a.inv_delta = inv_delta;
  a.s_w = s_w;
  a.bias = bias;
  a.y = Y;
  a.xq_dbg = dbg ? dbg->xq : nullptr;
  a.s_x_dbg = dbg ? dbg->s_x : nullptr;
  a.acc_dbg = dbg ? dbg->acc : nullptr;
  a.err = err_word(ws);
  *status = launch_small_gemv(int8, a, st);
  return true;
}

bool decode_gemv_takes(bool int8, int M, int N, int K, bool geglu, int sms) {
  return make_small_plan(int8, M, N, K, geglu ? EPI_GEGLU : EPI_BF16, sms, true).ok != 0;
}

// Calls with more tokens than the decode GEMV takes go to the tensor-core GEMM when its shape
// rules hold (W8A8: the weights' fp16 code copy must exist); false leaves them to the streaming
// kernel.  Below 64 tokens a 128-token tile is mostly padding; it still beats the streaming kernel
// on the decoder's linears (one wave of 128 x 64 tiles, measured 12-15 us against 20 us at M 16),
// but not on lm_head-sized outputs, where the streaming kernel's INT8 reads (half the bytes of the
// fp16 code copy) win.
constexpr int kTcMinTokens = 64, kTcMinTokensNarrow = 9, kTcNarrowMaxN = 16384;

static bool tc_path(bool int8, const void* W16, const uint16_t* X, int M, int N, int K, const float* bias, int kind,
                    const float* inv_delta, const float* s_w, uint16_t* Y, float* logits, int32_t* top1,
                    const w8a8_debug* dbg, void* ws, void* codes, float* s_x, void* part, cudaStream_t st,
                    w8a8_status* status, const PreCodes* pre = nullptr) {
  if (M < (N <= kTcNarrowMaxN ? kTcMinTokensNarrow : kTcMinTokens) || !W16 ||
      !tc_gemm_supported(M, N, K, kind, top1 != nullptr, max_top_keys()))
    return false;
  TcArgs a{};
  if (int8 && pre && pre->codes16 && !dbg) {  // the producer of X quantised it already
    a.A = pre->codes16;
    a.s_x = pre->s_x;
    a.qsum = pre->qsum;
    a.s_w = s_w;
  } else if (int8) {
    int* qsum = reinterpret_cast<int*>(s_x + M);  // beside s_x in the workspace
    w8a8_status q = launch_quantize_rows(X, M, K, inv_delta, dbg ? dbg->xq : nullptr,
                                         reinterpret_cast<uint16_t*>(codes), s_x, st, qsum);
    if (q == W8A8_OK && dbg && dbg->s_x)
      q = cudaMemcpyAsync(dbg->s_x, s_x, sizeof(float) * M, cudaMemcpyDeviceToDevice, st) == cudaSuccess
              ? W8A8_OK
              : W8A8_ERR_CUDA;
    if (q != W8A8_OK) {
      *status = q;
      return true;
    }
    a.A = codes;
    a.s_x = s_x;
    a.qsum = qsum;
    a.s_w = s_w;
    a.acc_dbg = dbg ? dbg->acc : nullptr;
  } else {
    a.A = X;
  }
  a.B = W16;
  a.M = M;
  a.N = N;
  a.K = K;
  a.kind = kind;
  a.bias = bias;
  a.y = Y;
  a.logits = logits;
  a.top1 = top1;
  StreamArgs r{};
  attach_reserved(r, ws);
  a.grid_counter = r.grid_counter;
  a.top_keys = r.top_keys;
  a.err = r.err;
  a.partials = part;
  a.tile_counters = r.tile_counters;
  *status = launch_tc_gemm(int8 ? TC_I8 : TC_BF16, a, st);
  return true;
}

// One W8A8 linear: K1 then the streaming GEMM.  s_x and the codes live in the workspace.
w8a8_status run_w8a8_linear(const w8a8_qweight* w, const uint16_t* X, int M, const float* bias, int kind,
                                   uint16_t* Y, float* logits, int32_t* top1, const w8a8_debug* dbg, void* ws,
                                   int sms, cudaStream_t st, const ResNorm* rn, const PreCodes* pre) {
  const int N = w->n, K = w->k;
  w8a8_status small_status = W8A8_OK;
  if (!logits && !top1 &&
      small_gemv(true, w->wq, w->inv_delta, w->s_w, X, M, N, K, bias, kind, Y, dbg, ws, rn, sms, st, &small_status))
    return small_status;
  W8A8_CHECK_ARG(!rn, W8A8_ERR_SHAPE, "fused residual norm: the decode GEMV does not take M=%d N=%d K=%d", M, N, K);
  LinearWs L = linear_ws(M, N, K, true, sms);
  char* base = reinterpret_cast<char*>(ws);
  void* codes = base + L.xf16;
  float* s_x = reinterpret_cast<float*>(base + L.sx);
  if (tc_path(true, w->wq_f16, X, M, N, K, bias, kind, w->inv_delta, w->s_w, Y, logits, top1, dbg, ws, codes, s_x,
              base + L.part, st, &small_status, pre))
    return small_status;
  StreamArgs a{};
  a.p = make_stream_plan(true, M, N, K, sms);
  W8A8_TRY(quantize_for(a.p, X, M, K, w->inv_delta, codes, dbg ? dbg->xq : nullptr, s_x, st));
  if (dbg && dbg->s_x) W8A8_CUDA(cudaMemcpyAsync(dbg->s_x, s_x, sizeof(float) * M, cudaMemcpyDeviceToDevice, st));
  a.W = w->wq;
  a.X = codes;
  a.M = M;
  a.N = N;
  a.K = K;
  a.kind = kind;
  a.s_x = s_x;
  a.s_w = w->s_w;
  a.bias = bias;
  a.y = Y;
  a.logits = logits;
  a.top1 = top1;
  a.acc_dbg = dbg ? dbg->acc : nullptr;
  a.partials = base + L.part;
  attach_reserved(a, ws);
  return launch_stream_gemm(true, a, st);
}

w8a8_status run_bf16_linear(const uint16_t* W, int N, int K, const uint16_t* X, int M, const float* bias,
                                   int kind, uint16_t* Y, float* logits, int32_t* top1, void* ws, int sms,
                                   cudaStream_t st, const ResNorm* rn) {
  w8a8_status small_status = W8A8_OK;
  if (!logits && !top1 &&
      small_gemv(false, W, nullptr, nullptr, X, M, N, K, bias, kind, Y, nullptr, ws, rn, sms, st, &small_status))
    return small_status;
  W8A8_CHECK_ARG(!rn, W8A8_ERR_SHAPE, "fused residual norm: the decode GEMV does not take M=%d N=%d K=%d", M, N, K);
  LinearWs L = linear_ws(M, N, K, false, sms);
  if (tc_path(false, W, X, M, N, K, bias, kind, nullptr, nullptr, Y, logits, top1, nullptr, ws, nullptr, nullptr,
              reinterpret_cast<char*>(ws) + L.part, st, &small_status))
    return small_status;
  StreamArgs a{};
  a.W = W;
  a.X = X;
  a.M = M;
  a.N = N;
  a.K = K;
  a.p = make_stream_plan(false, M, N, K, sms);
  a.kind = kind;
  a.bias = bias;
  a.y = Y;
  a.logits = logits;
  a.top1 = top1;
  a.partials = reinterpret_cast<char*>(ws) + L.part;
  attach_reserved(a, ws);
  return launch_stream_gemm(false, a, st);
}

// Internal: the W8A8 linear with its scratch at `scratch` (used by the no-allocation entry point).
size_t linear_scratch_bytes(int M, int N, int K, int sms) { return linear_ws(M, N, K, true, sms).total; }

w8a8_status linear_on_scratch(const w8a8_qweight* w, const uint16_t* X, int M, const float* bias, uint16_t* Y,
                              void* scratch, size_t scratch_bytes, cudaStream_t st) {
  DevInfo d;
  W8A8_TRY(dev_info(&d));
  W8A8_TRY(check_ws("w8a8_linear_noalloc", scratch, scratch_bytes, linear_ws(M, w->n, w->k, true, d.sms).total));
  return run_w8a8_linear(w, X, M, bias, EPI_BF16, Y, nullptr, nullptr, nullptr, scratch, d.sms, st);
}

w8a8_status check_linear_args(const char* who, const w8a8_qweight* w, const uint16_t* X, int M, const float* bias,
                              const uint16_t* Y) {
  W8A8_TRY(check_qweight(who, w));
  W8A8_CHECK_ARG(M >= 0, W8A8_ERR_INVALID_ARG, "%s: M=%d is negative", who, M);
  if (M == 0) return W8A8_OK;
  W8A8_CHECK_ARG(X && Y, W8A8_ERR_INVALID_ARG, "%s: null X or Y", who);
  W8A8_CHECK_ARG(aligned16(X) && aligned16(Y) && (!bias || aligned16(bias)), W8A8_ERR_ALIGN,
                 "%s: X, Y and bias must be 16-byte aligned", who);
  return W8A8_OK;
}

}  // namespace w8a8

using namespace w8a8;

extern "C" int w8a8_abi_version(void) { return 2; }

extern "C" w8a8_status w8a8_decode_gemv_plan(int weight_kind, int M, int N, int K, int geglu, int fused_norm, int sms,
                                             int* out) {
  W8A8_CHECK_ARG(out, W8A8_ERR_INVALID_ARG, "w8a8_decode_gemv_plan: null out");
  W8A8_CHECK_ARG(weight_kind >= SMALL_BF16 && weight_kind <= SMALL_FP8 && sms > 0, W8A8_ERR_INVALID_ARG,
                 "w8a8_decode_gemv_plan: weight kind %d or SM count %d out of range", weight_kind, sms);
  const SmallPlan p = make_small_plan(weight_kind, M, N, K, geglu ? EPI_GEGLU : EPI_BF16, sms, fused_norm != 0);
  const int v[W8A8_PLAN_FIELDS] = {p.ok,     p.MT,          p.RW,         p.P,          p.P > sms ? 2 : 1,
                                   p.cw,     p.ks,          p.nst,        p.stages,     p.stage_bytes,
                                   p.xbytes, p.abytes,      p.rbytes,     p.smem_bytes, p.kpad,
                                   p.nsub};
  for (int i = 0; i < W8A8_PLAN_FIELDS; ++i) out[i] = p.ok ? v[i] : 0;
  return W8A8_OK;
}

extern "C" w8a8_status w8a8_tc_gemm_plan(int mode, int M, int N, int K, int kind, int split_ok, int sms, int* out) {
  W8A8_CHECK_ARG(out, W8A8_ERR_INVALID_ARG, "w8a8_tc_gemm_plan: null out");
  W8A8_CHECK_ARG(mode >= TC_BF16 && mode <= TC_FP8 && kind >= EPI_BF16 && kind <= EPI_F32 && sms > 1,
                 W8A8_ERR_INVALID_ARG, "w8a8_tc_gemm_plan: mode %d, kind %d or SM count %d out of range", mode,
                 kind, sms);
  W8A8_CHECK_ARG(tc_gemm_supported(M, N, K, kind, false, 0), W8A8_ERR_SHAPE,
                 "w8a8_tc_gemm_plan: M=%d, N=%d, K=%d is not a tensor-core GEMM shape", M, N, K);
  const TcChoice c = tc_choose(mode, M, N, K, kind, split_ok != 0, sms);
  out[0] = c.pair;
  out[1] = c.bn;
  out[2] = c.ksplit;
  return W8A8_OK;
}

extern "C" w8a8_status w8a8_stream_gemm_plan(int int8_weights, int M, int N, int K, int sms, int* out) {
  W8A8_CHECK_ARG(out, W8A8_ERR_INVALID_ARG, "w8a8_stream_gemm_plan: null out");
  W8A8_CHECK_ARG(M >= 1 && N >= 1 && K >= 16 && sms > 0, W8A8_ERR_INVALID_ARG,
                 "w8a8_stream_gemm_plan: M=%d, N=%d, K=%d or SM count %d out of range", M, N, K, sms);
  const StreamPlan p = make_stream_plan(int8_weights != 0, M, N, K, sms);
  const int v[W8A8_STREAM_PLAN_FIELDS] = {p.dp4a, p.whole, p.dp4a ? p.MT : 0, p.NB, p.TOK,
                                          p.Z,    p.G,     p.KC,               p.C,  p.P,
                                          p.dp4a || p.NB <= 4 ? 2 : 1,        p.stages,
                                          p.stage_bytes,   p.smem_bytes,       (int)p.partial_bytes};
  for (int i = 0; i < W8A8_STREAM_PLAN_FIELDS; ++i) out[i] = v[i];
  return W8A8_OK;
}

extern "C" w8a8_status w8a8_set_kernel_events(void* start_event, void* stop_event) {
  W8A8_CHECK_ARG((start_event == nullptr) == (stop_event == nullptr), W8A8_ERR_INVALID_ARG,
                 "w8a8_set_kernel_events: give both events or neither");
  set_kernel_events(start_event, stop_event);
  return W8A8_OK;
}

extern "C" w8a8_status w8a8_workspace_check(void* workspace, void* stream) {
  W8A8_CHECK_ARG(workspace != nullptr, W8A8_ERR_INVALID_ARG, "w8a8_workspace_check: null workspace");
  cudaStream_t st = as_stream(stream);
  unsigned int* err = reinterpret_cast<unsigned int*>(reinterpret_cast<char*>(workspace) + kErrWordOffset);
  unsigned int host = 0;
  W8A8_CUDA(cudaMemcpyAsync(&host, err, sizeof(host), cudaMemcpyDeviceToHost, st));
  W8A8_CUDA(cudaStreamSynchronize(st));
  if (host == 0) return W8A8_OK;
  W8A8_CUDA(cudaMemsetAsync(err, 0, sizeof(unsigned int), st));
  W8A8_CUDA(cudaStreamSynchronize(st));
  set_error("a device-side wait gave up (error bits 0x%x: 1 consumer, 2 producer, 4 drain); results of the "
            "affected calls are undefined", host);
  return W8A8_ERR_TIMEOUT;
}
extern "C" const char* w8a8_last_error(void) { return get_error(); }

// ---------------------------------------------------------------------------- linear
extern "C" w8a8_status w8a8_linear_workspace_size(int M, int N, int K, size_t* bytes) {
  W8A8_CHECK_ARG(bytes && M >= 0 && N >= 0 && K >= 0, W8A8_ERR_INVALID_ARG, "w8a8_linear_workspace_size: bad argument");
  *bytes = linear_ws(M, N, K, true, device_sms()).total;
  return W8A8_OK;
}

extern "C" w8a8_status w8a8_linear(const w8a8_qweight* w, const uint16_t* X, int M, const float* bias, uint16_t* Y,
                                   const w8a8_debug* dbg, void* workspace, size_t ws_bytes, void* stream) {
  W8A8_TRY(check_qweight("w8a8_linear", w));
  W8A8_CHECK_ARG(M >= 0, W8A8_ERR_INVALID_ARG, "w8a8_linear: M=%d is negative", M);
  if (M == 0) return W8A8_OK;
  W8A8_CHECK_ARG(X && Y, W8A8_ERR_INVALID_ARG, "w8a8_linear: null X or Y");
  W8A8_CHECK_ARG(aligned16(X) && aligned16(Y) && (!bias || aligned16(bias)), W8A8_ERR_ALIGN,
                 "w8a8_linear: X, Y and bias must be 16-byte aligned");
  if (dbg)
    W8A8_CHECK_ARG((!dbg->xq || aligned16(dbg->xq)) && (!dbg->s_x || aligned16(dbg->s_x)) &&
                       (!dbg->acc || aligned16(dbg->acc)),
                   W8A8_ERR_ALIGN, "w8a8_linear: debug outputs must be 16-byte aligned");
  DevInfo d;
  W8A8_TRY(dev_info(&d));
  W8A8_TRY(check_ws("w8a8_linear", workspace, ws_bytes, linear_ws(M, w->n, w->k, true, d.sms).total));
  return run_w8a8_linear(w, X, M, bias, EPI_BF16, Y, nullptr, nullptr, dbg, workspace, d.sms, as_stream(stream));
}

extern "C" w8a8_status w8a8_linear_bf16_workspace_size(int M, int N, int K, size_t* bytes) {
  W8A8_CHECK_ARG(bytes && M >= 0 && N >= 0 && K >= 0, W8A8_ERR_INVALID_ARG,
                 "w8a8_linear_bf16_workspace_size: bad argument");
  *bytes = linear_ws(M, N, K, false, device_sms()).total;
  return W8A8_OK;
}

extern "C" w8a8_status w8a8_linear_bf16(const uint16_t* W, int N, int K, const uint16_t* X, int M, const float* bias,
                                        uint16_t* Y, void* workspace, size_t ws_bytes, void* stream) {
  W8A8_CHECK_ARG(M >= 0 && N > 0 && K > 0, W8A8_ERR_SHAPE, "w8a8_linear_bf16: bad shape M=%d N=%d K=%d", M, N, K);
  W8A8_CHECK_ARG(K % 16 == 0 && K <= W8A8_MAX_K, W8A8_ERR_SHAPE, "w8a8_linear_bf16: K=%d must be a multiple of 16", K);
  if (M == 0) return W8A8_OK;
  W8A8_CHECK_ARG(W && X && Y, W8A8_ERR_INVALID_ARG, "w8a8_linear_bf16: null pointer");
  W8A8_CHECK_ARG(aligned16(W) && aligned16(X) && aligned16(Y) && (!bias || aligned16(bias)), W8A8_ERR_ALIGN,
                 "w8a8_linear_bf16: pointers must be 16-byte aligned");
  DevInfo d;
  W8A8_TRY(dev_info(&d));
  W8A8_TRY(check_ws("w8a8_linear_bf16", workspace, ws_bytes, linear_ws(M, N, K, false, d.sms).total));
  return run_bf16_linear(W, N, K, X, M, bias, EPI_BF16, Y, nullptr, nullptr, workspace, d.sms, as_stream(stream));
}

// ------------------------------------------------------------------------------- FFN
// Layout: [reserved | h bf16 [M,F] | gate/up linear scratch | down linear scratch]

namespace w8a8 {

FfnWs ffn_ws(int M, int H, int F, int sms) {
  FfnWs w{};
  size_t off = W8A8_WS_RESERVED;
  w.h = off;
  off += round_up((size_t)M * F * 2, 256);
  const LinearWs a = linear_ws(M, 2 * F, H, true, sms);
  const LinearWs b = linear_ws(M, H, F, true, sms);
  w.gu = off;
  off += a.total - W8A8_WS_RESERVED;
  w.dn = off;
  off += b.total - W8A8_WS_RESERVED;
  w.rowmax = off;  // gate/up's partial row maxima for down's quantiser (decode GEMV, 16 slots at most)
  off += round_up((size_t)2 * std::max(sms, 1) * 16 * 4, 256);
  w.total = off;
  return w;
}

w8a8_status run_ffn(const w8a8_ffn_weights* f, int precision, const uint16_t* X, int M, uint16_t* Y, uint16_t* h_dbg,
                    void* workspace, int sms, cudaStream_t st, const ResNorm* rn_gate_up, const PreCodes* pre_gate_up) {
  const int H = f->hidden, F = f->inter;
  const FfnWs L = ffn_ws(M, H, F, sms);
  char* base = reinterpret_cast<char*>(workspace);
  uint16_t* h = h_dbg ? h_dbg : reinterpret_cast<uint16_t*>(base + L.h);
  // The two linears run one after the other on `stream` and share the FFN workspace's reserved
  // counters (each leaves them zero); their scratch regions are disjoint.
  if (precision == W8A8_PREC_W8A8) {
    // gate/up: scratch at L.gu.  At 5-16 tokens, when both linears run the decode GEMV's tensor-core
    // path, gate/up's GeGLU epilogue also hands down the partial maxima of its quantiser's first pass.
    w8a8_status ss = W8A8_OK;
    const SmallPlan pg = make_small_plan(true, M, 2 * F, H, EPI_GEGLU, sms, rn_gate_up != nullptr);
    const SmallPlan pd = make_small_plan(true, M, H, F, EPI_BF16, sms, false);
    const bool handoff = pg.ok && pd.ok && pg.MT >= 8 && pd.MT == pg.MT;
    float* rowmax = reinterpret_cast<float*>(base + L.rowmax);
    const RowMax rm_gu{rowmax, f->down.inv_delta, nullptr, 0}, rm_dn{nullptr, nullptr, rowmax, pg.P};
    if (small_gemv(true, f->gate_up.wq, f->gate_up.inv_delta, f->gate_up.s_w, X, M, 2 * F, H, nullptr, EPI_GEGLU, h,
                   nullptr, workspace, rn_gate_up, sms, st, &ss, handoff ? &rm_gu : nullptr)) {
      W8A8_TRY(ss);
    } else if (rn_gate_up) {
      W8A8_CHECK_ARG(false, W8A8_ERR_SHAPE, "fused residual norm: the decode GEMV does not take gate/up at M=%d", M);
    } else if (tc_path(true, f->gate_up.wq_f16, X, M, 2 * F, H, nullptr, EPI_GEGLU, f->gate_up.inv_delta,
                       f->gate_up.s_w, h, nullptr, nullptr, nullptr, workspace,
                       base + L.gu + (linear_ws(M, 2 * F, H, true, sms).xf16 - W8A8_WS_RESERVED),
                       reinterpret_cast<float*>(base + L.gu + (linear_ws(M, 2 * F, H, true, sms).sx - W8A8_WS_RESERVED)),
                       base + L.gu + (linear_ws(M, 2 * F, H, true, sms).part - W8A8_WS_RESERVED), st, &ss,
                       pre_gate_up)) {
      W8A8_TRY(ss);
    } else {
      const LinearWs A = linear_ws(M, 2 * F, H, true, sms);
      void* codes = base + L.gu + (A.xf16 - W8A8_WS_RESERVED);
      float* s_x = reinterpret_cast<float*>(base + L.gu + (A.sx - W8A8_WS_RESERVED));
      StreamArgs a{};
      a.p = make_stream_plan(true, M, 2 * F, H, sms);
      W8A8_TRY(quantize_for(a.p, X, M, H, f->gate_up.inv_delta, codes, nullptr, s_x, st));
      a.W = f->gate_up.wq;
      a.X = codes;
      a.M = M;
      a.N = 2 * F;
      a.K = H;
      a.kind = EPI_GEGLU;
      a.s_x = s_x;
      a.s_w = f->gate_up.s_w;
      a.y = h;
      a.partials = base + L.gu + (A.part - W8A8_WS_RESERVED);
      attach_reserved(a, workspace);
      W8A8_TRY(launch_stream_gemm(true, a, st));
    }
    if (small_gemv(true, f->down.wq, f->down.inv_delta, f->down.s_w, h, M, H, F, nullptr, EPI_BF16, Y, nullptr,
                   workspace, nullptr, sms, st, &ss, handoff ? &rm_dn : nullptr)) {
      W8A8_TRY(ss);
    } else if (tc_path(true, f->down.wq_f16, h, M, H, F, nullptr, EPI_BF16, f->down.inv_delta, f->down.s_w, Y,
                       nullptr, nullptr, nullptr, workspace,
                       base + L.dn + (linear_ws(M, H, F, true, sms).xf16 - W8A8_WS_RESERVED),
                       reinterpret_cast<float*>(base + L.dn + (linear_ws(M, H, F, true, sms).sx - W8A8_WS_RESERVED)),
                       base + L.dn + (linear_ws(M, H, F, true, sms).part - W8A8_WS_RESERVED), st, &ss)) {
      W8A8_TRY(ss);
    } else {
      const LinearWs B = linear_ws(M, H, F, true, sms);
      void* codes = base + L.dn + (B.xf16 - W8A8_WS_RESERVED);
      float* s_x = reinterpret_cast<float*>(base + L.dn + (B.sx - W8A8_WS_RESERVED));
      StreamArgs a{};
      a.p = make_stream_plan(true, M, H, F, sms);
      W8A8_TRY(quantize_for(a.p, h, M, F, f->down.inv_delta, codes, nullptr, s_x, st));
      a.W = f->down.wq;
      a.X = codes;
      a.M = M;
      a.N = H;
      a.K = F;
      a.kind = EPI_BF16;
      a.s_x = s_x;
      a.s_w = f->down.s_w;
      a.y = Y;
      a.partials = base + L.dn + (B.part - W8A8_WS_RESERVED);
      attach_reserved(a, workspace);
      W8A8_TRY(launch_stream_gemm(true, a, st));
    }
  } else {
    w8a8_status ss = W8A8_OK;
    if (small_gemv(false, f->gate_up_bf16, nullptr, nullptr, X, M, 2 * F, H, nullptr, EPI_GEGLU, h, nullptr,
                   workspace, rn_gate_up, sms, st, &ss)) {
      W8A8_TRY(ss);
    } else if (rn_gate_up) {
      W8A8_CHECK_ARG(false, W8A8_ERR_SHAPE, "fused residual norm: the decode GEMV does not take gate/up at M=%d", M);
    } else if (tc_path(false, f->gate_up_bf16, X, M, 2 * F, H, nullptr, EPI_GEGLU, nullptr, nullptr, h, nullptr,
                       nullptr, nullptr, workspace, nullptr, nullptr,
                       base + L.gu + (linear_ws(M, 2 * F, H, false, sms).part - W8A8_WS_RESERVED), st, &ss)) {
      W8A8_TRY(ss);
    } else {
      const LinearWs A = linear_ws(M, 2 * F, H, false, sms);
      StreamArgs a{};
      a.W = f->gate_up_bf16;
      a.X = X;
      a.M = M;
      a.N = 2 * F;
      a.K = H;
      a.p = make_stream_plan(false, M, 2 * F, H, sms);
      a.kind = EPI_GEGLU;
      a.y = h;
      a.partials = base + L.gu + (A.part - W8A8_WS_RESERVED);
      attach_reserved(a, workspace);
      W8A8_TRY(launch_stream_gemm(false, a, st));
    }
    if (small_gemv(false, f->down_bf16, nullptr, nullptr, h, M, H, F, nullptr, EPI_BF16, Y, nullptr, workspace,
                   nullptr, sms, st, &ss)) {
      W8A8_TRY(ss);
    } else if (tc_path(false, f->down_bf16, h, M, H, F, nullptr, EPI_BF16, nullptr, nullptr, Y, nullptr, nullptr,
                       nullptr, workspace, nullptr, nullptr,
                       base + L.dn + (linear_ws(M, H, F, false, sms).part - W8A8_WS_RESERVED), st, &ss)) {
      W8A8_TRY(ss);
    } else {
      const LinearWs B = linear_ws(M, H, F, false, sms);
      StreamArgs a{};
      a.W = f->down_bf16;
      a.X = h;
      a.M = M;
      a.N = H;
      a.K = F;
      a.p = make_stream_plan(false, M, H, F, sms);
      a.kind = EPI_BF16;
      a.y = Y;
      a.partials = base + L.dn + (B.part - W8A8_WS_RESERVED);
      attach_reserved(a, workspace);
      W8A8_TRY(launch_stream_gemm(false, a, st));
    }
  }
  return W8A8_OK;
}
}  // namespace w8a8

extern "C" w8a8_status w8a8_ffn_workspace_size(int M, int hidden, int inter, size_t* bytes) {
  W8A8_CHECK_ARG(bytes && M >= 0 && hidden >= 0 && inter >= 0, W8A8_ERR_INVALID_ARG, "w8a8_ffn_workspace_size: bad argument");
  *bytes = ffn_ws(M, hidden, inter, device_sms()).total;
  return W8A8_OK;
}

extern "C" w8a8_status w8a8_ffn_block(const w8a8_ffn_weights* f, int precision, const uint16_t* X, int M, uint16_t* Y,
                                      uint16_t* h_dbg, void* workspace, size_t ws_bytes, void* stream) {
  W8A8_CHECK_ARG(f != nullptr, W8A8_ERR_INVALID_ARG, "w8a8_ffn_block: null FFN descriptor");
  W8A8_CHECK_ARG(precision == W8A8_PREC_BF16 || precision == W8A8_PREC_W8A8, W8A8_ERR_INVALID_ARG,
                 "w8a8_ffn_block: precision %d", precision);
  const int H = f->hidden, F = f->inter;
  W8A8_CHECK_ARG(H > 0 && F > 0 && H % 16 == 0 && F % 16 == 0 && H <= W8A8_MAX_K && F <= W8A8_MAX_K, W8A8_ERR_SHAPE,
                 "w8a8_ffn_block: hidden=%d inter=%d must be positive multiples of 16", H, F);
  W8A8_CHECK_ARG(M >= 0, W8A8_ERR_INVALID_ARG, "w8a8_ffn_block: M=%d is negative", M);
  if (M == 0) return W8A8_OK;
  W8A8_CHECK_ARG(X && Y, W8A8_ERR_INVALID_ARG, "w8a8_ffn_block: null X or Y");
  W8A8_CHECK_ARG(aligned16(X) && aligned16(Y) && (!h_dbg || aligned16(h_dbg)), W8A8_ERR_ALIGN,
                 "w8a8_ffn_block: X, Y, h must be 16-byte aligned");
  if (precision == W8A8_PREC_W8A8) {
    W8A8_TRY(check_qweight("w8a8_ffn_block(gate_up)", &f->gate_up));
    W8A8_TRY(check_qweight("w8a8_ffn_block(down)", &f->down));
    W8A8_CHECK_ARG(f->gate_up.n == 2 * F && f->gate_up.k == H && f->down.n == H && f->down.k == F, W8A8_ERR_SHAPE,
                   "w8a8_ffn_block: weight shapes do not match hidden=%d inter=%d", H, F);
  } else {
    W8A8_CHECK_ARG(f->gate_up_bf16 && f->down_bf16, W8A8_ERR_INVALID_ARG, "w8a8_ffn_block: null bf16 weights");
    W8A8_CHECK_ARG(aligned16(f->gate_up_bf16) && aligned16(f->down_bf16), W8A8_ERR_ALIGN,
                   "w8a8_ffn_block: bf16 weights must be 16-byte aligned");
  }
  DevInfo d;
  W8A8_TRY(dev_info(&d));
  const FfnWs L = ffn_ws(M, H, F, d.sms);
  W8A8_TRY(check_ws("w8a8_ffn_block", workspace, ws_bytes, L.total));
  return run_ffn(f, precision, X, M, Y, h_dbg, workspace, d.sms, as_stream(stream));
}

// --------------------------------------------------------------------------- lm_head
extern "C" w8a8_status w8a8_lm_head_workspace_size(int M, int vocab, int hidden, size_t* bytes) {
  W8A8_CHECK_ARG(bytes && M >= 0 && vocab >= 0 && hidden >= 0, W8A8_ERR_INVALID_ARG, "w8a8_lm_head_workspace_size: bad argument");
  *bytes = linear_ws(M, vocab, hidden, true, device_sms()).total;
  return W8A8_OK;
}

extern "C" w8a8_status w8a8_lm_head(const w8a8_head_weights* hd, int precision, const uint16_t* X, int M, float* logits,
                                    int32_t* top1, void* workspace, size_t ws_bytes, void* stream) {
  W8A8_CHECK_ARG(hd != nullptr, W8A8_ERR_INVALID_ARG, "w8a8_lm_head: null head descriptor");
  W8A8_CHECK_ARG(precision == W8A8_PREC_BF16 || precision == W8A8_PREC_W8A8, W8A8_ERR_INVALID_ARG,
                 "w8a8_lm_head: precision %d", precision);
  const int V = hd->vocab, D = hd->hidden;
  W8A8_CHECK_ARG(V > 0 && D > 0 && D % 16 == 0 && D <= W8A8_MAX_K, W8A8_ERR_SHAPE, "w8a8_lm_head: vocab=%d hidden=%d", V, D);
  W8A8_CHECK_ARG(M >= 0, W8A8_ERR_INVALID_ARG, "w8a8_lm_head: M=%d is negative", M);
  if (M == 0) return W8A8_OK;
  W8A8_CHECK_ARG(M <= max_top_keys(), W8A8_ERR_SHAPE, "w8a8_lm_head: M=%d exceeds %d tokens per call", M, max_top_keys());
  W8A8_CHECK_ARG(X && top1, W8A8_ERR_INVALID_ARG, "w8a8_lm_head: null X or top1");
  W8A8_CHECK_ARG(aligned16(X) && aligned16(top1) && (!logits || aligned16(logits)), W8A8_ERR_ALIGN,
                 "w8a8_lm_head: pointers must be 16-byte aligned");
  DevInfo d;
  W8A8_TRY(dev_info(&d));
  cudaStream_t st = as_stream(stream);
  if (precision == W8A8_PREC_W8A8) {
    W8A8_TRY(check_qweight("w8a8_lm_head", &hd->q));
    W8A8_CHECK_ARG(hd->q.n == V && hd->q.k == D, W8A8_ERR_SHAPE, "w8a8_lm_head: weight shape mismatch");
    W8A8_TRY(check_ws("w8a8_lm_head", workspace, ws_bytes, linear_ws(M, V, D, true, d.sms).total));
    return run_w8a8_linear(&hd->q, X, M, nullptr, EPI_F32, nullptr, logits, top1, nullptr, workspace, d.sms, st);
  }
  W8A8_CHECK_ARG(hd->bf16 && aligned16(hd->bf16), W8A8_ERR_INVALID_ARG, "w8a8_lm_head: null or unaligned bf16 table");
  W8A8_TRY(check_ws("w8a8_lm_head", workspace, ws_bytes, linear_ws(M, V, D, false, d.sms).total));
  return run_bf16_linear(hd->bf16, V, D, X, M, nullptr, EPI_F32, nullptr, logits, top1, workspace, d.sms, st);
}
