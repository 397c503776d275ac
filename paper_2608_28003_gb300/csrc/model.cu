// The Gemma-3-1B-shaped decoder under a per-layer precision mask, its calibration and weight
// preparation, CUDA-graph decode steps, the token NLL, and the mask allocator (host C++ driving
// the library's kernels).
#include <algorithm>
#include <chrono>
#include <cmath>
#include <map>
#include <tuple>
#include <utility>
#include <vector>

#include "decoder_kernels.cuh"
#include "ops.cuh"
#include "stream_gemm.cuh"

using namespace w8a8;

namespace {

struct QW {
  int8_t* wq = nullptr;
  uint16_t* wq_f16 = nullptr;  // the same codes as fp16, for the tensor-core GEMM of prefill
  float* s_w = nullptr;
  float* delta = nullptr;
  float* inv_delta = nullptr;
};

constexpr int kHeadChunk = 2048;  // lm_head rows per launch (top-1 keys per call)

}  // namespace

struct w8a8_model {
  w8a8_model_cfg cfg{};
  int sms = 152;
  std::vector<w8a8_layer_bf16> L;
  const uint16_t* embed = nullptr;
  const float* final_norm = nullptr;
  int q_dim = 0, kv_dim = 0, qkv_dim = 0;
  float embed_scale = 1.0f;

  uint16_t* gu_bf16 = nullptr;  // [layers][2F][H] bf16, 8-row gate/up interleave
  std::vector<QW> q_qkv, q_o, q_gu, q_down;
  QW q_lm;
  bool prepared = false;
  int prep_version = 0;
  float* stats = nullptr;  // per layer: [H] qkv input, [q_dim] o input, [H] gate/up input, [F] down input; then [H] lm

  uint32_t ffn_bits = 0, attn_bits = 0;
  int lm = 0;

  float* r = nullptr;
  float* r2 = nullptr;  // the residual stream ping-pongs between r and r2 when its update is fused
  uint16_t *a = nullptr, *qkv = nullptr, *o = nullptr, *y = nullptr, *h = nullptr;
  float* q = nullptr;
  uint16_t *kc = nullptr, *vc = nullptr;
  float *cos_l = nullptr, *sin_l = nullptr, *cos_g = nullptr, *sin_g = nullptr;
  int* d_pos = nullptr;
  int32_t* d_tokens = nullptr;
  float* d_logits = nullptr;
  int32_t* d_top1 = nullptr;
  void* ws = nullptr;
  size_t ws_bytes = 0;
  void* attn_ws = nullptr;
  size_t attn_ws_bytes = 0;
  // the next W8A8 linear's quantised input written by the norm kernels at 9+ tokens ([max_tokens,
  // hidden] fp16 codes, [max_tokens] scales and sums of |codes|), so that its GEMM needs no
  // quantiser launch
  uint16_t* pcodes = nullptr;
  float* psx = nullptr;
  int* psum = nullptr;
  // diagnostics: when set, a forward copies every layer's output (the residual stream after its
  // post-FFN step, fp32 [M, H]) to capture + l M H
  float* capture = nullptr;
  // diagnostics: when trace_on, a forward copies every layer's intermediate tensors into the
  // caller's trace buffers (w8a8_model_set_trace)
  bool trace_on = false;
  w8a8_trace trace{};

  cudaStream_t st = nullptr;  // private stream for graph capture / replay
  cudaEvent_t ev_in = nullptr, ev_out = nullptr;
  struct Graph {
    cudaGraphExec_t exec;
    int kernels;  // kernel nodes
  };
  std::map<std::tuple<int, uint32_t, uint32_t, int, int, int>, Graph> graphs;
  std::vector<void*> allocs;

  size_t stats_stride() const { return (size_t)2 * cfg.hidden + q_dim + cfg.inter; }
  float* stat_qkv(int l) const { return stats + l * stats_stride(); }
  float* stat_o(int l) const { return stat_qkv(l) + cfg.hidden; }
  float* stat_gu(int l) const { return stat_o(l) + q_dim; }
  float* stat_down(int l) const { return stat_gu(l) + cfg.hidden; }
  float* stat_lm() const { return stats + (size_t)cfg.layers * stats_stride(); }
  size_t cache_layer_elems() const { return (size_t)cfg.max_batch * cfg.max_seq * kv_dim; }
  bool is_global(int l) const {
    for (int i = 0; i < cfg.n_global; ++i)
      if (cfg.global_layers[i] == l) return true;
    return false;
  }
};

namespace {

template <class T>
w8a8_status dalloc(w8a8_model* m, T** p, size_t count) {
  void* v = nullptr;
  W8A8_CUDA(cudaMalloc(&v, std::max<size_t>(count * sizeof(T), 16)));
  m->allocs.push_back(v);
  *p = reinterpret_cast<T*>(v);
  return W8A8_OK;
}

void free_all(w8a8_model* m) {
  for (auto& kv : m->graphs) cudaGraphExecDestroy(kv.second.exec);
  m->graphs.clear();
  for (void* p : m->allocs) cudaFree(p);
  m->allocs.clear();
  if (m->ev_in) cudaEventDestroy(m->ev_in);
  if (m->ev_out) cudaEventDestroy(m->ev_out);
  if (m->st) cudaStreamDestroy(m->st);
}

w8a8_qweight qdesc(const QW& q, int n, int k) { return w8a8_qweight{n, k, q.wq, q.s_w, q.inv_delta, q.wq_f16}; }

w8a8_status linear(w8a8_model* m, bool int8, const QW& qw, const uint16_t* Wbf, int N, int K, const uint16_t* X, int M,
                   uint16_t* Y, cudaStream_t st, const ResNorm* rn, const PreCodes* pre = nullptr) {
  if (int8) {
    const w8a8_qweight w = qdesc(qw, N, K);
    return run_w8a8_linear(&w, X, M, nullptr, 0, Y, nullptr, nullptr, nullptr, m->ws, m->sms, st, rn, pre);
  }
  return run_bf16_linear(Wbf, N, K, X, M, nullptr, 0, Y, nullptr, nullptr, m->ws, m->sms, st, rn);
}

// At decode the residual step (residual add + the two RMSNorms) runs inside the next linear's
// decode GEMV: q/k/v takes the step after the previous layer's FFN, gate/up the step after o.
// It needs the decode GEMV to take both linears of every layer under the current mask.
bool fuse_residual(const w8a8_model* m, int M, bool calib) {
  if (calib || M > 8 || m->capture || m->trace_on) return false;
  const int H = m->cfg.hidden, F = m->cfg.inter;
  for (int l = 0; l < m->cfg.layers; ++l) {
    const bool att8 = m->prepared && ((m->attn_bits >> l) & 1u);
    const bool ffn8 = m->prepared && ((m->ffn_bits >> l) & 1u);
    if (!decode_gemv_takes(att8, M, m->qkv_dim, H, false, m->sms)) return false;
    if (!decode_gemv_takes(ffn8, M, 2 * F, H, true, m->sms)) return false;
  }
  return true;
}

// The decoder over M = B * T rows whose positions start at *m->d_pos (set by the caller).
w8a8_status forward_core(w8a8_model* m, const int32_t* tokens, int B, int T, float* logits, int32_t* top1, bool calib,
                         cudaStream_t st) {
  const w8a8_model_cfg& c = m->cfg;
  const int M = B * T, H = c.hidden, F = c.inter;
  const bool fuse = fuse_residual(m, M, calib);
  float* rc = m->r;   // the residual stream as of now
  float* rn = m->r2;  // where a fused update writes the next one
  // 9+ tokens: the norm kernels quantise the input of the next W8A8 linear themselves (its
  // tensor-core GEMM then needs no quantiser launch); fewer tokens run the decode GEMV, which
  // quantises inside
  const bool preq = !calib && M >= 9 && m->prepared;
  const PreCodes pc{m->pcodes, m->psx, m->psum};
  auto att8_of = [&](int l) { return !calib && m->prepared && ((m->attn_bits >> l) & 1u); };
  const bool pre0 = preq && att8_of(0);
  W8A8_TRY(launch_embed_norm(tokens, M, m->embed, c.vocab, H, m->embed_scale, m->L[0].ln_in, c.eps, rc, m->a, st,
                             pre0 ? m->q_qkv[0].inv_delta : nullptr, m->pcodes, m->psx, m->psum));
  bool pre_qkv = pre0;  // whether the codes of the current q/k/v input exist
  const w8a8_trace* tr = m->trace_on && !calib ? &m->trace : nullptr;
  W8A8_CHECK_ARG(!tr || M <= tr->max_rows, W8A8_ERR_SHAPE, "trace: %d rows exceed the trace's %d", M, tr ? tr->max_rows : 0);
  // copy this call's M rows of a [rows, width] tensor into slice l of a [L][max_rows][width] trace buffer
  auto trace_copy = [&](void* base, int l, const void* src, int width, size_t elem) -> w8a8_status {
    if (!base) return W8A8_OK;
    char* dst = static_cast<char*>(base) + ((size_t)l * tr->max_rows) * width * elem;
    W8A8_CUDA(cudaMemcpyAsync(dst, src, (size_t)M * width * elem, cudaMemcpyDeviceToDevice, st));
    return W8A8_OK;
  };
  for (int l = 0; l < c.layers; ++l) {
    const w8a8_layer_bf16& W = m->L[l];
    const bool att8 = !calib && m->prepared && ((m->attn_bits >> l) & 1u);
    const bool ffn8 = !calib && m->prepared && ((m->ffn_bits >> l) & 1u);
    const bool glob = m->is_global(l);
    if (calib) W8A8_TRY(launch_act_absmax(m->a, M, H, m->stat_qkv(l), st));
    AttnShape s{B, T, c.n_q, c.n_kv, c.head_dim, c.max_seq, glob ? 0 : c.window,
                (float)(1.0 / std::sqrt((double)c.head_dim))};
    uint16_t* kc = m->kc + (size_t)l * m->cache_layer_elems();
    uint16_t* vc = m->vc + (size_t)l * m->cache_layer_elems();
    const float* qn = c.qk_norm ? W.q_norm : nullptr;
    const float* kn = c.qk_norm ? W.k_norm : nullptr;
    const float* cs = glob ? m->cos_g : m->cos_l;
    const float* sn = glob ? m->sin_g : m->sin_l;
    const QW& qq = m->q_qkv[l];
    if (fuse && l > 0) {  // the previous layer's post-FFN step, then q/k/v
      const ResNorm R{m->y, rc, rn, m->L[l - 1].ln_post_ffn, W.ln_in, c.eps};
      W8A8_TRY(linear(m, att8, qq, W.wqkv, m->qkv_dim, H, nullptr, M, m->qkv, st, &R));
      std::swap(rc, rn);
    } else {
      if (tr) W8A8_TRY(trace_copy(tr->a_in, l, m->a, H, 2));
      W8A8_TRY(linear(m, att8, qq, W.wqkv, m->qkv_dim, H, m->a, M, m->qkv, st, nullptr, pre_qkv ? &pc : nullptr));
      if (tr) W8A8_TRY(trace_copy(tr->qkv, l, m->qkv, m->qkv_dim, 2));
    }
    if (attn_decode_supported(s)) {
      W8A8_TRY(launch_attn_decode(m->qkv, s, m->d_pos, qn, kn, c.eps, cs, sn, kc, vc, m->o, st));
    } else {
      W8A8_TRY(launch_qk_rope(m->qkv, s, m->d_pos, qn, kn, c.eps, cs, sn, m->q, kc, vc, st));
      if (attention_prefill_supported(s))
        W8A8_TRY(launch_attention_prefill(m->q, kc, vc, s, m->d_pos, m->o, st));
      else
        W8A8_TRY(launch_attention(m->q, kc, vc, s, m->d_pos, 0, m->o, m->attn_ws, m->sms, st));
    }
    if (calib) W8A8_TRY(launch_act_absmax(m->o, M, m->q_dim, m->stat_o(l), st));
    if (tr) W8A8_TRY(trace_copy(tr->attn, l, m->o, m->q_dim, 2));
    W8A8_TRY(linear(m, att8, m->q_o[l], W.wo, H, m->q_dim, m->o, M, m->y, st, nullptr));
    if (tr) W8A8_TRY(trace_copy(tr->y_o, l, m->y, H, 2));
    w8a8_ffn_weights f{H,
                       F,
                       qdesc(m->q_gu[l], 2 * F, H),
                       qdesc(m->q_down[l], H, F),
                       m->gu_bf16 + (size_t)l * 2 * F * H,
                       W.wdown};
    const int prec = ffn8 ? W8A8_PREC_W8A8 : W8A8_PREC_BF16;
    if (fuse) {  // the post-attention step inside gate/up
      const ResNorm R{m->y, rc, rn, W.ln_post_attn, W.ln_pre_ffn, c.eps};
      W8A8_TRY(run_ffn(&f, prec, nullptr, M, m->y, nullptr, m->ws, m->sms, st, &R));
      std::swap(rc, rn);
    } else {
      const bool pre_gu = preq && ffn8;
      W8A8_TRY(launch_residual_norm(m->y, M, H, W.ln_post_attn, W.ln_pre_ffn, c.eps, rc, m->a, st,
                                    pre_gu ? m->q_gu[l].inv_delta : nullptr, m->pcodes, m->psx, m->psum));
      if (calib) W8A8_TRY(launch_act_absmax(m->a, M, H, m->stat_gu(l), st));
      if (tr) W8A8_TRY(trace_copy(tr->a_ffn, l, m->a, H, 2));
      uint16_t* h_out = calib ? m->h : nullptr;
      if (tr && tr->h) h_out = tr->h + (size_t)l * tr->max_rows * F;  // the block writes h there
      W8A8_TRY(run_ffn(&f, prec, m->a, M, m->y, h_out, m->ws, m->sms, st, nullptr, pre_gu ? &pc : nullptr));
      if (tr) W8A8_TRY(trace_copy(tr->y_f, l, m->y, H, 2));
    }
    if (calib) W8A8_TRY(launch_act_absmax(m->h, M, F, m->stat_down(l), st));
    if (!fuse || l + 1 == c.layers) {
      const float* next = l + 1 < c.layers ? m->L[l + 1].ln_in : m->final_norm;
      pre_qkv = preq && l + 1 < c.layers && att8_of(l + 1);
      W8A8_TRY(launch_residual_norm(m->y, M, H, W.ln_post_ffn, next, c.eps, rc, m->a, st,
                                    pre_qkv ? m->q_qkv[l + 1].inv_delta : nullptr, m->pcodes, m->psx, m->psum));
    }
    if (m->capture)
      W8A8_CUDA(cudaMemcpyAsync(m->capture + (size_t)l * M * H, rc, sizeof(float) * M * H, cudaMemcpyDeviceToDevice, st));
    if (tr) W8A8_TRY(trace_copy(tr->r, l, rc, H, 4));
  }
  if (tr) W8A8_TRY(trace_copy(tr->a_fin, 0, m->a, H, 2));
  if (calib) return launch_act_absmax(m->a, M, H, m->stat_lm(), st);
  const bool lm8 = m->prepared && m->lm;
  for (int r0 = 0; r0 < M; r0 += kHeadChunk) {
    const int rows = std::min(kHeadChunk, M - r0);
    const uint16_t* X = m->a + (size_t)r0 * H;
    float* lg = logits ? logits + (size_t)r0 * c.vocab : nullptr;
    int32_t* tp = top1 + r0;
    if (lm8) {
      const w8a8_qweight w = qdesc(m->q_lm, c.vocab, H);
      W8A8_TRY(run_w8a8_linear(&w, X, rows, nullptr, 2, nullptr, lg, tp, nullptr, m->ws, m->sms, st));
    } else {
      W8A8_TRY(run_bf16_linear(m->embed, c.vocab, H, X, rows, nullptr, 2, nullptr, lg, tp, m->ws, m->sms, st));
    }
  }
  return W8A8_OK;
}

w8a8_status check_call(w8a8_model* m, int B, int T, int start_pos) {
  W8A8_CHECK_ARG(m != nullptr, W8A8_ERR_INVALID_ARG, "null model");
  W8A8_CHECK_ARG(B > 0 && T > 0 && B <= m->cfg.max_batch && B * T <= m->cfg.max_tokens, W8A8_ERR_SHAPE,
                 "B=%d T=%d exceeds the model's capacity (max_batch %d, max_tokens %d)", B, T, m->cfg.max_batch,
                 m->cfg.max_tokens);
  W8A8_CHECK_ARG(start_pos >= 0 && start_pos + T <= m->cfg.max_seq, W8A8_ERR_SHAPE,
                 "positions %d..%d exceed max_seq %d", start_pos, start_pos + T - 1, m->cfg.max_seq);
  return W8A8_OK;
}

// ------------------------------------------------------------------------------ NLL kernel
// Eq. sqnr-ffn / sqnr-block: the sums of y_ref^2 and (y_ref - y_q)^2 in fp64.  Each of the
// kSqnrBlocks blocks strides over the elements and reduces its 256 threads in a fixed tree; the
// host adds the blocks' partials in block order (deterministic).
constexpr int kSqnrBlocks = 256;
__global__ void sqnr_partial_kernel(const float* __restrict__ ref, const float* __restrict__ q, size_t n,
                                    double* __restrict__ part) {
  __shared__ double ss[256], se[256];
  double s = 0.0, e = 0.0;
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x) {
    const double r = ref[i], d = r - (double)q[i];
    s += r * r;
    e += d * d;
  }
  ss[threadIdx.x] = s;
  se[threadIdx.x] = e;
  __syncthreads();
  for (int o = 128; o > 0; o >>= 1) {
    if ((int)threadIdx.x < o) {
      ss[threadIdx.x] += ss[threadIdx.x + o];
      se[threadIdx.x] += se[threadIdx.x + o];
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    part[2 * blockIdx.x] = ss[0];
    part[2 * blockIdx.x + 1] = se[0];
  }
}

__global__ void nll_kernel(const float* __restrict__ logits, const int32_t* __restrict__ targets, int V,
                           float* __restrict__ nll) {
  __shared__ double red[32];
  __shared__ float s_max;
  const int row = blockIdx.x;
  const float* z = logits + (size_t)row * V;
  float mx = -INFINITY;
  for (int i = threadIdx.x; i < V; i += blockDim.x) mx = fmaxf(mx, z[i]);
  mx = warp_max(mx);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = mx;
  __syncthreads();
  if (threadIdx.x == 0) {
    float v = -INFINITY;
    for (int i = 0; i < (int)(blockDim.x >> 5); ++i) v = fmaxf(v, (float)red[i]);
    s_max = v;
  }
  __syncthreads();
  const float m = s_max;
  double sum = 0.0;
  for (int i = threadIdx.x; i < V; i += blockDim.x) sum += exp((double)(z[i] - m));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
  __syncthreads();
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = sum;
  __syncthreads();
  if (threadIdx.x == 0) {
    double s = 0.0;
    for (int i = 0; i < (int)(blockDim.x >> 5); ++i) s += red[i];
    const int tg = targets[row];
    nll[row] = (float)(log(s) + (double)m - (double)z[tg]);
  }
}

__global__ void shift_targets_kernel(const int32_t* tokens, int B, int T, int32_t* targets) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= B * T) return;
  const int t = i % T;
  targets[i] = t + 1 < T ? tokens[i + 1] : tokens[i];
}

__global__ void fill_tokens_kernel(int32_t* tokens, int n, int vocab) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) tokens[i] = (int32_t)(((long long)i * 7919 + 13) % vocab);
}

}  // namespace

// ====================================================================================== ABI
extern "C" w8a8_status w8a8_model_create(const w8a8_model_cfg* cfg, const w8a8_layer_bf16* layers,
                                         const uint16_t* embed, const float* final_norm, w8a8_model** out) {
  W8A8_CHECK_ARG(cfg && layers && embed && final_norm && out, W8A8_ERR_INVALID_ARG, "w8a8_model_create: null argument");
  const w8a8_model_cfg& c = *cfg;
  W8A8_CHECK_ARG(c.layers > 0 && c.layers <= 32 && c.hidden > 0 && c.hidden % 16 == 0 && c.hidden <= 4096 &&
                     c.inter > 0 && c.inter % 16 == 0 && c.head_dim == 256 && c.n_kv > 0 && c.n_q % c.n_kv == 0 &&
                     c.n_q / c.n_kv <= 8 && c.n_q + 2 * c.n_kv <= 32 && c.vocab > 0 && c.max_batch > 0 &&
                     c.max_seq > 0 && c.max_tokens > 0 && c.n_global >= 0 && c.n_global <= 32,
                 W8A8_ERR_SHAPE, "w8a8_model_create: unsupported configuration");
  W8A8_CHECK_ARG(aligned16(embed) && aligned16(final_norm), W8A8_ERR_ALIGN, "w8a8_model_create: unaligned pointer");
  for (int l = 0; l < c.layers; ++l) {
    const w8a8_layer_bf16& W = layers[l];
    W8A8_CHECK_ARG(W.wqkv && W.wo && W.wgate && W.wup && W.wdown && W.ln_in && W.ln_post_attn && W.ln_pre_ffn &&
                       W.ln_post_ffn && (!c.qk_norm || (W.q_norm && W.k_norm)),
                   W8A8_ERR_INVALID_ARG, "w8a8_model_create: layer %d has a null pointer", l);
    W8A8_CHECK_ARG(aligned16(W.wqkv) && aligned16(W.wo) && aligned16(W.wgate) && aligned16(W.wup) &&
                       aligned16(W.wdown),
                   W8A8_ERR_ALIGN, "w8a8_model_create: layer %d weight not 16-byte aligned", l);
  }
  DevInfo d;
  W8A8_TRY(dev_info(&d));
  w8a8_model* m = new w8a8_model();
  m->cfg = c;
  m->sms = d.sms;
  m->L.assign(layers, layers + c.layers);
  m->embed = embed;
  m->final_norm = final_norm;
  m->q_dim = c.n_q * c.head_dim;
  m->kv_dim = c.n_kv * c.head_dim;
  m->qkv_dim = m->q_dim + 2 * m->kv_dim;
  m->embed_scale = (float)std::sqrt((double)c.hidden);
  m->q_qkv.resize(c.layers);
  m->q_o.resize(c.layers);
  m->q_gu.resize(c.layers);
  m->q_down.resize(c.layers);
  auto fail = [&](w8a8_status s) {
    free_all(m);
    delete m;
    return s;
  };
#define W8A8_MTRY(expr)             \
  do {                              \
    w8a8_status s_ = (expr);        \
    if (s_ != W8A8_OK) return fail(s_); \
  } while (0)
  const int H = c.hidden, F = c.inter, Mx = c.max_tokens;
  W8A8_MTRY(cudaStreamCreateWithFlags(&m->st, cudaStreamNonBlocking) == cudaSuccess ? W8A8_OK : W8A8_ERR_CUDA);
  W8A8_MTRY(cudaEventCreateWithFlags(&m->ev_in, cudaEventDisableTiming) == cudaSuccess ? W8A8_OK : W8A8_ERR_CUDA);
  W8A8_MTRY(cudaEventCreateWithFlags(&m->ev_out, cudaEventDisableTiming) == cudaSuccess ? W8A8_OK : W8A8_ERR_CUDA);
  W8A8_MTRY(dalloc(m, &m->gu_bf16, (size_t)c.layers * 2 * F * H));
  W8A8_MTRY(dalloc(m, &m->stats, (size_t)c.layers * m->stats_stride() + H));
  W8A8_MTRY(dalloc(m, &m->r, (size_t)Mx * H));
  W8A8_MTRY(dalloc(m, &m->r2, (size_t)Mx * H));
  W8A8_MTRY(dalloc(m, &m->a, (size_t)Mx * H));
  W8A8_MTRY(dalloc(m, &m->qkv, (size_t)Mx * m->qkv_dim));
  W8A8_MTRY(dalloc(m, &m->q, (size_t)Mx * m->q_dim));
  W8A8_MTRY(dalloc(m, &m->o, (size_t)Mx * m->q_dim));
  W8A8_MTRY(dalloc(m, &m->y, (size_t)Mx * H));
  W8A8_MTRY(dalloc(m, &m->h, (size_t)Mx * F));
  W8A8_MTRY(dalloc(m, &m->kc, (size_t)c.layers * m->cache_layer_elems()));
  W8A8_MTRY(dalloc(m, &m->vc, (size_t)c.layers * m->cache_layer_elems()));
  const size_t rope = (size_t)c.max_seq * (c.head_dim / 2);
  W8A8_MTRY(dalloc(m, &m->cos_l, rope));
  W8A8_MTRY(dalloc(m, &m->sin_l, rope));
  W8A8_MTRY(dalloc(m, &m->cos_g, rope));
  W8A8_MTRY(dalloc(m, &m->sin_g, rope));
  W8A8_MTRY(dalloc(m, &m->d_pos, 4));
  W8A8_MTRY(dalloc(m, &m->d_tokens, (size_t)c.max_batch));
  W8A8_MTRY(dalloc(m, &m->d_logits, (size_t)c.max_batch * c.vocab));
  W8A8_MTRY(dalloc(m, &m->d_top1, (size_t)c.max_batch));
  // GEMM workspace: the largest of the model's linears at max_tokens rows (lm_head in chunks)
  size_t ws = 0;
  const int Mh = std::min(Mx, kHeadChunk);
  ws = std::max(ws, linear_ws(Mx, m->qkv_dim, H, true, d.sms).total);
  ws = std::max(ws, linear_ws(Mx, m->qkv_dim, H, false, d.sms).total);
  ws = std::max(ws, linear_ws(Mx, H, m->q_dim, true, d.sms).total);
  ws = std::max(ws, linear_ws(Mx, H, m->q_dim, false, d.sms).total);
  ws = std::max(ws, ffn_ws(Mx, H, F, d.sms).total);
  ws = std::max(ws, linear_ws(Mh, c.vocab, H, true, d.sms).total);
  ws = std::max(ws, linear_ws(Mh, c.vocab, H, false, d.sms).total);
  m->ws_bytes = ws;
  W8A8_MTRY(dalloc(m, reinterpret_cast<char**>(&m->ws), ws));
  W8A8_MTRY((size_t)Mx * c.n_kv * 4 <= 65536 ? W8A8_OK : W8A8_ERR_SHAPE);  // attention counters
  size_t aws = 0;
  for (int rows = 1; rows <= Mx; ++rows) {  // the split count depends on the row count: take the maximum
    AttnShape s{1, rows, c.n_q, c.n_kv, c.head_dim, c.max_seq, 0, 1.0f};
    aws = std::max(aws, attention_workspace_bytes(s, d.sms));
  }
  m->attn_ws_bytes = aws;
  W8A8_MTRY(dalloc(m, reinterpret_cast<char**>(&m->attn_ws), aws));
  W8A8_MTRY(dalloc(m, &m->pcodes, (size_t)c.max_tokens * H));
  W8A8_MTRY(dalloc(m, &m->psx, (size_t)c.max_tokens + 4));
  W8A8_MTRY(dalloc(m, &m->psum, (size_t)c.max_tokens + 4));
  cudaStream_t st = m->st;
  W8A8_MTRY(cudaMemsetAsync(m->ws, 0, W8A8_WS_RESERVED, st) == cudaSuccess ? W8A8_OK : W8A8_ERR_CUDA);
  W8A8_MTRY(cudaMemsetAsync(m->attn_ws, 0, aws, st) == cudaSuccess ? W8A8_OK : W8A8_ERR_CUDA);
  W8A8_MTRY(cudaMemsetAsync(m->stats, 0, ((size_t)c.layers * m->stats_stride() + H) * 4, st) == cudaSuccess
                ? W8A8_OK
                : W8A8_ERR_CUDA);
  W8A8_MTRY(launch_rope_table(m->cos_l, m->sin_l, c.max_seq, c.head_dim, c.rope_local, st));
  W8A8_MTRY(launch_rope_table(m->cos_g, m->sin_g, c.max_seq, c.head_dim, c.rope_global, st));
  for (int l = 0; l < c.layers; ++l)
    W8A8_MTRY(w8a8_interleave_gate_up(layers[l].wgate, layers[l].wup, F, H, m->gu_bf16 + (size_t)l * 2 * F * H, st));
  W8A8_MTRY(cudaStreamSynchronize(st) == cudaSuccess ? W8A8_OK : W8A8_ERR_CUDA);
#undef W8A8_MTRY
  *out = m;
  return W8A8_OK;
}

extern "C" w8a8_status w8a8_model_destroy(w8a8_model* m) {
  if (!m) return W8A8_OK;
  cudaStreamSynchronize(m->st);
  free_all(m);
  delete m;
  return W8A8_OK;
}

extern "C" w8a8_status w8a8_model_reset_calibration(w8a8_model* m, void* stream) {
  W8A8_CHECK_ARG(m, W8A8_ERR_INVALID_ARG, "null model");
  W8A8_CUDA(cudaMemsetAsync(m->stats, 0, ((size_t)m->cfg.layers * m->stats_stride() + m->cfg.hidden) * 4,
                            as_stream(stream)));
  return W8A8_OK;
}

extern "C" size_t w8a8_model_stats_count(const w8a8_model* m) {
  return m ? (size_t)m->cfg.layers * m->stats_stride() + m->cfg.hidden : 0;
}

extern "C" w8a8_status w8a8_model_get_stats(const w8a8_model* m, float* host_out) {
  W8A8_CHECK_ARG(m && host_out, W8A8_ERR_INVALID_ARG, "w8a8_model_get_stats: null argument");
  W8A8_CUDA(cudaDeviceSynchronize());
  W8A8_CUDA(cudaMemcpy(host_out, m->stats, w8a8_model_stats_count(m) * 4, cudaMemcpyDeviceToHost));
  return W8A8_OK;
}

extern "C" w8a8_status w8a8_model_set_stats(w8a8_model* m, const float* host_in) {
  W8A8_CHECK_ARG(m && host_in, W8A8_ERR_INVALID_ARG, "w8a8_model_set_stats: null argument");
  W8A8_CUDA(cudaDeviceSynchronize());
  W8A8_CUDA(cudaMemcpy(m->stats, host_in, w8a8_model_stats_count(m) * 4, cudaMemcpyHostToDevice));
  return W8A8_OK;
}

extern "C" w8a8_status w8a8_model_calibrate(w8a8_model* m, const int32_t* tokens, int B, int T, void* stream) {
  W8A8_TRY(check_call(m, B, T, 0));
  W8A8_CHECK_ARG(tokens && aligned16(tokens), W8A8_ERR_INVALID_ARG, "w8a8_model_calibrate: null or unaligned tokens");
  cudaStream_t st = as_stream(stream);
  W8A8_TRY(launch_set_int(m->d_pos, 0, st));
  return forward_core(m, tokens, B, T, nullptr, nullptr, true, st);
}

extern "C" w8a8_status w8a8_model_prepare(w8a8_model* m, float alpha, int smooth, void* stream) {
  W8A8_CHECK_ARG(m, W8A8_ERR_INVALID_ARG, "null model");
  const w8a8_model_cfg& c = m->cfg;
  const int H = c.hidden, F = c.inter;
  auto ensure = [&](QW& q, int n, int k) -> w8a8_status {
    if (q.wq) return W8A8_OK;
    W8A8_TRY(dalloc(m, &q.wq, (size_t)n * k));
    W8A8_TRY(dalloc(m, &q.wq_f16, (size_t)n * k));
    W8A8_TRY(dalloc(m, &q.s_w, (size_t)n));
    W8A8_TRY(dalloc(m, &q.delta, (size_t)k));
    W8A8_TRY(dalloc(m, &q.inv_delta, (size_t)k));
    return W8A8_OK;
  };
  for (int l = 0; l < c.layers; ++l) {
    W8A8_TRY(ensure(m->q_qkv[l], m->qkv_dim, H));
    W8A8_TRY(ensure(m->q_o[l], H, m->q_dim));
    W8A8_TRY(ensure(m->q_gu[l], 2 * F, H));
    W8A8_TRY(ensure(m->q_down[l], H, F));
  }
  W8A8_TRY(ensure(m->q_lm, c.vocab, H));
  for (int l = 0; l < c.layers; ++l) {
    const w8a8_layer_bf16& W = m->L[l];
    QW* q = &m->q_qkv[l];
    W8A8_TRY(w8a8_prepare_weights(W.wqkv, m->qkv_dim, H, m->stat_qkv(l), alpha, smooth, q->wq, q->s_w, q->delta,
                                  q->inv_delta, q->wq_f16, stream));
    q = &m->q_o[l];
    W8A8_TRY(w8a8_prepare_weights(W.wo, H, m->q_dim, m->stat_o(l), alpha, smooth, q->wq, q->s_w, q->delta,
                                  q->inv_delta, q->wq_f16, stream));
    q = &m->q_gu[l];
    W8A8_TRY(w8a8_prepare_gate_up(W.wgate, W.wup, F, H, m->stat_gu(l), alpha, smooth, q->wq, q->s_w, q->delta,
                                  q->inv_delta, q->wq_f16, stream));
    q = &m->q_down[l];
    W8A8_TRY(w8a8_prepare_weights(W.wdown, H, F, m->stat_down(l), alpha, smooth, q->wq, q->s_w, q->delta,
                                  q->inv_delta, q->wq_f16, stream));
  }
  W8A8_TRY(w8a8_prepare_weights(m->embed, c.vocab, H, m->stat_lm(), alpha, smooth, m->q_lm.wq, m->q_lm.s_w,
                                m->q_lm.delta, m->q_lm.inv_delta, m->q_lm.wq_f16, stream));
  m->prepared = true;
  ++m->prep_version;
  return W8A8_OK;
}

extern "C" w8a8_status w8a8_set_layer_precision(w8a8_model* m, int layer, int sublayer, int precision) {
  W8A8_CHECK_ARG(m, W8A8_ERR_INVALID_ARG, "null model");
  W8A8_CHECK_ARG(precision == W8A8_PREC_BF16 || precision == W8A8_PREC_W8A8, W8A8_ERR_INVALID_ARG,
                 "w8a8_set_layer_precision: precision %d", precision);
  W8A8_CHECK_ARG(precision == W8A8_PREC_BF16 || m->prepared, W8A8_ERR_INVALID_ARG,
                 "w8a8_set_layer_precision: W8A8 needs w8a8_model_prepare first");
  if (sublayer == W8A8_SUB_LM) {
    m->lm = precision;
    return W8A8_OK;
  }
  W8A8_CHECK_ARG(sublayer == W8A8_SUB_FFN || sublayer == W8A8_SUB_ATTN, W8A8_ERR_INVALID_ARG,
                 "w8a8_set_layer_precision: sublayer %d", sublayer);
  W8A8_CHECK_ARG(layer >= 0 && layer < m->cfg.layers, W8A8_ERR_INVALID_ARG, "w8a8_set_layer_precision: layer %d", layer);
  uint32_t& bits = sublayer == W8A8_SUB_FFN ? m->ffn_bits : m->attn_bits;
  if (precision == W8A8_PREC_W8A8)
    bits |= 1u << layer;
  else
    bits &= ~(1u << layer);
  return W8A8_OK;
}

extern "C" w8a8_status w8a8_set_mask(w8a8_model* m, uint32_t ffn_bits, uint32_t attn_bits, int lm) {
  W8A8_CHECK_ARG(m, W8A8_ERR_INVALID_ARG, "null model");
  const uint32_t all = m->cfg.layers >= 32 ? 0xFFFFFFFFu : ((1u << m->cfg.layers) - 1u);
  W8A8_CHECK_ARG((ffn_bits & ~all) == 0 && (attn_bits & ~all) == 0, W8A8_ERR_INVALID_ARG,
                 "w8a8_set_mask: bits beyond layer %d", m->cfg.layers - 1);
  W8A8_CHECK_ARG(m->prepared || (ffn_bits == 0 && attn_bits == 0 && lm == 0), W8A8_ERR_INVALID_ARG,
                 "w8a8_set_mask: W8A8 needs w8a8_model_prepare first");
  m->ffn_bits = ffn_bits;
  m->attn_bits = attn_bits;
  m->lm = lm ? 1 : 0;
  return W8A8_OK;
}

extern "C" w8a8_status w8a8_get_mask(const w8a8_model* m, uint32_t* ffn_bits, uint32_t* attn_bits, int* lm) {
  W8A8_CHECK_ARG(m && ffn_bits && attn_bits && lm, W8A8_ERR_INVALID_ARG, "w8a8_get_mask: null argument");
  *ffn_bits = m->ffn_bits;
  *attn_bits = m->attn_bits;
  *lm = m->lm;
  return W8A8_OK;
}

extern "C" w8a8_status w8a8_decoder_forward(w8a8_model* m, const int32_t* tokens, int B, int T, int start_pos,
                                            float* logits, int32_t* top1, void* stream) {
  W8A8_TRY(check_call(m, B, T, start_pos));
  W8A8_CHECK_ARG(tokens && top1, W8A8_ERR_INVALID_ARG, "w8a8_decoder_forward: null tokens or top1");
  W8A8_CHECK_ARG(aligned16(tokens) && aligned16(top1) && (!logits || aligned16(logits)), W8A8_ERR_ALIGN,
                 "w8a8_decoder_forward: pointers must be 16-byte aligned");
  cudaStream_t st = as_stream(stream);
  W8A8_TRY(launch_set_int(m->d_pos, start_pos, st));
  return forward_core(m, tokens, B, T, logits, top1, false, st);
}

extern "C" w8a8_status w8a8_decoder_decode_step(w8a8_model* m, const int32_t* tokens, int B, int pos, float* logits,
                                                int32_t* top1, void* stream) {
  W8A8_TRY(check_call(m, B, 1, pos));
  W8A8_CHECK_ARG(tokens && top1, W8A8_ERR_INVALID_ARG, "w8a8_decoder_decode_step: null tokens or top1");
  cudaStream_t user = as_stream(stream), st = m->st;
  W8A8_CUDA(cudaEventRecord(m->ev_in, user));
  W8A8_CUDA(cudaStreamWaitEvent(st, m->ev_in, 0));
  W8A8_CUDA(cudaMemcpyAsync(m->d_tokens, tokens, sizeof(int32_t) * B, cudaMemcpyDeviceToDevice, st));
  W8A8_TRY(launch_set_int(m->d_pos, pos, st));
  const int want_logits = logits != nullptr;
  if (m->trace_on) {  // traced steps run eagerly (a cached graph holds no trace copies)
    W8A8_TRY(forward_core(m, m->d_tokens, B, 1, want_logits ? m->d_logits : nullptr, m->d_top1, false, st));
    W8A8_CUDA(cudaMemcpyAsync(top1, m->d_top1, sizeof(int32_t) * B, cudaMemcpyDeviceToDevice, st));
    if (logits)
      W8A8_CUDA(cudaMemcpyAsync(logits, m->d_logits, sizeof(float) * B * (size_t)m->cfg.vocab,
                                cudaMemcpyDeviceToDevice, st));
    W8A8_CUDA(cudaEventRecord(m->ev_out, st));
    W8A8_CUDA(cudaStreamWaitEvent(user, m->ev_out, 0));
    return W8A8_OK;
  }
  const auto key = std::make_tuple(B, m->ffn_bits, m->attn_bits, m->lm | (m->prepared ? 2 : 0),
                                   m->prep_version, want_logits);
  auto it = m->graphs.find(key);
  if (it == m->graphs.end()) {
    // one eager step first: every lazily set kernel attribute exists before capture; it computes
    // exactly what the graph computes (same cache position, same outputs)
    W8A8_TRY(forward_core(m, m->d_tokens, B, 1, want_logits ? m->d_logits : nullptr, m->d_top1, false, st));
    cudaGraph_t g = nullptr;
    W8A8_CUDA(cudaStreamBeginCapture(st, cudaStreamCaptureModeThreadLocal));
    const w8a8_status s = forward_core(m, m->d_tokens, B, 1, want_logits ? m->d_logits : nullptr, m->d_top1, false, st);
    const cudaError_t e = cudaStreamEndCapture(st, &g);
    W8A8_TRY(s);
    W8A8_CUDA(e);
    int kernels = 0;
    size_t n_nodes = 0;
    if (cudaGraphGetNodes(g, nullptr, &n_nodes) == cudaSuccess) {
      std::vector<cudaGraphNode_t> nodes(n_nodes);
      if (cudaGraphGetNodes(g, nodes.data(), &n_nodes) == cudaSuccess)
        for (cudaGraphNode_t nd : nodes) {
          cudaGraphNodeType t;
          if (cudaGraphNodeGetType(nd, &t) == cudaSuccess && t == cudaGraphNodeTypeKernel) ++kernels;
        }
    }
    cudaGraphExec_t exec = nullptr;
    const cudaError_t ei = cudaGraphInstantiate(&exec, g, 0);
    cudaGraphDestroy(g);
    W8A8_CUDA(ei);
    it = m->graphs.emplace(key, w8a8_model::Graph{exec, kernels}).first;
  }
  W8A8_CUDA(cudaGraphLaunch(it->second.exec, st));
  W8A8_CUDA(cudaMemcpyAsync(top1, m->d_top1, sizeof(int32_t) * B, cudaMemcpyDeviceToDevice, st));
  if (logits)
    W8A8_CUDA(cudaMemcpyAsync(logits, m->d_logits, sizeof(float) * B * (size_t)m->cfg.vocab, cudaMemcpyDeviceToDevice,
                              st));
  W8A8_CUDA(cudaEventRecord(m->ev_out, st));
  W8A8_CUDA(cudaStreamWaitEvent(user, m->ev_out, 0));
  return W8A8_OK;
}

extern "C" w8a8_status w8a8_model_set_trace(w8a8_model* m, const w8a8_trace* t) {
  W8A8_CHECK_ARG(m, W8A8_ERR_INVALID_ARG, "w8a8_model_set_trace: null model");
  if (!t) {
    m->trace_on = false;
    m->trace = w8a8_trace{};
    return W8A8_OK;
  }
  W8A8_CHECK_ARG(t->max_rows > 0, W8A8_ERR_INVALID_ARG, "w8a8_model_set_trace: max_rows must be positive");
  const void* ptrs[] = {t->a_in, t->qkv, t->attn, t->y_o, t->a_ffn, t->h, t->y_f, t->r, t->a_fin};
  for (const void* p : ptrs)
    W8A8_CHECK_ARG(!p || aligned16(p), W8A8_ERR_ALIGN, "w8a8_model_set_trace: buffers must be 16-byte aligned");
  m->trace = *t;
  m->trace_on = true;
  return W8A8_OK;
}

extern "C" w8a8_status w8a8_model_decode_kernels(const w8a8_model* m, int B, int want_logits, int* kernels) {
  W8A8_CHECK_ARG(m && kernels, W8A8_ERR_INVALID_ARG, "w8a8_model_decode_kernels: null argument");
  const auto key = std::make_tuple(B, m->ffn_bits, m->attn_bits, m->lm | (m->prepared ? 2 : 0),
                                   m->prep_version, want_logits ? 1 : 0);
  const auto it = m->graphs.find(key);
  W8A8_CHECK_ARG(it != m->graphs.end(), W8A8_ERR_INVALID_ARG,
                 "w8a8_model_decode_kernels: no decode step of B=%d under this mask yet", B);
  *kernels = it->second.kernels + 1;  // + the position update launched beside the graph
  return W8A8_OK;
}

extern "C" w8a8_status w8a8_token_nll(const float* logits, const int32_t* targets, int M, int V, float* nll,
                                      void* stream) {
  W8A8_CHECK_ARG(M >= 0 && V > 0, W8A8_ERR_INVALID_ARG, "w8a8_token_nll: bad size");
  if (M == 0) return W8A8_OK;
  W8A8_CHECK_ARG(logits && targets && nll, W8A8_ERR_INVALID_ARG, "w8a8_token_nll: null pointer");
  W8A8_TRY(check_device());
  nll_kernel<<<M, 256, 0, as_stream(stream)>>>(logits, targets, V, nll);
  W8A8_LAUNCH_CHECK();
  return W8A8_OK;
}

extern "C" int w8a8_choose_mask(const float* latency, const float* top1, const float* ppl_delta, const int32_t* n_int8,
                                int n, float min_top1, float max_ppl_delta) {
  int best = -1;
  for (int i = 0; i < n; ++i) {
    if (!(top1[i] >= min_top1 && ppl_delta[i] <= max_ppl_delta)) continue;
    if (best < 0 || latency[i] < latency[best] || (latency[i] == latency[best] && n_int8[i] < n_int8[best])) best = i;
  }
  return best;
}

namespace {

// The measurements both allocators make (Problem Statement; Combined Configurations): a mask's
// quality against the all-bf16 decoder on a teacher-forced evaluation stream (Top-1 agreement over
// the positions with a next token, and the perplexity ratio minus one), and its decode latency
// (median over reps of the mean ms per step of decode_steps CUDA-graph steps after a prefill).
// Buffers live from init() to the destructor; the model's mask is whatever was set last.
struct AllocRun {
  w8a8_model* m;
  const int32_t* eval_tokens;
  int eval_B, eval_T, decode_B, prefill_T, decode_steps, reps;
  void* stream;
  cudaStream_t st;
  int V = 0, Me = 0, Mp = 0;
  float *logits = nullptr, *nll = nullptr;
  int32_t *targets = nullptr, *top_ref = nullptr, *top_c = nullptr, *ptok = nullptr, *dtok = nullptr;
  std::vector<void*> tmp;
  std::vector<float> nll_h;
  std::vector<int32_t> top_h, ref_h;
  double ref_nll = 0.0;
  cudaEvent_t e0 = nullptr, e1 = nullptr;

  ~AllocRun() {
    cudaStreamSynchronize(st);
    for (void* p : tmp) cudaFree(p);
    if (e0) cudaEventDestroy(e0);
    if (e1) cudaEventDestroy(e1);
  }
  w8a8_status talloc(void** p, size_t bytes) {
    W8A8_CUDA(cudaMalloc(p, std::max<size_t>(bytes, 16)));
    tmp.push_back(*p);
    return W8A8_OK;
  }
  double mean_nll() const {
    double sum = 0.0;
    int n = 0;
    for (int b = 0; b < eval_B; ++b)
      for (int t = 0; t + 1 < eval_T; ++t, ++n) sum += nll_h[b * eval_T + t];
    return sum / n;
  }
  w8a8_status forward_eval(int32_t* top_out, double* mnll) {
    W8A8_TRY(w8a8_decoder_forward(m, eval_tokens, eval_B, eval_T, 0, logits, top_out, stream));
    W8A8_TRY(w8a8_token_nll(logits, targets, Me, V, nll, stream));
    W8A8_CUDA(cudaMemcpyAsync(nll_h.data(), nll, (size_t)Me * 4, cudaMemcpyDeviceToHost, st));
    W8A8_CUDA(cudaStreamSynchronize(st));
    *mnll = mean_nll();
    return W8A8_OK;
  }
  // buffers, the shifted targets, the prefill tokens and the all-bf16 reference (sets that mask)
  w8a8_status init() {
    st = as_stream(stream);
    V = m->cfg.vocab;
    Me = eval_B * eval_T;
    Mp = decode_B * prefill_T;
    W8A8_TRY(talloc((void**)&logits, (size_t)Me * V * 4));
    W8A8_TRY(talloc((void**)&nll, (size_t)Me * 4));
    W8A8_TRY(talloc((void**)&targets, (size_t)Me * 4));
    W8A8_TRY(talloc((void**)&top_ref, (size_t)Me * 4));
    W8A8_TRY(talloc((void**)&top_c, (size_t)std::max(Me, m->cfg.max_tokens) * 4));
    W8A8_TRY(talloc((void**)&ptok, (size_t)Mp * 4));
    W8A8_TRY(talloc((void**)&dtok, (size_t)decode_B * 4));
    W8A8_CUDA(cudaEventCreate(&e0));
    W8A8_CUDA(cudaEventCreate(&e1));
    nll_h.resize(Me);
    top_h.resize(Me);
    ref_h.resize(Me);
    shift_targets_kernel<<<(Me + 255) / 256, 256, 0, st>>>(eval_tokens, eval_B, eval_T, targets);
    W8A8_LAUNCH_CHECK();
    fill_tokens_kernel<<<(Mp + 255) / 256, 256, 0, st>>>(ptok, Mp, V);
    W8A8_LAUNCH_CHECK();
    W8A8_TRY(w8a8_set_mask(m, 0, 0, 0));
    W8A8_TRY(forward_eval(top_ref, &ref_nll));
    W8A8_CUDA(cudaMemcpy(ref_h.data(), top_ref, (size_t)Me * 4, cudaMemcpyDeviceToHost));
    return W8A8_OK;
  }
  w8a8_status quality(const w8a8_mask& c, float* top1, float* ppl_delta) {
    W8A8_TRY(w8a8_set_mask(m, c.ffn_bits, c.attn_bits, c.lm));
    double cn = 0.0;
    W8A8_TRY(forward_eval(top_c, &cn));
    W8A8_CUDA(cudaMemcpy(top_h.data(), top_c, (size_t)Me * 4, cudaMemcpyDeviceToHost));
    int agree = 0, cnt = 0;
    for (int b = 0; b < eval_B; ++b)
      for (int t = 0; t + 1 < eval_T; ++t, ++cnt) agree += top_h[b * eval_T + t] == ref_h[b * eval_T + t];
    *top1 = (float)agree / (float)cnt;
    *ppl_delta = (float)(std::exp(cn) / std::exp(ref_nll) - 1.0);
    return W8A8_OK;
  }
  // prefill, then decode steps from CUDA graphs fed by their own top-1 (greedy)
  w8a8_status latency(const w8a8_mask& c, float* ms_per_step) {
    W8A8_TRY(w8a8_set_mask(m, c.ffn_bits, c.attn_bits, c.lm));
    std::vector<float> runs;
    for (int r = 0; r < reps; ++r) {
      // prefill in chunks of at most max_tokens rows (the KV cache carries the earlier chunks)
      const int chunk = std::max(1, m->cfg.max_tokens / decode_B);
      for (int t0 = 0; t0 < prefill_T; t0 += chunk) {
        const int tl = std::min(chunk, prefill_T - t0);
        W8A8_TRY(w8a8_decoder_forward(m, ptok + (size_t)decode_B * t0, decode_B, tl, t0, nullptr, top_c, stream));
      }
      W8A8_CUDA(cudaMemcpyAsync(dtok, top_c, 4 * (size_t)decode_B, cudaMemcpyDeviceToDevice, st));
      // warm the graph of this mask outside the timed region
      W8A8_TRY(w8a8_decoder_decode_step(m, dtok, decode_B, prefill_T, nullptr, dtok, stream));
      W8A8_CUDA(cudaEventRecord(e0, st));
      for (int s = 0; s < decode_steps; ++s)
        W8A8_TRY(w8a8_decoder_decode_step(m, dtok, decode_B, prefill_T + s, nullptr, dtok, stream));
      W8A8_CUDA(cudaEventRecord(e1, st));
      W8A8_CUDA(cudaEventSynchronize(e1));
      float ms = 0.0f;
      W8A8_CUDA(cudaEventElapsedTime(&ms, e0, e1));
      runs.push_back(ms / (float)decode_steps);
    }
    std::sort(runs.begin(), runs.end());
    *ms_per_step = runs[runs.size() / 2];
    return W8A8_OK;
  }
};

w8a8_status check_alloc_args(w8a8_model* m, const int32_t* eval_tokens, int eval_B, int eval_T, int decode_B,
                             int prefill_T, int decode_steps, int reps, const char* who) {
  W8A8_CHECK_ARG(m && eval_tokens, W8A8_ERR_INVALID_ARG, "%s: null argument", who);
  W8A8_CHECK_ARG(m->prepared, W8A8_ERR_INVALID_ARG, "%s: w8a8_model_prepare first", who);
  W8A8_TRY(check_call(m, eval_B, eval_T, 0));
  W8A8_CHECK_ARG(decode_B > 0 && decode_B <= m->cfg.max_batch && prefill_T > 0, W8A8_ERR_SHAPE,
                 "%s: decode_B %d / prefill_T %d", who, decode_B, prefill_T);
  W8A8_TRY(check_call(m, decode_B, 1, prefill_T + decode_steps - 1));
  W8A8_CHECK_ARG(eval_T >= 2 && decode_steps > 0 && reps > 0, W8A8_ERR_INVALID_ARG,
                 "%s: eval_T >= 2, decode_steps > 0, reps > 0", who);
  return W8A8_OK;
}

}  // namespace

extern "C" w8a8_status w8a8_allocate_mask(w8a8_model* m, const w8a8_alloc_opts* o, w8a8_alloc_report* rep,
                                          void* stream) {
  W8A8_CHECK_ARG(m && o && rep && o->candidates && o->n_candidates > 0 && rep->latency_ms && rep->top1 &&
                     rep->ppl_delta,
                 W8A8_ERR_INVALID_ARG, "w8a8_allocate_mask: null argument");
  W8A8_TRY(check_alloc_args(m, o->eval_tokens, o->eval_B, o->eval_T, o->decode_B, o->prefill_T, o->decode_steps,
                            o->reps, "w8a8_allocate_mask"));
  const uint32_t saved_ffn = m->ffn_bits, saved_attn = m->attn_bits;
  const int saved_lm = m->lm;
  std::vector<int32_t> n8(o->n_candidates);
  w8a8_status status = W8A8_OK;
  {
    AllocRun run{m, o->eval_tokens, o->eval_B, o->eval_T, o->decode_B, o->prefill_T, o->decode_steps, o->reps, stream};
    status = run.init();
    for (int i = 0; i < o->n_candidates && status == W8A8_OK; ++i) {
      const w8a8_mask& c = o->candidates[i];
      n8[i] = __builtin_popcount(c.ffn_bits) + __builtin_popcount(c.attn_bits) + (c.lm ? 1 : 0);
      status = run.quality(c, &rep->top1[i], &rep->ppl_delta[i]);
      if (status == W8A8_OK) status = run.latency(c, &rep->latency_ms[i]);
    }
  }
  if (status != W8A8_OK) {
    m->ffn_bits = saved_ffn;
    m->attn_bits = saved_attn;
    m->lm = saved_lm;
    return status;
  }
  rep->chosen = w8a8_choose_mask(rep->latency_ms, rep->top1, rep->ppl_delta, n8.data(), o->n_candidates, o->min_top1,
                                 o->max_ppl_delta);
  if (rep->chosen >= 0) {
    const w8a8_mask& c = o->candidates[rep->chosen];
    return w8a8_set_mask(m, c.ffn_bits, c.attn_bits, c.lm);
  }
  return w8a8_set_mask(m, 0, 0, 0);
}

extern "C" int w8a8_greedy_order(const float* gain_ms, const float* top1, const float* ppl_delta, int n,
                                 float min_top1, float max_ppl_delta, int32_t* order) {
  if (!gain_ms || !top1 || !ppl_delta || !order || n <= 0) return 0;
  const double t_scale = std::max(1e-6, 1.0 - (double)min_top1), p_scale = std::max(1e-6, (double)max_ppl_delta);
  std::vector<std::pair<double, int>> keep;
  for (int i = 0; i < n; ++i) {
    if (!(gain_ms[i] > 0.0f) || !(top1[i] >= min_top1 && ppl_delta[i] <= max_ppl_delta)) continue;
    const double cost = std::max(0.0, 1.0 - (double)top1[i]) / t_scale + std::max(0.0, (double)ppl_delta[i]) / p_scale;
    keep.emplace_back((double)gain_ms[i] / (cost + 1e-3), i);
  }
  std::stable_sort(keep.begin(), keep.end(), [](const std::pair<double, int>& a, const std::pair<double, int>& b) {
    return a.first > b.first;  // stable: equal scores keep the lower index first
  });
  for (size_t k = 0; k < keep.size(); ++k) order[k] = keep[k].second;
  return (int)keep.size();
}

extern "C" w8a8_status w8a8_allocate_layers(w8a8_model* m, const w8a8_layer_alloc_opts* o,
                                            w8a8_layer_alloc_report* rep, void* stream) {
  W8A8_CHECK_ARG(m && o && rep && rep->gain_ms && rep->top1 && rep->ppl_delta && rep->order, W8A8_ERR_INVALID_ARG,
                 "w8a8_allocate_layers: null argument");
  W8A8_TRY(check_alloc_args(m, o->eval_tokens, o->eval_B, o->eval_T, o->decode_B, o->prefill_T, o->decode_steps,
                            o->reps, "w8a8_allocate_layers"));
  const int L = m->cfg.layers, n = 2 * L + 1;
  auto single = [&](int i) {
    w8a8_mask c{0u, 0u, 0};
    if (i < L) c.ffn_bits = 1u << i;
    else if (i < 2 * L) c.attn_bits = 1u << (i - L);
    else c.lm = 1;
    return c;
  };
  const uint32_t saved_ffn = m->ffn_bits, saved_attn = m->attn_bits;
  const int saved_lm = m->lm;
  w8a8_mask chosen{0u, 0u, 0};
  w8a8_status status = W8A8_OK;
  {
    AllocRun run{m, o->eval_tokens, o->eval_B, o->eval_T, o->decode_B, o->prefill_T, o->decode_steps, o->reps, stream};
    status = run.init();
    if (status == W8A8_OK) status = run.latency(chosen, &rep->base_ms);
    for (int i = 0; i < n && status == W8A8_OK; ++i) {
      float ms = 0.0f;
      status = run.quality(single(i), &rep->top1[i], &rep->ppl_delta[i]);
      if (status == W8A8_OK) status = run.latency(single(i), &ms);
      rep->gain_ms[i] = rep->base_ms - ms;
    }
    rep->n_order = 0;
    rep->n_accepted = 0;
    rep->chosen_top1 = 1.0f;
    rep->chosen_ppl_delta = 0.0f;
    if (status == W8A8_OK)
      rep->n_order = w8a8_greedy_order(rep->gain_ms, rep->top1, rep->ppl_delta, n, o->min_top1, o->max_ppl_delta,
                                       rep->order);
    for (int k = 0; k < rep->n_order && status == W8A8_OK; ++k) {
      const w8a8_mask s1 = single(rep->order[k]);
      const w8a8_mask trial{chosen.ffn_bits | s1.ffn_bits, chosen.attn_bits | s1.attn_bits, chosen.lm | s1.lm};
      float t1 = 0.0f, pd = 0.0f;
      status = run.quality(trial, &t1, &pd);
      if (status == W8A8_OK && t1 >= o->min_top1 && pd <= o->max_ppl_delta) {
        chosen = trial;
        rep->chosen_top1 = t1;
        rep->chosen_ppl_delta = pd;
        ++rep->n_accepted;
      }
    }
    if (status == W8A8_OK) {
      if (rep->n_accepted > 0) status = run.latency(chosen, &rep->chosen_ms);
      else rep->chosen_ms = rep->base_ms;
    }
  }
  if (status != W8A8_OK) {
    m->ffn_bits = saved_ffn;
    m->attn_bits = saved_attn;
    m->lm = saved_lm;
    return status;
  }
  rep->chosen = chosen;
  return w8a8_set_mask(m, chosen.ffn_bits, chosen.attn_bits, chosen.lm);
}

extern "C" w8a8_status w8a8_sqnr_db(const float* y_ref, const float* y_q, size_t n, double* out_db, void* stream) {
  W8A8_CHECK_ARG(y_ref && y_q && out_db, W8A8_ERR_INVALID_ARG, "w8a8_sqnr_db: null pointer");
  W8A8_CHECK_ARG(n > 0, W8A8_ERR_INVALID_ARG, "w8a8_sqnr_db: no elements");
  W8A8_TRY(check_device());
  cudaStream_t st = as_stream(stream);
  double* part = nullptr;
  W8A8_CUDA(cudaMalloc(&part, sizeof(double) * 2 * kSqnrBlocks));
  sqnr_partial_kernel<<<kSqnrBlocks, 256, 0, st>>>(y_ref, y_q, n, part);
  std::vector<double> h(2 * kSqnrBlocks);
  cudaError_t e = cudaGetLastError();
  if (e == cudaSuccess) e = cudaMemcpyAsync(h.data(), part, sizeof(double) * h.size(), cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  cudaFree(part);
  W8A8_CUDA(e);
  double sig = 0.0, err = 0.0;
  for (int b = 0; b < kSqnrBlocks; ++b) {
    sig += h[2 * b];
    err += h[2 * b + 1];
  }
  *out_db = err > 0.0 ? 10.0 * std::log10(sig / err) : INFINITY;
  return W8A8_OK;
}

extern "C" w8a8_status w8a8_sqnr_profile(w8a8_model* m, const int32_t* tokens, int B, int T, const w8a8_mask* mask,
                                         int isolated, float* layer_db, float* lm_db, void* stream) {
  W8A8_CHECK_ARG(m && tokens && mask && layer_db && lm_db, W8A8_ERR_INVALID_ARG, "w8a8_sqnr_profile: null argument");
  W8A8_CHECK_ARG(m->prepared, W8A8_ERR_INVALID_ARG, "w8a8_sqnr_profile: w8a8_model_prepare first");
  W8A8_CHECK_ARG(T >= 2, W8A8_ERR_SHAPE, "w8a8_sqnr_profile: T >= 2 (a prefill)");
  W8A8_TRY(check_call(m, B, T, 0));
  const int L = m->cfg.layers, M = B * T, H = m->cfg.hidden, V = m->cfg.vocab;
  cudaStream_t st = as_stream(stream);
  const uint32_t saved_ffn = m->ffn_bits, saved_attn = m->attn_bits;
  const int saved_lm = m->lm;
  std::vector<void*> tmp;
  auto talloc = [&](void** p, size_t bytes) -> w8a8_status {
    W8A8_CUDA(cudaMalloc(p, bytes));
    tmp.push_back(*p);
    return W8A8_OK;
  };
  float *h_ref = nullptr, *h_q = nullptr, *lg_ref = nullptr, *lg_q = nullptr;
  int32_t* top = nullptr;
  const size_t hl = (size_t)M * H;
  auto run = [&](uint32_t f, uint32_t a, int l, float* hcap, float* lg) -> w8a8_status {
    W8A8_TRY(w8a8_set_mask(m, f, a, l));
    m->capture = hcap;
    const w8a8_status s = w8a8_decoder_forward(m, tokens, B, T, 0, lg, top, stream);
    m->capture = nullptr;
    return s;
  };
  auto sqnr = [&](const float* r, const float* q, size_t n, float* out) -> w8a8_status {
    double db = 0.0;
    W8A8_TRY(w8a8_sqnr_db(r, q, n, &db, stream));
    *out = (float)db;
    return W8A8_OK;
  };
  w8a8_status s = W8A8_OK;
  do {
    if ((s = talloc((void**)&h_ref, sizeof(float) * hl * L)) != W8A8_OK) break;
    if ((s = talloc((void**)&h_q, sizeof(float) * hl * L)) != W8A8_OK) break;
    if ((s = talloc((void**)&lg_ref, sizeof(float) * (size_t)M * V)) != W8A8_OK) break;
    if ((s = talloc((void**)&lg_q, sizeof(float) * (size_t)M * V)) != W8A8_OK) break;
    if ((s = talloc((void**)&top, sizeof(int32_t) * (size_t)std::max(M, 4))) != W8A8_OK) break;
    if ((s = run(0u, 0u, 0, h_ref, lg_ref)) != W8A8_OK) break;  // the reference: all bf16
    if (!isolated) {  // one pass under the whole mask: errors accumulate
      if ((s = run(mask->ffn_bits, mask->attn_bits, mask->lm, h_q, lg_q)) != W8A8_OK) break;
      for (int l = 0; l < L && s == W8A8_OK; ++l) s = sqnr(h_ref + l * hl, h_q + l * hl, hl, &layer_db[l]);
      if (s == W8A8_OK) s = sqnr(lg_ref, lg_q, (size_t)M * V, lm_db);
      break;
    }
    // isolated: each layer's quantised sublayers alone, so the layer takes the reference input
    for (int l = 0; l < L && s == W8A8_OK; ++l) {
      const uint32_t f = mask->ffn_bits & (1u << l), a = mask->attn_bits & (1u << l);
      if (!f && !a) {
        layer_db[l] = INFINITY;  // nothing quantised: the reference output itself
        continue;
      }
      if ((s = run(f, a, 0, h_q, nullptr)) == W8A8_OK) s = sqnr(h_ref + l * hl, h_q + l * hl, hl, &layer_db[l]);
    }
    if (s != W8A8_OK) break;
    if (mask->lm) {
      if ((s = run(0u, 0u, 1, h_q, lg_q)) == W8A8_OK) s = sqnr(lg_ref, lg_q, (size_t)M * V, lm_db);
    } else {
      *lm_db = INFINITY;
    }
  } while (0);
  cudaStreamSynchronize(st);
  for (void* p : tmp) cudaFree(p);
  m->capture = nullptr;
  m->ffn_bits = saved_ffn;
  m->attn_bits = saved_attn;
  m->lm = saved_lm;
  return s;
}
