/*
 * w8a8.h - C ABI of libw8a8.so: the W8A8 SmoothQuant hot path of
 * "A Method for Layer Bit-Width Allocation in LLM Quantization via Performance Maximization
 * Under a Quality-Degradation Constraint" (arXiv 2608.28003) on one GB300 (sm_103a).
 *
 * Conventions (every entry point):
 *   - Returns a w8a8_status.  Nothing is thrown across the ABI.  On a non-OK status,
 *     w8a8_last_error() returns a message for the calling thread.
 *   - Tensors are caller-owned DEVICE pointers unless a parameter says "host".  The library
 *     allocates no device memory on any compute entry point; scratch space comes from a
 *     caller-provided workspace whose size a *_workspace_size query returns.
 *   - bf16 and fp16 tensors are passed as uint16_t bit patterns.  Matrices are row-major.  A
 *     weight [N, K] has one row per output channel i and one column per input channel j
 *     (the paper's W_{i,j}).
 *   - `stream` is a cudaStream_t passed as void* (NULL = the legacy default stream).  Compute
 *     calls are asynchronous on it.  Errors found on the host (arguments, shapes,
 *     alignment) are reported before anything is launched.  Errors of a launch are
 *     reported as W8A8_ERR_CUDA.
 *   - Alignment: every tensor pointer must be 16-byte aligned, and every K (input channels)
 *     must be a multiple of 16.  Otherwise the call returns W8A8_ERR_ALIGN or W8A8_ERR_SHAPE.
 *   - Workspace: its first W8A8_WS_RESERVED bytes hold split-K arrival counters.  They must be
 *     zero before the workspace is first used (cudaMemset once after allocating).  Every call
 *     leaves them zero again when it completes.  A workspace must not be used by two calls
 *     that can run concurrently.
 *   - Exactness: INT8 codes and INT32 accumulators are exact.  Every step that decides an INT8
 *     code runs in IEEE fp32 with round-to-nearest-even, in the order documented below.
 */
#ifndef W8A8_H
#define W8A8_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  W8A8_OK = 0,
  W8A8_ERR_INVALID_ARG = 1, /* a required pointer is NULL, a size is negative, an enum is out of range */
  W8A8_ERR_SHAPE = 2,       /* a shape the entry point does not support (K % 16 != 0, a limit exceeded) */
  W8A8_ERR_ALIGN = 3,       /* a tensor pointer is not 16-byte aligned */
  W8A8_ERR_CUDA = 4,        /* a CUDA runtime call or a kernel launch failed */
  W8A8_ERR_UNSUPPORTED = 5, /* the current device is not an sm_103 GPU, or the feature is not built */
  W8A8_ERR_TIMEOUT = 6,     /* a bounded device-side wait gave up (the kernel returned early) */
  W8A8_ERR_WORKSPACE = 7    /* the workspace is NULL or smaller than the size query returned */
} w8a8_status;

enum { W8A8_PREC_BF16 = 0, W8A8_PREC_W8A8 = 1 };

#define W8A8_WS_RESERVED 65536 /* bytes of counters at the start of every workspace */
#define W8A8_MAX_K 65536       /* largest K (input channels) any entry point accepts */

/* Version of this ABI (incremented on incompatible changes). */
int w8a8_abi_version(void);

/* Message for the last non-OK status returned on the calling thread ("" if none). */
const char* w8a8_last_error(void);

/* Waits for `stream`, then reads and clears the workspace's device error word.  Kernels never
 * wait without a bound: a wait that gives up (about 2 s) sets a bit of this word, skips the rest
 * of its work and returns, so the context stays usable.  Returns W8A8_ERR_TIMEOUT if any bit was
 * set since the last check (the outputs of the calls in between are then undefined), W8A8_OK
 * otherwise.  This call is synchronous. */
w8a8_status w8a8_workspace_check(void* workspace, void* stream);

/* Measurement aid: the calling thread's next weight-streaming GEMM launch (inside w8a8_linear,
 * w8a8_linear_bf16, w8a8_ffn_block or w8a8_lm_head) records `start_event` (a cudaEvent_t) on its
 * stream just before the kernel and `stop_event` just after it, then forgets both.  The events
 * bracket the GEMM kernel alone, not the per-token quantiser launched before it.  Both or
 * neither (NULL, NULL clears a pending request). */
w8a8_status w8a8_set_kernel_events(void* start_event, void* stop_event);

/* Measurement aid (no counterpart in the paper; not a compute entry point: it allocates and frees a
 * small sink buffer and synchronises `stream`): the sustained rate, in TOPS (two ops per
 * multiply-add), of an exact integer route for the INT8 GEMM on the current GPU, measured by one
 * launch over every SM with CUDA events: route 0 = dp4a, 1 = mma.sync m16n8k32 s8 x s8 -> s32,
 * 2 = mma.sync m16n8k16 fp16 x fp16 -> fp32 (the decode GEMV's tensor-core path on INT8 codes
 * carried as fp16).  The tcgen05 route's rate is the fp16 / bf16 tensor rate (kind::f16). */
w8a8_status w8a8_route_peak(int route, double* tops, void* stream);

/* ---------------------------------------------------------------------------------------
 * Prepared W8A8 weight of one linear (produced by w8a8_prepare_weights /
 * w8a8_prepare_gate_up, owned by the caller).
 *   wq        [n, k] INT8 codes of the smoothed weight, in [-127, 127]          (Eq. si, what-ffn)
 *   s_w       [n]    per-output-channel scale s_i^W = max_j |W_hat_ij| / 127      (Eq. si)
 *   inv_delta [k]    1 / delta_j, the activation side of the smoothing            (Eq. xhat-lmhead)
 *   wq_f16    [n, k] nullable: the same codes as fp16 values (exact).  Linears with large
 *                    token counts use it as the tensor-core operand.
 * ------------------------------------------------------------------------------------- */
typedef struct {
  int32_t n, k;
  const int8_t* wq;
  const float* s_w;
  const float* inv_delta;
  const uint16_t* wq_f16;
} w8a8_qweight;

/* Optional per-call debug outputs of w8a8_linear (each pointer nullable). */
typedef struct {
  int8_t* xq;   /* [M, K] INT8 activation codes (Eq. xint8) */
  float* s_x;   /* [M]    per-token scale s_t^x (Eq. stx) */
  int32_t* acc; /* [M, N] INT32 accumulator sum_j xq_tj * wq_ij (Eq. gemm-final) */
} w8a8_debug;

/* ------------------------------------------------------------------ calibration (offline)
 * Running per-channel maximum of |X| over calibration tokens, the max_t |X_{t,j}| of
 * Eq. delta-attn / delta-lmhead (LM Head section: collected by a forward hook).
 *   X       [T, K] bf16 activations at a linear's input
 *   absmax  [K] fp32, in/out: absmax[j] = max(absmax[j], max_t |X_tj|).  Zero it before the
 *           first batch.  Entries must be non-negative.
 * T == 0 is a no-op. */
w8a8_status w8a8_act_absmax(const uint16_t* X, int T, int K, float* absmax, void* stream);

/* ------------------------------------------------------------ weight preparation (offline)
 * SmoothQuant preparation of one linear (Eq. delta-attn / delta-lmhead, what-lmhead, then
 * Eq. si / what-ffn on the smoothed rows):
 *   delta_j   = max_t|X_tj|^alpha / max_i|W_ij|^(1-alpha).  For alpha == 0.5 this is
 *               fl32(sqrt(ax_j)) / fl32(sqrt(aw_j)) exactly rounded.  Other alpha values are
 *               evaluated in fp64 and rounded once.  delta_j = 1 where either statistic is 0.
 *   inv_delta = fl32(1 / delta)
 *   W_hat_ij  = fl32(W_ij * delta_j);  m_i = max_j |W_hat_ij|;  s_w_i = fl32(m_i / 127)
 *   wq_ij     = clamp(rint(fl32(W_hat_ij * fl32(127 / m_i))), -127, 127)  (0 for an all-zero row)
 * W [N, K] bf16; act_absmax [K] from w8a8_act_absmax.  smooth == 0 gives delta = 1 (the
 * paper's no-smoothing ablation).  Outputs (caller-owned): wq [N, K], s_w [N], delta [K],
 * inv_delta [K].  wq_f16 (nullable) receives the codes as fp16. */
w8a8_status w8a8_prepare_weights(const uint16_t* W, int N, int K, const float* act_absmax,
                                 float alpha, int smooth, int8_t* wq, float* s_w, float* delta,
                                 float* inv_delta, uint16_t* wq_f16, void* stream);

/* Fused gate/up preparation for the FFN block (FFN section).  gate and up share their input, so
 * one delta is computed over the column maxima of BOTH matrices (2F rows).  Output row p of the
 * fused [2F, H] matrix holds, for block q = p / 16 and r = p % 16:
 *   r < 8 : gate row 8q + r        r >= 8 : up row 8q + r - 8
 * (blocks of 8 gate rows then the 8 matching up rows), and s_w follows the same order.
 * F must be a multiple of 8. */
w8a8_status w8a8_prepare_gate_up(const uint16_t* W_gate, const uint16_t* W_up, int F, int H,
                                 const float* act_absmax, float alpha, int smooth, int8_t* wq,
                                 float* s_w, float* delta, float* inv_delta, uint16_t* wq_f16,
                                 void* stream);

/* The same 8-row interleave for a bf16 pass-through gate/up pair: out [2F, H] bf16. */
w8a8_status w8a8_interleave_gate_up(const uint16_t* W_gate, const uint16_t* W_up, int F, int H,
                                    uint16_t* out, void* stream);

/* ------------------------------------------------------ per-token activation quantisation
 * Dynamic per-token quantisation of the smoothed input (Eq. xhat-lmhead, stx, xint8):
 *   x_hat_tj = fl32(x_tj * inv_delta_j);  m_t = max_j |x_hat_tj|;  s_x_t = fl32(m_t / 127)
 *   xq_tj    = clamp(rint(fl32(x_hat_tj * fl32(127 / m_t))), -127, 127)   (0 for a zero row)
 * X [M, K] bf16.  Outputs: xq [M, K] int8 (nullable), xq_f16 [M, K] the same codes as fp16
 * (nullable), s_x [M] fp32. */
w8a8_status w8a8_quantize_activations(const uint16_t* X, int M, int K, const float* inv_delta,
                                      int8_t* xq, uint16_t* xq_f16, float* s_x, void* stream);

/* ------------------------------------------------------------------------ W8A8 linear
 * Y = W8A8 linear of X (LM Head section, Eq. xhat-lmhead .. gemm-final):
 *   acc_ti = sum_j xq_tj * wq_ij (exact INT32);
 *   y_ti   = fl32(fl32(s_x_t * s_w_i) * fl32(acc_ti)), then + bias_i (fp32), then bf16 (RNE).
 * X [M, K] bf16, Y [M, N] bf16, bias [N] fp32 nullable.  dbg nullable. */
w8a8_status w8a8_linear_workspace_size(int M, int N, int K, size_t* bytes);
w8a8_status w8a8_linear(const w8a8_qweight* w, const uint16_t* X, int M, const float* bias,
                        uint16_t* Y, const w8a8_debug* dbg, void* workspace, size_t ws_bytes,
                        void* stream);

/* The W8A8 linear of w8a8_linear for callers that cannot allocate device memory (no counterpart in
 * the paper: it exists for integration).  Callers that run where cudaMalloc is not allowed, such
 * as code inside a framework that owns all device memory or a path with a memory budget fixed at
 * start-up, cannot provide a workspace; this entry point uses a scratch array built into the
 * library instead (w8a8_linear_noalloc_capacity() bytes, 8 MiB, held by every GPU that loads the
 * library until the process exits) and allocates nothing.
 *   - Same arguments and results as w8a8_linear without the debug outputs and the workspace.
 *   - Returns W8A8_ERR_SHAPE when M, N, K need more scratch than the array holds (about 32 tokens
 *     for the Gemma-3-1B shapes); w8a8_linear with a workspace has no such limit.
 *   - The first call on a device looks up the array's device address (cudaGetSymbolAddress) with
 *     that device current; make that first call before any stream capture.
 *   - Every call on a device shares the one array and clears its counter region with a
 *     cudaMemsetAsync on `stream` before launching, so calls whose execution overlaps on the GPU
 *     (different streams, or concurrent host threads) race and give undefined results; serialise
 *     them.
 *   - A bounded device-side wait that gives up sets the array's error word, which the next calls
 *     leave set; w8a8_linear_noalloc_check reports it. */
size_t w8a8_linear_noalloc_capacity(void);
w8a8_status w8a8_linear_noalloc(const w8a8_qweight* w, const uint16_t* X, int M, const float* bias,
                                uint16_t* Y, void* stream);
/* w8a8_workspace_check for the built-in scratch array of the current device: waits for `stream`,
 * then reads and clears the array's device error word.  W8A8_ERR_TIMEOUT if a wait gave up in a
 * w8a8_linear_noalloc call since the last check (their outputs are then undefined).  Synchronous. */
w8a8_status w8a8_linear_noalloc_check(void* stream);

/* bf16 pass-through linear of a layer outside the INT8 set (FFN section: such layers keep the
 * original precision): Y = bf16(sum_j x_tj * w_ij (fp32 accumulation) + bias_i).
 * W [N, K] bf16. */
w8a8_status w8a8_linear_bf16_workspace_size(int M, int N, int K, size_t* bytes);
w8a8_status w8a8_linear_bf16(const uint16_t* W, int N, int K, const uint16_t* X, int M,
                             const float* bias, uint16_t* Y, void* workspace, size_t ws_bytes,
                             void* stream);

/* ------------------------------------------------------------------------- FFN block
 * Gemma-3 FFN (FFN section): [g | u] = gate/up linear of X (fp32 out of the epilogue),
 * h = bf16(gelu_tanh(g) * u), Y = down linear of h (bf16).  precision W8A8_PREC_W8A8 uses
 * w8a8 (both linears W8A8), W8A8_PREC_BF16 uses the bf16 weights.
 * gelu_tanh is evaluated by a fixed fp32 recipe (every operation rounded to nearest-even in
 * this order): g2 = g*g; g3 = g2*g; t = g + 0.044715f*g3; z = 0.7978845608f*t;
 * w = clamp(-2.8853900818f*z, -126, 126); e = 2^w, where 2^w = 2^n * p(f) with n = rint(w),
 * f = w - n and p the degree-7 Taylor polynomial of 2^f by Horner's rule; gelu = g / (1 + e).
 *   h_dbg [M, F] bf16 nullable: receives h. */
typedef struct {
  int32_t hidden, inter;
  w8a8_qweight gate_up;         /* n = 2*inter, k = hidden, 8-row interleave */
  w8a8_qweight down;            /* n = hidden, k = inter */
  const uint16_t* gate_up_bf16; /* [2*inter, hidden] bf16, 8-row interleave; nullable if unused */
  const uint16_t* down_bf16;    /* [hidden, inter] bf16; nullable if unused */
} w8a8_ffn_weights;

w8a8_status w8a8_ffn_workspace_size(int M, int hidden, int inter, size_t* bytes);
w8a8_status w8a8_ffn_block(const w8a8_ffn_weights* ffn, int precision, const uint16_t* X, int M,
                           uint16_t* Y, uint16_t* h_dbg, void* workspace, size_t ws_bytes,
                           void* stream);

/* ------------------------------------------------------------------ FP8 (e4m3) variant
 * The paper's Future Work moves from INT8 to FP8 on Blackwell; it gives no scheme, so this variant
 * keeps the INT8 path's SmoothQuant structure (Eq. delta-attn / delta-lmhead, what-lmhead,
 * xhat-lmhead) and replaces the integer grid by e4m3 (1 sign, 4 exponent bits with bias 7, 3
 * mantissa bits, subnormals down to 2^-9, largest value 448):
 *   s_w_i = fl32(m_i / 448), wq_ij = e4m3(fl32(W_hat_ij * fl32(448 / m_i)))   (m_i = max_j |W_hat_ij|)
 *   s_x_t = fl32(m_t / 448), xq_tj = e4m3(fl32(x_hat_tj * fl32(448 / m_t)))   (m_t = max_j |x_hat_tj|)
 *   acc_ti = sum_j xq_tj * wq_ij in fp32 (every product exact; the sum's rounding depends on the
 *            kernel's order: not bit-exact, within K * 2^-23 * sum_j |xq_tj wq_ij|)
 *   y_ti   = fl32(fl32(s_x_t * s_w_i) * acc_ti), then + bias_i, then bf16 (RNE)
 * e4m3(v): nearest e4m3 value, ties to even, saturating at +-448; an all-zero row or token has scale
 * 0 and codes 0.  Codes are stored as bytes (sign | exponent | mantissa).
 *   wq [n, k] e4m3 codes; s_w [n]; inv_delta [k] = fl32(1 / delta) as for INT8. */
typedef struct {
  int32_t n, k;
  const uint8_t* wq;
  const float* s_w;
  const float* inv_delta;
} w8a8_fp8_weight;

/* Preparation of one linear (w8a8_prepare_weights with the e4m3 rule above), and of the fused
 * gate/up pair with the 8-row interleave of w8a8_prepare_gate_up.  Outputs (caller-owned):
 * wq [N, K] (or [2F, H]) codes, s_w, delta, inv_delta. */
w8a8_status w8a8_fp8_prepare_weights(const uint16_t* W, int N, int K, const float* act_absmax, float alpha,
                                     int smooth, uint8_t* wq, float* s_w, float* delta, float* inv_delta,
                                     void* stream);
w8a8_status w8a8_fp8_prepare_gate_up(const uint16_t* W_gate, const uint16_t* W_up, int F, int H,
                                     const float* act_absmax, float alpha, int smooth, uint8_t* wq,
                                     float* s_w, float* delta, float* inv_delta, void* stream);

/* Per-token e4m3 quantisation of the smoothed input: X [M, K] bf16 -> xq [M, K] codes, s_x [M]. */
w8a8_status w8a8_fp8_quantize_activations(const uint16_t* X, int M, int K, const float* inv_delta,
                                          uint8_t* xq, float* s_x, void* stream);

/* Y [M, N] bf16 = FP8 linear of X [M, K] bf16 (rule above).  N and K multiples of 16.
 * xq_dbg [M, K] and s_x_dbg [M] (nullable) receive the activation codes and scales.  The workspace
 * is sized by w8a8_linear_workspace_size. */
w8a8_status w8a8_fp8_linear(const w8a8_fp8_weight* w, const uint16_t* X, int M, const float* bias,
                            uint16_t* Y, uint8_t* xq_dbg, float* s_x_dbg, void* workspace, size_t ws_bytes,
                            void* stream);

/* The FFN block of w8a8_ffn_block with both linears in FP8: [g | u] = FP8 gate/up linear of X (fp32
 * out of the epilogue), h = bf16(gelu_tanh(g) * u) (the same fp32 recipe), Y = FP8 down linear of h.
 * The workspace is sized by w8a8_ffn_workspace_size; h_dbg [M, F] (nullable) receives h. */
typedef struct {
  int32_t hidden, inter;
  w8a8_fp8_weight gate_up; /* n = 2*inter, k = hidden, 8-row interleave */
  w8a8_fp8_weight down;    /* n = hidden, k = inter */
} w8a8_fp8_ffn_weights;

w8a8_status w8a8_fp8_ffn_block(const w8a8_fp8_ffn_weights* ffn, const uint16_t* X, int M, uint16_t* Y,
                               uint16_t* h_dbg, void* workspace, size_t ws_bytes, void* stream);

/* --------------------------------------------------------------------------- lm_head
 * Logits over the tied [V, d] table (LM Head section) and the top-1 index.
 *   W8A8: logits_tv = fl32(fl32(s_x_t * s_w_v) * fl32(acc_tv)) (fp32, not rounded further).
 *   BF16: logits_tv = sum_j x_tj * w_vj in fp32.
 *   top1_t = argmax_v logits_tv (ties go to the lowest v).
 * X [M, d] bf16 (the final-norm output); logits [M, V] fp32 nullable; top1 [M] int32. */
typedef struct {
  int32_t vocab, hidden;
  w8a8_qweight q;        /* n = vocab, k = hidden */
  const uint16_t* bf16;  /* [vocab, hidden] bf16 (the embedding table); nullable if unused */
} w8a8_head_weights;

w8a8_status w8a8_lm_head_workspace_size(int M, int vocab, int hidden, size_t* bytes);
w8a8_status w8a8_lm_head(const w8a8_head_weights* head, int precision, const uint16_t* X, int M,
                         float* logits, int32_t* top1, void* workspace, size_t ws_bytes,
                         void* stream);

/* ---------------------------------------------------------------------------- decoder
 * A Gemma-3-1B-shaped decoder (Problem Statement: 26 layers, hidden 1152, 4 query heads sharing
 * 1 key/value head of dim 256, FFN 6912, vocab 262144, lm_head tied to the embedding; Attention
 * section: sliding window on local layers) under a per-layer precision mask: FFN layer l is W8A8
 * when bit l of ffn_bits is set (the sets Q_FFN of Eq. ffn55, ffn1010, ffnall26), the attention
 * projections of layer l when bit l of attn_bits is set (Q_ATT, Eq. attnffn55, attnffn1010), the
 * lm_head when lm != 0 (LM Head section); everything else runs the bf16 pass-through.
 *
 * Per layer: a = bf16(rmsnorm(r) * ln_in); qkv = Linear(a); q, k = rope(rmsnorm_head(q|k) * q_norm|k_norm);
 * K/V cache <- k, v; o = bf16(softmax(q k^T / sqrt(head_dim)) v) over keys p - window < j <= p
 * (all j <= p on global layers); r += rmsnorm(Linear(o)) * ln_post_attn; a = bf16(rmsnorm(r) *
 * ln_pre_ffn); r += rmsnorm(FFN(a)) * ln_post_ffn.  r starts as embed[token] * fl32(sqrt(hidden))
 * (fp32 residual stream); logits = lm_head(bf16(rmsnorm(r) * final_norm)).
 *
 * The model object owns device buffers it allocates at creation and preparation (KV cache,
 * activations, workspaces, the fused gate/up bf16 copy, prepared INT8 weights); forward and
 * decode calls allocate nothing.  All pointers in the structs below are caller-owned device
 * memory that must outlive the model. */
typedef struct {
  int32_t layers, hidden, inter, n_q, n_kv, head_dim, vocab;
  float eps;                  /* RMSNorm epsilon */
  float rope_local, rope_global; /* RoPE bases of local / global layers */
  int32_t window;             /* sliding window of local layers */
  int32_t n_global;           /* number of global layers listed in global_layers */
  int32_t global_layers[32];
  int32_t qk_norm;            /* 1: RMS-normalise q and k per head */
  int32_t max_batch, max_seq; /* KV-cache capacity: sequences x positions */
  int32_t max_tokens;         /* largest B * T of one forward call */
} w8a8_model_cfg;

typedef struct {
  const uint16_t* wqkv;  /* [(n_q + 2 n_kv) * head_dim, hidden] bf16: q rows, then k, then v */
  const uint16_t* wo;    /* [hidden, n_q * head_dim] */
  const uint16_t* wgate; /* [inter, hidden] */
  const uint16_t* wup;   /* [inter, hidden] */
  const uint16_t* wdown; /* [hidden, inter] */
  const float *ln_in, *ln_post_attn, *ln_pre_ffn, *ln_post_ffn; /* [hidden] RMSNorm multipliers */
  const float *q_norm, *k_norm;                                 /* [head_dim] (used when qk_norm) */
} w8a8_layer_bf16;

typedef struct w8a8_model w8a8_model;

enum { W8A8_SUB_FFN = 0, W8A8_SUB_ATTN = 1, W8A8_SUB_LM = 2 };

/* layers: array of cfg->layers descriptors; embed [vocab, hidden] bf16 (also the lm_head);
 * final_norm [hidden].  The mask starts all-bf16. */
w8a8_status w8a8_model_create(const w8a8_model_cfg* cfg, const w8a8_layer_bf16* layers, const uint16_t* embed,
                              const float* final_norm, w8a8_model** out);
w8a8_status w8a8_model_destroy(w8a8_model* m);

/* Calibration (LM Head section: max_t |X_tj| at every linear's input, collected over calibration
 * tokens): runs the all-bf16 decoder over tokens [B, T] (device int32) from position 0 and folds
 * each linear input's per-channel absolute maximum into the model's statistics.
 * w8a8_model_reset_calibration zeroes them. */
w8a8_status w8a8_model_calibrate(w8a8_model* m, const int32_t* tokens, int B, int T, void* stream);
w8a8_status w8a8_model_reset_calibration(w8a8_model* m, void* stream);

/* The statistics as one fp32 array of w8a8_model_stats_count() values: for each layer l,
 * [hidden] at the qkv input, [n_q * head_dim] at the o input, [hidden] at the gate/up input and
 * [inter] at the down input; then [hidden] at the lm_head input.  get / set copy to / from HOST
 * memory and are synchronous (set replaces statistics gathered so far). */
size_t w8a8_model_stats_count(const w8a8_model* m);
w8a8_status w8a8_model_get_stats(const w8a8_model* m, float* host_out);
w8a8_status w8a8_model_set_stats(w8a8_model* m, const float* host_in);

/* Prepares the W8A8 weights of every linear (qkv, o, fused gate/up, down, lm_head) from the
 * statistics (w8a8_prepare_weights / w8a8_prepare_gate_up semantics).  Required before a mask
 * selects W8A8 for any sublayer. */
w8a8_status w8a8_model_prepare(w8a8_model* m, float alpha, int smooth, void* stream);

/* Host-side, synchronous.  layer in [0, layers) for FFN / ATTN; LM ignores layer. */
w8a8_status w8a8_set_layer_precision(w8a8_model* m, int layer, int sublayer, int precision);
w8a8_status w8a8_set_mask(w8a8_model* m, uint32_t ffn_bits, uint32_t attn_bits, int lm);
w8a8_status w8a8_get_mask(const w8a8_model* m, uint32_t* ffn_bits, uint32_t* attn_bits, int* lm);

/* Runs tokens [B, T] (device int32, row b * T + t at position start_pos + t) through the decoder,
 * appending to the KV cache.  logits [B * T, vocab] fp32 (nullable), top1 [B * T] int32. */
w8a8_status w8a8_decoder_forward(w8a8_model* m, const int32_t* tokens, int B, int T, int start_pos, float* logits,
                                 int32_t* top1, void* stream);

/* One decode step of B sequences (one token each, at position pos) replayed from a CUDA graph
 * captured on first use for this (B, mask, logits wanted) and kept until the mask or the
 * preparation changes.  tokens [B], logits [B, vocab] (nullable), top1 [B]: device memory. */
w8a8_status w8a8_decoder_decode_step(w8a8_model* m, const int32_t* tokens, int B, int pos, float* logits,
                                     int32_t* top1, void* stream);

/* Diagnostic trace (no counterpart in the paper; it lets a reference check every step of every
 * layer on the GPU's own inputs): while set, each w8a8_decoder_forward and w8a8_decoder_decode_step
 * of M = B * T <= max_rows rows copies, for every layer l, these tensors into caller-owned DEVICE
 * buffers laid out [layers][max_rows][width] (rows [0, M) of slice l are written; each pointer
 * nullable):
 *   a_in  bf16 [., ., hidden]    the q/k/v input bf16(rmsnorm(r) * ln_in)
 *   qkv   bf16 [., ., (n_q + 2 n_kv) head_dim]
 *   attn  bf16 [., ., n_q head_dim]   the attention output (the o projection's input)
 *   y_o   bf16 [., ., hidden]    the o projection's output
 *   a_ffn bf16 [., ., hidden]    the FFN block's input
 *   h     bf16 [., ., inter]     the GeGLU output (the down projection's input)
 *   y_f   bf16 [., ., hidden]    the FFN block's output
 *   r     fp32 [., ., hidden]    the residual stream after the layer
 * and a_fin bf16 [max_rows][hidden], the lm_head's input.  Tracing turns off the fusion of the
 * residual step into the decode GEMV (the traced path computes the same values through the
 * stand-alone residual-norm kernel).  NULL clears the trace.  Host-side, synchronous. */
typedef struct {
  uint16_t *a_in, *qkv, *attn, *y_o, *a_ffn, *h, *y_f;
  float* r;
  uint16_t* a_fin;
  int32_t max_rows;
} w8a8_trace;
w8a8_status w8a8_model_set_trace(w8a8_model* m, const w8a8_trace* t);

/* Measurement aid with no counterpart in the paper: *kernels = the number of kernel launches
 * one w8a8_decoder_decode_step of B sequences makes under the current mask (the kernel nodes of
 * its CUDA graph plus the position update launched beside it; copies are not counted).  The
 * graph must exist: W8A8_ERR_INVALID_ARG before the first decode step of this (B, mask). */
w8a8_status w8a8_model_decode_kernels(const w8a8_model* m, int B, int want_logits, int* kernels);

/* Test and measurement aid with no counterpart in the paper (host only, no device access): the
 * launch plan the decode GEMV (the row-owning kernel behind w8a8_linear, w8a8_linear_bf16,
 * w8a8_ffn_block and the decoder at 1-16 tokens) makes for an [N, K] linear over M tokens.
 * weight_kind: 0 bf16, 1 INT8 codes, 2 e4m3 codes; geglu: the FFN's gate/up epilogue; fused_norm:
 * the decoder's residual step computed in the prologue; sms: the device's SM count.  out receives
 * W8A8_PLAN_FIELDS ints: taken (0: the shape goes to another kernel, every field 0), token slots,
 * weight rows per warp, CTAs, CTAs per SM, consumer warps, 512-byte sub-slices per stage, pipeline
 * steps, ring stages, stage bytes, activation bytes, residual-row bytes, partial-sum bytes, dynamic
 * shared memory bytes, padded K, sub-slices over K.  W8A8_ERR_INVALID_ARG for a null out, a weight
 * kind outside 0-2 or sms < 1. */
#define W8A8_PLAN_FIELDS 16
w8a8_status w8a8_decode_gemv_plan(int weight_kind, int M, int N, int K, int geglu, int fused_norm, int sms,
                                  int* out);

/* Test and measurement aid with no counterpart in the paper (host only, no device access): the
 * plan of the persistent weight-streaming kernel behind the lm_head (and W8A8 linears prepared
 * without the fp16 code copy) for an [N, K] linear over M tokens.  out receives
 * W8A8_STREAM_PLAN_FIELDS ints: dp4a GEMV (1) or MMA streaming (0), whole 128-row groups per CTA,
 * dp4a token slots (0 on the MMA path), 8-token blocks per token group, tokens per group, token
 * groups, 128-row weight groups, k elements per stage, k chunks per row group, CTAs, CTAs per SM,
 * ring stages, stage bytes, dynamic shared memory bytes, partial-sum bytes.  W8A8_ERR_INVALID_ARG
 * for a null out, M, N < 1, K < 16 or sms < 1. */
#define W8A8_STREAM_PLAN_FIELDS 15
w8a8_status w8a8_stream_gemm_plan(int int8_weights, int M, int N, int K, int sms, int* out);

/* Test and measurement aid with no counterpart in the paper (host only, no device access): the
 * tile shape and k split the tcgen05 GEMM takes for an [N, K] linear over M tokens.  mode: 0 bf16,
 * 1 INT8 codes (carried as fp16), 2 e4m3; kind: 0 bf16 output, 1 GeGLU, 2 fp32 logits; split_ok:
 * the caller's workspace holds the partials and tile counters a k split needs; sms: the SM count.
 * out[0] = 1 for CTA pairs on 256-token tiles, 0 for single CTAs on 128-token tiles; out[1] = the
 * tile's channels (256, 192 or 128 on pairs; 128 or 64 on single CTAs); out[2] = the k parts of a
 * single-CTA tile (1: no split).  W8A8_ERR_INVALID_ARG for a null out, a mode or kind out of range or
 * sms < 2; W8A8_ERR_SHAPE where the GEMM does not take the shape (K or N not a multiple of 16). */
w8a8_status w8a8_tc_gemm_plan(int mode, int M, int N, int K, int kind, int split_ok, int sms, int* out);

/* Negative log-likelihood of targets under softmax(logits) per row (LM Head section's
 * perplexity): nll[i] = logsumexp(logits[i, :]) - logits[i, targets[i]], fp32. */
w8a8_status w8a8_token_nll(const float* logits, const int32_t* targets, int M, int V, float* nll, void* stream);

/* ------------------------------------------------------------------------ allocation
 * The allocation rule (Problem Statement; Combined Configurations): among the candidates whose
 * Top-1 agreement with the all-bf16 decoder is >= min_top1 and whose perplexity change is
 * <= max_ppl_delta, the one with the smallest per-token latency; ties go to fewer INT8
 * sublayers, then to the earlier candidate.  Host arrays of length n.  Returns the index, or -1
 * if no candidate is feasible. */
int w8a8_choose_mask(const float* latency, const float* top1, const float* ppl_delta, const int32_t* n_int8, int n,
                     float min_top1, float max_ppl_delta);

typedef struct {
  uint32_t ffn_bits, attn_bits;
  int32_t lm;
} w8a8_mask;

typedef struct {
  const w8a8_mask* candidates; /* host array of n_candidates masks */
  int32_t n_candidates;
  const int32_t* eval_tokens;  /* device [eval_B, eval_T]: teacher-forced evaluation stream */
  int32_t eval_B, eval_T;
  int32_t decode_B;            /* latency: decode steps of decode_B sequences ... */
  int32_t prefill_T;           /* ... after a prefill of prefill_T tokens ... */
  int32_t decode_steps;        /* ... timed over decode_steps steps, median of reps runs */
  int32_t reps;
  float min_top1, max_ppl_delta;
} w8a8_alloc_opts;

typedef struct {
  int32_t chosen;     /* index into candidates, -1 if none is feasible */
  float* latency_ms;  /* host [n_candidates]: median ms per decode step */
  float* top1;        /* host [n_candidates]: Top-1 agreement with the all-bf16 decoder */
  float* ppl_delta;   /* host [n_candidates]: PPL / PPL(bf16) - 1 on the evaluation stream */
} w8a8_alloc_report;

/* The allocator: measures every candidate (latency with CUDA events; quality against the all-bf16
 * decoder on the evaluation stream) and applies w8a8_choose_mask.  Leaves the chosen mask set
 * (the all-bf16 mask if none is feasible).  Synchronous; requires w8a8_model_prepare. */
w8a8_status w8a8_allocate_mask(w8a8_model* m, const w8a8_alloc_opts* opts, w8a8_alloc_report* report, void* stream);

/* Allocation per sublayer, below the groups of the Combined Configurations (the finer granularity
 * the paper's title names; its own search stops at groups).  Sublayer i: 0 .. L-1 the FFN of
 * layer i, L .. 2L-1 the attention projections of layer i - L, 2L the lm_head.
 *
 * The ranking rule (host code, exported for tests): the sublayers with a positive latency gain
 * whose single-sublayer mask meets the budget by itself, in descending order of
 * gain / (cost + 1e-3), where cost = max(0, 1 - top1) / max(1e-6, 1 - min_top1)
 *                                  + max(0, ppl_delta) / max(1e-6, max_ppl_delta)
 * (evaluated in double precision); ties go to the lower index.  Host arrays of length n; writes the
 * ranked indices to order (length n) and returns how many there are. */
int w8a8_greedy_order(const float* gain_ms, const float* top1, const float* ppl_delta, int n, float min_top1,
                      float max_ppl_delta, int32_t* order);

typedef struct {
  const int32_t* eval_tokens;  /* device [eval_B, eval_T]: teacher-forced evaluation stream */
  int32_t eval_B, eval_T;
  int32_t decode_B, prefill_T, decode_steps, reps;  /* latency, as in w8a8_alloc_opts */
  float min_top1, max_ppl_delta;
} w8a8_layer_alloc_opts;

typedef struct {
  w8a8_mask chosen;        /* the accepted sublayers (all-bf16 if none) */
  float base_ms;           /* decode ms per step of the all-bf16 mask */
  float chosen_ms;         /* ... and of the chosen mask */
  float chosen_top1, chosen_ppl_delta;
  float* gain_ms;          /* host [2L + 1]: base_ms - ms of each single-sublayer mask */
  float* top1;             /* host [2L + 1]: Top-1 agreement of each single-sublayer mask */
  float* ppl_delta;        /* host [2L + 1]: its perplexity change */
  int32_t* order;          /* host [2L + 1]: the ranked sublayers, n_order of them */
  int32_t n_order;
  int32_t n_accepted;      /* how many of them the chosen mask holds */
} w8a8_layer_alloc_report;

/* The per-sublayer allocator: measures every single-sublayer mask (quality and latency, as
 * w8a8_allocate_mask does), ranks the sublayers with w8a8_greedy_order, then adds them one at a
 * time in that order, keeping each one only if the cumulative mask still meets the budget (its
 * quality measured again); finally times the chosen mask and leaves it set.  Synchronous; requires
 * w8a8_model_prepare and at most 32 layers. */
w8a8_status w8a8_allocate_layers(w8a8_model* m, const w8a8_layer_alloc_opts* opts, w8a8_layer_alloc_report* report,
                                 void* stream);

/* SQNR in dB (Eq. sqnr-ffn; Eq. sqnr-block is the same ratio of means):
 * 10 log10(sum y_ref^2 / sum (y_ref - y_q)^2) over n device floats, the sums taken in fp64 in a
 * fixed order (deterministic); +inf when the two arrays are equal.  Synchronous. */
w8a8_status w8a8_sqnr_db(const float* y_ref, const float* y_q, size_t n, double* out_db, void* stream);

/* SQNR diagnostics of a mask over a prefill of tokens [B, T] (device, T >= 2) from position 0,
 * against the all-bf16 decoder (Combined Configurations: the isolated and propagated regimes).
 * layer_db (host [L]): the SQNR of every decoder block's output (the residual stream after its
 * post-FFN step, Eq. sqnr-block); lm_db (host [1]): of the lm_head's fp32 logits.
 *   propagated (isolated = 0): one pass under the whole mask, so errors accumulate;
 *   isolated (isolated = 1): for each layer a pass with only that layer's sublayers of the mask
 *   quantised, so the layer takes the reference input (+inf where the mask quantises nothing in
 *   the layer); the lm_head likewise alone (+inf if the mask leaves it in bf16).
 * Leaves the model's mask as it was; overwrites the layers' KV cache rows [0, T).  Synchronous;
 * requires w8a8_model_prepare (with or without smoothing: the delta = 1 ablation is a prepare
 * with smooth = 0). */
w8a8_status w8a8_sqnr_profile(w8a8_model* m, const int32_t* tokens, int B, int T, const w8a8_mask* mask, int isolated,
                              float* layer_db, float* lm_db, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* W8A8_H */
