// Supporting kernels of the Gemma-3-1B-shaped decoder (bf16 activations, fp32 residual stream).
#pragma once

#include "common.cuh"

namespace w8a8 {

struct AttnShape {
  int B, T;            // sequences, new tokens per sequence (rows are b * T + t)
  int n_q, n_kv, hd;   // query heads, key/value heads, head dim (hd == 256 supported)
  int max_seq;         // KV-cache capacity per sequence
  int window;          // sliding window (keys p - window < j <= p), or 0 for global attention
  float scale;         // attention scale
};

// r = fp32(embed[token]) * embed_scale; a = bf16(rmsnorm(r) * w) (token ids outside [0, vocab) read row 0).
// q_inv_delta non-null: also the next linear's per-token quantiser on a (fp16 codes [M, H] and
// s_x [M], bit-identical to the stand-alone quantiser), so that linear needs no launch of its own.
w8a8_status launch_embed_norm(const int32_t* tokens, int M, const uint16_t* embed, int vocab, int H, float embed_scale,
                              const float* w, float eps, float* r, uint16_t* a, cudaStream_t st,
                              const float* q_inv_delta = nullptr, uint16_t* q_codes = nullptr, float* q_sx = nullptr,
                              int* q_sum = nullptr);

// r += rmsnorm(y) * w_post;  a = bf16(rmsnorm(r) * w_next); the quantiser as above
w8a8_status launch_residual_norm(const uint16_t* y, int M, int H, const float* w_post, const float* w_next, float eps,
                                 float* r, uint16_t* a, cudaStream_t st, const float* q_inv_delta = nullptr,
                                 uint16_t* q_codes = nullptr, float* q_sx = nullptr, int* q_sum = nullptr);

// Per row: q heads and k head RMS-normalised (weights qn, kn; skipped when null), RoPE at position
// *pos0 + t, q -> fp32 [M, n_q*hd], k and v -> bf16 KV cache [B][max_seq][n_kv*hd] of this layer.
w8a8_status launch_qk_rope(const uint16_t* qkv, const AttnShape& s, const int* pos0, const float* qn, const float* kn,
                           float eps, const float* rope_cos, const float* rope_sin, float* q, uint16_t* kcache,
                           uint16_t* vcache, cudaStream_t st);

// Causal softmax attention over the cache; o bf16 [M, n_q*hd].  Long key ranges are split across
// CTAs; the last CTA of a row combines the splits (workspace: partials + per-row counters, the
// counters zero before and after).
size_t attention_workspace_bytes(const AttnShape& s, int sm_count);
w8a8_status launch_attention(const float* q, const uint16_t* kcache, const uint16_t* vcache, const AttnShape& s,
                             const int* pos0, int max_pos_hint, uint16_t* o, void* ws, int sm_count, cudaStream_t st);

// Decode (T == 1): QK-norm + RoPE of the new row, its key/value into the cache, and attention over
// the cache, in one launch (clusters of 8 CTAs combine their key ranges in distributed shared
// memory).  Same results as launch_qk_rope followed by launch_attention up to fp32 summation order.
bool attn_decode_supported(const AttnShape& s);
w8a8_status launch_attn_decode(const uint16_t* qkv, const AttnShape& s, const int* pos0, const float* qn,
                               const float* kn, float eps, const float* rope_cos, const float* rope_sin,
                               uint16_t* kcache, uint16_t* vcache, uint16_t* o, cudaStream_t st);

// Prefill (T > 1): flash-attention-style attention of q (fp32, after QK-norm and RoPE) over the
// cache on the tensor cores (fp16 operands, fp32 accumulation and softmax); o bf16 [M, n_q*hd].
bool attention_prefill_supported(const AttnShape& s);
w8a8_status launch_attention_prefill(const float* q, const uint16_t* kcache, const uint16_t* vcache, const AttnShape& s,
                                     const int* pos0, uint16_t* o, cudaStream_t st);

// cos/sin tables [max_seq][hd/2] of RoPE with the given base, computed in fp64
w8a8_status launch_rope_table(float* cos_t, float* sin_t, int max_seq, int hd, double base, cudaStream_t st);

w8a8_status launch_set_int(int* dst, int value, cudaStream_t st);

}  // namespace w8a8
