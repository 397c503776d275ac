// Persistent decode kernel: every decoder layer of one decode step (batch 1, one new token) in one
// cooperative launch.
#pragma once

#include "common.cuh"

namespace w8a8 {

// One decoder layer as the persistent kernel reads it (device-resident array, one entry per layer).
// Linear j in {0: q/k/v, 1: o, 2: gate/up (rows interleaved in blocks of 8 gate, 8 up), 3: down}:
// bf16 weights [N, K] always; INT8 codes [N, K] with per-row scales and 1 / delta when prepared.
struct MegaLayer {
  const uint16_t* w16[4];
  const int8_t* w8[4];
  const float* s_w[4];
  const float* inv_delta[4];
  const float* ln_in;         // pre-attention RMSNorm weight
  const float* ln_post_attn;  // post-attention RMSNorm weight
  const float* ln_pre_ffn;    // pre-FFN RMSNorm weight
  const float* ln_post_ffn;   // post-FFN RMSNorm weight
  const float* q_norm;        // QK-norm weights (nullable: no QK-norm)
  const float* k_norm;
  const float* rope_cos;      // [max_seq][128]
  const float* rope_sin;
  int window;                 // sliding window, 0 = global attention
  uint16_t* kc;               // this layer's KV cache, [max_seq][n_kv * 256] bf16 (sequence 0)
  uint16_t* vc;
};

struct MegaArgs {
  const MegaLayer* layers;
  int L, H, F, n_q, n_kv, max_seq;  // head dim 256
  float eps, scale;
  uint32_t attn_bits, ffn_bits;     // W8A8 sublayers (bit l: layer l)
  const int* pos;                   // position of the new token
  const uint16_t* a0;               // layer 0's normalised input [H] bf16
  float* r0;                        // residual stream [H] fp32 (input), ping-pong with r1
  float* r1;
  uint16_t* qkv;                    // scratch activations: [(n_q + 2 n_kv) 256], [n_q 256], [H], [F]
  uint16_t* att;
  uint16_t* y;                      // o output, then the FFN output (the last layer's stays here)
  uint16_t* h;
  float* part;                      // attention partials: n_q x kMegaMaxSplits x (256 + 2) floats
  unsigned int* sync;               // counters, mega_sync_words(L, n_q) words, zero at launch
  unsigned int* err;                // device error word
};

constexpr int kMegaMaxSplits = 32;  // CTAs per query head in the attention step, at most
constexpr int kPartStride = 260;    // floats per attention partial: o[256], m, l, 2 of padding (16-byte rows)
inline size_t mega_sync_words(int L, int n_q) { return (size_t)L * (5 + n_q); }
inline size_t mega_part_floats(int n_q) { return (size_t)n_q * kMegaMaxSplits * kPartStride; }

// Shapes the kernel takes: head dim 256, 2 or 4 query heads per key/value head, H and F multiples of
// 16 up to 8192, a cooperative grid of one CTA per SM with at least n_q * 8 CTAs.
bool decode_mega_supported(int H, int F, int n_q, int n_kv, int hd, int sms);
// The layers take 2 L - 1 residual steps (all but layer 0's pre-attention one), each moving the
// residual stream from one buffer to the other: afterwards it is in r1, and y holds the last
// layer's FFN output (the final residual step and norm are left to the caller).
w8a8_status launch_decode_mega(const MegaArgs& a, cudaStream_t st);

}  // namespace w8a8
