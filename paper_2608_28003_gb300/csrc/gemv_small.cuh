// Decode GEMV for up to 16 tokens whose CTAs own whole weight rows (no split of the k sum across
// CTAs): the W8A8 path with the per-token quantiser (K1) fused into its prologue, its e4m3 (FP8)
// variant, and the bf16 pass-through.
#pragma once

#include "common.cuh"

namespace w8a8 {

// Weight kinds: bf16, INT8 codes (W8A8), e4m3 codes (the FP8 variant: codes widened to fp32 for
// FMAs at 1-4 token slots, to fp16 for the tensor cores at 8 / 16).
enum { SMALL_BF16 = 0, SMALL_INT8 = 1, SMALL_FP8 = 2 };

struct SmallPlan {
  int ok;           // 0: this shape is left to the weight-streaming kernel
  int MT;           // token slots: 1, 2, 4, 8 or 16 (8 and 16: the tensor-core paths)
  int RW;           // weight rows per consumer warp: 1, 2, 4 or 6 (R = 8 RW rows per CTA)
  int P;            // CTAs
  int sub;          // k elements per 512-byte sub-slice of a row (256 bf16, 512 INT8)
  int nsub;         // sub-slices covering K
  int kpad;         // nsub * sub
  int ks;           // sub-slices per pipeline stage (1, 2 or 4)
  int nst;          // pipeline steps per CTA (nsub / ks, rounded up)
  int stages;       // ring depth
  int stage_bytes;  // ks x R rows x 512 bytes
  int xbytes;       // activations in shared memory: MT x kpad bf16 or INT8 codes
  int abytes;       // W8A8 with a fused residual norm: the bf16 rows it produces, before K1
  int rbytes;       // 5-8 tokens (tensor-core paths): the consumer warps' partial sums
  int smem_bytes;
  int cw;           // consumer warps: 8, or 16 on the tensor-core paths when the grid has one CTA per SM
};

// The decoder's residual step in front of a decode linear, fused into the GEMV's prologue:
// r_out = r_in + rmsnorm(y) * w_post, and the linear's input X = bf16(rmsnorm(r_out) * w_next),
// with the arithmetic of the stand-alone residual-norm kernel (bit-identical results).  Every CTA
// computes the rows it needs; the first CTA writes r_out, so r_out must not alias r_in.
struct ResNorm {
  const uint16_t* y;    // [M, K] bf16: the previous linear's output
  const float* r_in;    // [M, K] fp32 residual stream before
  float* r_out;         // [M, K] fp32 residual stream after
  const float* w_post;  // [K] weights of the norm of y
  const float* w_next;  // [K] weights of the norm of the new residual (this linear's input norm)
  float eps;
};

struct SmallArgs {
  const void* W;           // [N, K] INT8 codes, e4m3 codes or bf16, row = output channel
  const uint16_t* X;       // [M, K] bf16 activations
  int M, N, K;
  int kind;                // EPI_BF16 or EPI_GEGLU (gate/up rows interleaved in blocks of 8)
  const float* inv_delta;  // [K] INT8 path: 1 / delta_j
  const float* s_w;        // [N] INT8 path
  const float* bias;       // [N] nullable
  uint16_t* y;             // [M, N] bf16 or [M, N / 2] for GeGLU
  int8_t* xq_dbg;          // [M, K] nullable: the INT8 (or e4m3) activation codes
  float* s_x_dbg;          // [M] nullable: the per-token scales
  int32_t* acc_dbg;        // [M, N] nullable: the INT32 sums (INT8 codes only)
  int has_rn;              // 1: X is computed from rn (X unused)
  ResNorm rn;
  unsigned int* err;       // device error word
  SmallPlan p;
  // The FFN's down projection at 5-16 tokens (token slots 8 or 16): the gate/up launch (GeGLU) writes,
  // per CTA and token slot, the maximum of |fl(h * next_inv_delta)| over its h channels (rowmax_out
  // [P][MT]); the down launch (W8A8) takes m_t as the maximum of rowmax_n such rows (rowmax_in) and
  // skips the first pass of its quantiser.  Both nullable.
  float* rowmax_out;
  const float* next_inv_delta;  // [N / 2] the down projection's 1 / delta
  const float* rowmax_in;
  int rowmax_n;
};

// fused_norm: the call computes its input with a ResNorm (needs K <= 2048)
SmallPlan make_small_plan(int wkind, int M, int N, int K, int kind, int sm_count, bool fused_norm = false);
w8a8_status launch_small_gemv(int wkind, const SmallArgs& a, cudaStream_t st);

}  // namespace w8a8
