// Tensor-core GEMM for prefill-sized token counts on the 5th-generation tensor cores (tcgen05):
// the W8A8 path (INT8 codes carried as fp16, exact), the FP8 variant (e4m3 codes) and the bf16
// pass-through.
#pragma once

#include "common.cuh"

namespace w8a8 {

// Operand modes: bf16, INT8 codes carried as fp16 (kind::f16, exact INT32 by folding every 1024 k),
// e4m3 codes (kind::f8f6f4, fp32 accumulation).
enum { TC_BF16 = 0, TC_I8 = 1, TC_FP8 = 2 };

struct TcArgs {
  const void* A;        // [M, K] activations: fp16 INT8 codes (TC_I8), e4m3 codes (TC_FP8) or bf16, row-major
  const void* B;        // [N, K] weights in the same type as A, row = output channel
  int M, N, K;
  int kind;             // EPI_BF16, EPI_GEGLU or EPI_F32
  const float* s_x;     // [M] W8A8 / FP8: per-token scales
  const int* qsum;      // [M] W8A8, nullable: sum_k |q_tk| per token; a tile whose tokens all have
                        // 127 qsum <= 2^24 runs one exact fp32 accumulator over all of k (no folds)
  const float* s_w;     // [N] W8A8 / FP8: per-channel scales
  const float* bias;    // [N] nullable
  uint16_t* y;          // bf16 [M, N] (EPI_BF16) or [M, N / 2] (EPI_GEGLU)
  float* logits;        // [M, N] nullable (EPI_F32)
  int32_t* top1;        // [M] nullable (EPI_F32)
  int32_t* acc_dbg;     // [M, N] nullable (W8A8): the INT32 sums
  unsigned int* grid_counter;     // top-1: one counter, zero between calls
  unsigned long long* top_keys;   // top-1: [M] keys, zero between calls
  unsigned int* err;              // device error word
  // split-K (few output tiles): the k range of a tile is cut into ksplit parts on different CTAs
  int ksplit;                     // set by the launcher (1: no split)
  void* partials;                 // tc_split_partial_bytes(M) bytes of workspace
  unsigned int* tile_counters;    // one per output tile, zero between calls
};

// Shapes the tensor-core GEMM takes: K a multiple of 16, N a multiple of 16, top-1 for at most
// max_top rows.
bool tc_gemm_supported(int M, int N, int K, int kind, bool want_top, int max_top);

// The tile shape and k split the tcgen05 GEMM takes for a call (host only): pair = 1 for CTA pairs
// on 256-token tiles of bn = 256, 192 or 128 channels, 0 for single CTAs on 128-token tiles of bn =
// 128 or 64 channels; ksplit = the k parts of a single-CTA tile (1: none).  mode: TC_BF16, TC_I8 or
// TC_FP8; kind: the epilogue; split_ok: partials and tile counters are available; sms: SM count.
struct TcChoice {
  int pair;
  int bn;
  int ksplit;
};
TcChoice tc_choose(int mode, int M, int N, int K, int kind, bool split_ok, int sms);
// Workspace bytes the split-K partials of an M-token call may take (an upper bound over N and K,
// non-decreasing in M).
size_t tc_split_partial_bytes(int M, int sms);
w8a8_status launch_tc_gemm(int mode, const TcArgs& a, cudaStream_t st);

}  // namespace w8a8
