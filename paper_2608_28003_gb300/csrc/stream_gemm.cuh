// Weight-streaming GEMM for decode-sized token counts (K3: W8A8; K6: bf16 pass-through).
#pragma once

#include "common.cuh"

namespace w8a8 {

enum EpiKind { EPI_BF16 = 0, EPI_GEGLU = 1, EPI_F32 = 2 };

// Static decomposition of one call (host computes it; the kernel re-derives unit ranges).
struct StreamPlan {
  int dp4a;     // 1: INT8 GEMV on INT8 activation codes with dp4a (M <= 4, X resident in shared memory)
  int whole;    // 1: every CTA takes whole (z, g) groups (no partial tiles); 0: even split of units
  int MT;       // dp4a path: token slots (1, 2 or 4)
  int NB;       // 8-token blocks per token group (1, 2, 4 or 8)
  int TOK;      // tokens per group = 8 * NB
  int Z;        // token groups
  int G;        // 128-row weight groups
  int KC;       // k elements per pipeline stage
  int C;        // k chunks per row group
  int P;        // CTAs (persistent, one per SM)
  int stages;   // pipeline depth
  int stage_bytes;
  int smem_bytes;
  size_t partial_bytes;  // [P][2][128][TOK] int32/fp32
};

struct StreamArgs {
  const void* W;       // [N, K] int8 codes or bf16
  const void* X;       // [M, K]: fp16 codes (INT8 MMA path), INT8 codes (dp4a path) or bf16
  int M, N, K;
  StreamPlan p;
  // epilogue
  int kind;
  const float* s_x;    // [M] (int path)
  const float* s_w;    // [N] (int path)
  const float* bias;   // [N] nullable
  uint16_t* y;         // bf16 [M, N] (EPI_BF16) or [M, N/2] (EPI_GEGLU)
  float* logits;       // [M, N] nullable (EPI_F32)
  int32_t* acc_dbg;    // [M, N] nullable (int path)
  int32_t* top1;       // [M] nullable (EPI_F32)
  // workspace pieces
  void* partials;
  unsigned int* tile_counters;     // [P]
  unsigned int* grid_counter;      // one counter (top-1)
  unsigned long long* top_keys;    // [M]
  unsigned int* err;               // device error word
};

StreamPlan make_stream_plan(bool int8_weights, int M, int N, int K, int sm_count);
void attach_reserved(StreamArgs& a, void* ws);  // counters, top-1 keys and error word in the reserved region
int max_top_keys();
void set_kernel_events(void* start, void* stop);  // next launch on this thread records them around the kernel
void take_kernel_events(void** start, void** stop);  // the pending pair (or nulls), cleared
w8a8_status launch_stream_gemm(bool int8_weights, const StreamArgs& a, cudaStream_t st);

}  // namespace w8a8
