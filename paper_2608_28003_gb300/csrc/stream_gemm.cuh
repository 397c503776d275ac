// Weight-streaming GEMM for decode-sized token counts (K3: W8A8; K6: bf16 pass-through).
#pragma once

#include "common.cuh"

namespace w8a8 {

enum EpiKind { EPI_BF16 = 0, EPI_GEGLU = 1, EPI_F32 = 2 };

struct StreamPlan {
  int NB;       // 8-token blocks per token group (1, 2, 4 or 8)
  int zgroups;  // token groups (grid.z)
  int RT;       // 16-row tiles
  int KS;       // 64-wide k steps
  int S;        // k slices in total
  int sps;      // k steps per slice
  int WS;       // warp slices per CTA
  int CS;       // CTA-level k splits
  int RPC;      // row tiles per CTA
  int groups;   // row-tile groups (grid.x / CS)
  size_t partial_bytes;
};

struct StreamArgs {
  const void* W;       // [N, K] int8 codes or bf16
  const uint16_t* X;   // [M, K] fp16 codes (int path) or bf16
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
  void* partials;                  // CS > 1: [zgroups][CS][RT*16][8*NB] int32/fp32
  unsigned int* tile_counters;     // [zgroups * groups]
  unsigned int* grid_counter;      // one counter (top-1)
  unsigned long long* top_keys;    // [M]
};

StreamPlan make_stream_plan(int M, int N, int K, int sm_count);
void attach_reserved(StreamArgs& a, void* ws);  // counters and top-1 keys in the reserved region
int max_top_keys();
w8a8_status launch_stream_gemm(bool int8_weights, const StreamArgs& a, cudaStream_t st);

}  // namespace w8a8
