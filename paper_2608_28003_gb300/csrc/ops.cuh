// Internal entry points shared by the C-ABI functions and the decoder (no argument checks).
#pragma once

#include "common.cuh"
#include "gemv_small.cuh"

namespace w8a8 {

struct DevInfo {
  int ok = -1;  // -1 unknown, 0 unsupported, 1 sm_103
  int sms = 0;
};
w8a8_status dev_info(DevInfo* out);
int device_sms();

struct LinearWs {
  size_t xf16, sx, part, total;
};
struct FfnWs {
  size_t h, gu, dn, rowmax, total;
};
LinearWs linear_ws(int M, int N, int K, bool int8_path, int sms);
FfnWs ffn_ws(int M, int H, int F, int sms);

// qsum (nullable): per row, sum_k |q_tk| (the tensor-core GEMM's exactness certificate)
w8a8_status launch_quantize_rows(const uint16_t* X, int M, int K, const float* inv_delta, int8_t* xq,
                                 uint16_t* xq_f16, float* s_x, cudaStream_t st, int* qsum = nullptr);
w8a8_status launch_quantize_rows_fp8(const uint16_t* X, int M, int K, const float* inv_delta, uint8_t* xq,
                                     float* s_x, cudaStream_t st);
w8a8_status launch_act_absmax(const uint16_t* X, int T, int K, float* absmax, cudaStream_t st);

// The per-token quantiser's outputs for X computed by the kernel that produced X (the decoder's
// norm kernels): fp16 codes [M, K], s_x [M] and the rows' sums of |codes| [M] (nullable).  A W8A8
// linear that runs the tensor-core GEMM then launches no quantiser of its own; other routes
// quantise X themselves and ignore them.
struct PreCodes {
  const uint16_t* codes16;
  const float* s_x;
  const int* qsum;
};

// kind: 0 bf16 output, 1 GeGLU, 2 fp32 logits (+ top-1)
w8a8_status run_w8a8_linear(const w8a8_qweight* w, const uint16_t* X, int M, const float* bias, int kind, uint16_t* Y,
                            float* logits, int32_t* top1, const w8a8_debug* dbg, void* ws, int sms, cudaStream_t st,
                            const ResNorm* rn = nullptr, const PreCodes* pre = nullptr);
w8a8_status run_bf16_linear(const uint16_t* W, int N, int K, const uint16_t* X, int M, const float* bias, int kind,
                            uint16_t* Y, float* logits, int32_t* top1, void* ws, int sms, cudaStream_t st,
                            const ResNorm* rn = nullptr);
w8a8_status run_ffn(const w8a8_ffn_weights* f, int precision, const uint16_t* X, int M, uint16_t* Y, uint16_t* h_dbg,
                    void* workspace, int sms, cudaStream_t st, const ResNorm* rn_gate_up = nullptr,
                    const PreCodes* pre_gate_up = nullptr);
// rn (decode only): the call's input is computed from the decoder's residual step inside the
// decode GEMV (X is ignored); W8A8_ERR_SHAPE when the decode GEMV does not take the call.
bool decode_gemv_takes(bool int8, int M, int N, int K, bool geglu, int sms);

}  // namespace w8a8
