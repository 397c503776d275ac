// Measurement aid (no counterpart in the paper): the sustained rate of each exact integer route the
// kernels can take for the INT8 GEMM on this GPU, as the denominator of their rooflines.
//   route 0: dp4a (four INT8 x INT8 products summed into INT32 per instruction and lane)
//   route 1: mma.sync m16n8k32 with s8 operands and s32 accumulation (the legacy INT8 tensor path)
//   route 2: mma.sync m16n8k16 with fp16 operands and fp32 accumulation (the decode GEMV's path on
//            INT8 codes carried as fp16)
// Every warp of a grid covering every SM runs independent chains of one instruction on register
// operands (eight accumulators in flight), timed with CUDA events around the launch; the
// accumulators are stored so that nothing is removed as dead.  Returns ops/s in TOPS (two ops per
// multiply-add).
#include "common.cuh"
#include "ops.cuh"

namespace w8a8 {

namespace {

constexpr int kPeakThreads = 256, kPeakChains = 8;

__global__ void __launch_bounds__(kPeakThreads) route_peak_kernel(int route, int iters, uint32_t seed, int* sink) {
  const uint32_t v = seed * (threadIdx.x + 1) + blockIdx.x;
  if (route == 0) {
    int acc[kPeakChains];
#pragma unroll
    for (int c = 0; c < kPeakChains; ++c) acc[c] = c;
    const int a = (int)v, b = (int)(v * 7u + 3u);
    for (int i = 0; i < iters; ++i) {
#pragma unroll
      for (int c = 0; c < kPeakChains; ++c)  // volatile: every instruction is issued as written
        asm volatile("dp4a.s32.s32 %0, %1, %2, %0;\n" : "+r"(acc[c]) : "r"(a), "r"(b));
    }
    int s = 0;
#pragma unroll
    for (int c = 0; c < kPeakChains; ++c) s += acc[c];
    sink[blockIdx.x * blockDim.x + threadIdx.x] = s;
  } else if (route == 1) {
    int d[kPeakChains][4];
#pragma unroll
    for (int c = 0; c < kPeakChains; ++c) d[c][0] = d[c][1] = d[c][2] = d[c][3] = 0;
    const uint32_t a0 = v, a1 = v * 3u, a2 = v * 5u, a3 = v * 9u, b0 = v * 17u, b1 = v * 33u;
    for (int i = 0; i < iters; ++i) {
#pragma unroll
      for (int c = 0; c < kPeakChains; ++c)
        asm volatile(
            "mma.sync.aligned.m16n8k32.row.col.s32.s8.s8.s32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
            "{%0,%1,%2,%3};\n"
            : "+r"(d[c][0]), "+r"(d[c][1]), "+r"(d[c][2]), "+r"(d[c][3])
            : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
    }
    int s = 0;
#pragma unroll
    for (int c = 0; c < kPeakChains; ++c) s += d[c][0] + d[c][1] + d[c][2] + d[c][3];
    sink[blockIdx.x * blockDim.x + threadIdx.x] = s;
  } else {
    float d[kPeakChains][4];
#pragma unroll
    for (int c = 0; c < kPeakChains; ++c) d[c][0] = d[c][1] = d[c][2] = d[c][3] = 0.0f;
    const uint32_t h = 0x3c003c00u ^ (v & 0x00ff00ffu);  // fp16 pairs near 1
    for (int i = 0; i < iters; ++i) {
#pragma unroll
      for (int c = 0; c < kPeakChains; ++c) mma_f16_16816(d[c], h, h, h, h, h, h);
    }
    float s = 0.0f;
#pragma unroll
    for (int c = 0; c < kPeakChains; ++c) s += d[c][0] + d[c][1] + d[c][2] + d[c][3];
    sink[blockIdx.x * blockDim.x + threadIdx.x] = __float_as_int(s);
  }
}

}  // namespace

}  // namespace w8a8

using namespace w8a8;

extern "C" w8a8_status w8a8_route_peak(int route, double* tops, void* stream) {
  W8A8_CHECK_ARG(tops && route >= 0 && route <= 2, W8A8_ERR_INVALID_ARG, "w8a8_route_peak: route %d", route);
  DevInfo d;
  W8A8_TRY(dev_info(&d));
  cudaStream_t st = as_stream(stream);
  // two CTAs (16 warps) per SM; about 0.1-0.3 s per measurement at the expected rates
  const int blocks = d.sms * 2, iters = route == 0 ? 2048 : route == 1 ? 256 : 1024;
  int* sink = nullptr;
  cudaEvent_t e0 = nullptr, e1 = nullptr;
  w8a8_status s = W8A8_OK;
  float ms = 0.0f;
  do {
    if (cudaMalloc(&sink, sizeof(int) * (size_t)blocks * kPeakThreads) != cudaSuccess ||
        cudaEventCreate(&e0) != cudaSuccess || cudaEventCreate(&e1) != cudaSuccess) {
      set_error("w8a8_route_peak: CUDA set-up failed");
      s = W8A8_ERR_CUDA;
      break;
    }
    route_peak_kernel<<<blocks, kPeakThreads, 0, st>>>(route, iters / 16, 1u, sink);  // warm-up
    cudaEventRecord(e0, st);
    route_peak_kernel<<<blocks, kPeakThreads, 0, st>>>(route, iters, 1u, sink);
    cudaEventRecord(e1, st);
    if (cudaEventSynchronize(e1) != cudaSuccess || cudaEventElapsedTime(&ms, e0, e1) != cudaSuccess ||
        cudaGetLastError() != cudaSuccess) {
      set_error("w8a8_route_peak: launch failed");
      s = W8A8_ERR_CUDA;
      break;
    }
  } while (0);
  if (sink) cudaFree(sink);
  if (e0) cudaEventDestroy(e0);
  if (e1) cudaEventDestroy(e1);
  if (s != W8A8_OK) return s;
  const double warps = (double)blocks * (kPeakThreads / 32);
  const double per_warp_instr = route == 0 ? 32.0 * 8.0 : route == 1 ? 16.0 * 8 * 32 * 2 : 16.0 * 8 * 16 * 2;
  *tops = warps * iters * kPeakChains * per_warp_instr / (ms * 1e-3) / 1e12;
  return W8A8_OK;
}
