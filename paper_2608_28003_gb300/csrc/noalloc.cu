// w8a8_linear_noalloc: the W8A8 linear for callers that cannot allocate device memory.
//
// Some callers cannot call cudaMalloc: code that runs while a memory pool or allocator must not be
// touched (for example inside a plug-in of a framework that owns all device memory, or on a path
// with a fixed memory budget decided at start-up).  This entry point needs no workspace from the
// caller: its scratch (per-token codes and scales, split-K partial tiles, counters) is one
// statically sized device array that the library image carries, so each GPU that loads the
// library holds kNoAllocScratchBytes of device memory until the process exits.
#include <mutex>

#include "common.cuh"
#include "ops.cuh"

namespace w8a8 {

size_t linear_scratch_bytes(int M, int N, int K, int sms);
w8a8_status linear_on_scratch(const w8a8_qweight* w, const uint16_t* X, int M, const float* bias, uint16_t* Y,
                              void* scratch, size_t scratch_bytes, cudaStream_t st);
w8a8_status check_linear_args(const char* who, const w8a8_qweight* w, const uint16_t* X, int M, const float* bias,
                              const uint16_t* Y);

namespace {

constexpr size_t kNoAllocScratchBytes = 8u << 20;  // 8 MiB, shared by every call on a device

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

// Device address of the scratch array, looked up once per device.  In host code the array's name
// only stands for the symbol; kernels must be given this address.
void* g_scratch_ptr[64] = {};
std::mutex g_scratch_mu;

w8a8_status scratch_for_current_device(void** out) {
  int dev = 0;
  W8A8_CUDA(cudaGetDevice(&dev));
  W8A8_CHECK_ARG(dev >= 0 && dev < 64, W8A8_ERR_UNSUPPORTED, "device ordinal %d out of range", dev);
  std::lock_guard<std::mutex> lk(g_scratch_mu);
  if (g_scratch_ptr[dev] == nullptr) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    W8A8_CHECK_ARG(e == cudaSuccess && p != nullptr, W8A8_ERR_CUDA,
                   "w8a8_linear_noalloc: cudaGetSymbolAddress of the scratch array failed: %s", cudaGetErrorString(e));
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
  return W8A8_OK;
}

}  // namespace

}  // namespace w8a8

using namespace w8a8;

extern "C" size_t w8a8_linear_noalloc_capacity(void) { return kNoAllocScratchBytes; }

extern "C" w8a8_status w8a8_linear_noalloc(const w8a8_qweight* w, const uint16_t* X, int M, const float* bias,
                                           uint16_t* Y, void* stream) {
  W8A8_TRY(check_linear_args("w8a8_linear_noalloc", w, X, M, bias, Y));
  if (M == 0) return W8A8_OK;
  DevInfo d;
  W8A8_TRY(dev_info(&d));  // an unsupported device is reported as such, before any sizing
  const size_t need = linear_scratch_bytes(M, w->n, w->k, d.sms);
  W8A8_CHECK_ARG(need <= kNoAllocScratchBytes, W8A8_ERR_SHAPE,
                 "w8a8_linear_noalloc: M=%d, N=%d, K=%d needs %zu bytes of scratch; the built-in array holds %zu "
                 "(use w8a8_linear with a workspace)",
                 M, w->n, w->k, need, kNoAllocScratchBytes);
  void* scratch = nullptr;
  W8A8_TRY(scratch_for_current_device(&scratch));
  cudaStream_t st = as_stream(stream);
  // The counters and top-1 keys at the start of the scratch must be zero when a call begins; the
  // array keeps whatever the previous call left, so clear them on every call (no allocation).  The
  // device error word between them is left alone: it stays set until w8a8_linear_noalloc_check
  // reads it, as a workspace's word stays set until w8a8_workspace_check.
  char* base = static_cast<char*>(scratch);
  W8A8_CUDA(cudaMemsetAsync(base, 0, kErrWordOffset, st));
  W8A8_CUDA(cudaMemsetAsync(base + kErrWordOffset + 16, 0, W8A8_WS_RESERVED - kErrWordOffset - 16, st));
  return linear_on_scratch(w, X, M, bias, Y, scratch, kNoAllocScratchBytes, st);
}

extern "C" w8a8_status w8a8_linear_noalloc_check(void* stream) {
  W8A8_TRY(check_device());
  void* scratch = nullptr;
  W8A8_TRY(scratch_for_current_device(&scratch));
  return w8a8_workspace_check(scratch, stream);
}
