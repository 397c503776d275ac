// Shared device/host helpers of libw8a8 (sm_103a).
#pragma once

#include <utility>

#include <cuda_runtime.h>
#include <cuda_fp16.h>
#include <cuda_bf16.h>
#include <cuda_fp8.h>
#include <stdint.h>
#include <stddef.h>

#include "../../include/w8a8.h"

namespace w8a8 {

// ------------------------------------------------------------------------- host status
void set_error(const char* fmt, ...);
const char* get_error();

#define W8A8_CHECK_ARG(cond, code, ...)   \
  do {                                    \
    if (!(cond)) {                        \
      ::w8a8::set_error(__VA_ARGS__);     \
      return code;                        \
    }                                     \
  } while (0)

#define W8A8_CUDA(call)                                                                        \
  do {                                                                                         \
    cudaError_t e_ = (call);                                                                   \
    if (e_ != cudaSuccess) {                                                                   \
      ::w8a8::set_error("CUDA error %s at %s:%d", cudaGetErrorString(e_), __FILE__, __LINE__); \
      return W8A8_ERR_CUDA;                                                                    \
    }                                                                                          \
  } while (0)

#define W8A8_LAUNCH_CHECK() W8A8_CUDA(cudaGetLastError())

// Programmatic dependent launch.  Kernels of the decoder path are launched with programmatic
// stream serialization: the next kernel in the stream may start while this one runs, so that it
// can set up and stream its weights (immutable) early.  Every such kernel calls pdl_wait() before
// its first read of data an earlier kernel wrote and before its first global write; pdl_wait()
// returns once the preceding grid has completed and its writes are visible (at once when the
// launch allowed no overlap).  Because every kernel waits before it can finish, completion is
// ordered along the whole stream.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;\n" ::: "memory"); }
// Let the next kernel in the stream begin launching (its CTAs start as resources free up).
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory"); }

template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                              Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

#define W8A8_TRY(expr)            \
  do {                            \
    w8a8_status s_ = (expr);      \
    if (s_ != W8A8_OK) return s_; \
  } while (0)

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
inline cudaStream_t as_stream(void* s) { return reinterpret_cast<cudaStream_t>(s); }
inline size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

w8a8_status check_device();  // current device must be sm_103

// ---------------------------------------------------------------------- exact conversions
__device__ __forceinline__ float bf16_bits_to_f32(uint32_t bits16) { return __uint_as_float(bits16 << 16); }
__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

__device__ __forceinline__ uint16_t f32_to_bf16_bits(float x) {
  __nv_bfloat16 b = __float2bfloat16_rn(x);
  return *reinterpret_cast<uint16_t*>(&b);
}

// int8 code (as int) -> fp16 bit pattern; exact for |q| <= 2048.
__device__ __forceinline__ uint16_t int_to_f16_bits(int q) {
  __half h = __int2half_rn(q);
  return *reinterpret_cast<uint16_t*>(&h);
}

// Four signed bytes of `w` (byte b0 lowest) -> two f16x2 words {f16(b0), f16(b1)} and
// {f16(b2), f16(b3)}, exact for codes in [-128, 127].  Flipping the sign bit of each byte gives
// u = b + 128 in [0, 255]; the half 0x6400 | u is 1024 + u exactly, so subtracting 1152 leaves b.
__device__ __forceinline__ void i8x4_to_f16x2x2(uint32_t w, uint32_t& lo, uint32_t& hi) {
  const uint32_t u = w ^ 0x80808080u;
  const uint32_t plo = __byte_perm(u, 0x64646464u, 0x4140u);
  const uint32_t phi = __byte_perm(u, 0x64646464u, 0x4342u);
  const __half2 bias = __halves2half2(__ushort_as_half(0x6480u), __ushort_as_half(0x6480u));  // 1152
  __half2 a = __hsub2(*reinterpret_cast<const __half2*>(&plo), bias);
  __half2 b = __hsub2(*reinterpret_cast<const __half2*>(&phi), bias);
  lo = *reinterpret_cast<uint32_t*>(&a);
  hi = *reinterpret_cast<uint32_t*>(&b);
}

// Two fp32 values -> two e4m3 codes (lo in the low byte): round to nearest even, saturating at
// +-448 (the hardware conversion with .satfinite).
__device__ __forceinline__ uint32_t e4m3x2_of(float lo, float hi) {
  return (uint32_t)__nv_cvt_float2_to_fp8x2(make_float2(lo, hi), __NV_SATFINITE, __NV_E4M3);
}
// Two e4m3 codes (low byte first) -> their values as an fp16 pair, low half first (exact: every
// e4m3 value is an fp16 value).
__device__ __forceinline__ uint32_t e4m3x2_to_f16x2(uint32_t codes16) {
  const __half2_raw h = __nv_cvt_fp8x2_to_halfraw2((__nv_fp8x2_storage_t)(codes16 & 0xFFFFu), __NV_E4M3);
  return (uint32_t)h.x | ((uint32_t)h.y << 16);
}

// ------------------------------------------------------------------------- legacy MMA
// D[16x8] += A[16x16] * B[16x8], fp32 accumulate.
__device__ __forceinline__ void mma_f16_16816(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                              uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};\n"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void mma_bf16_16816(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                               uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};\n"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// ----------------------------------------------------------------- streaming global loads
__device__ __forceinline__ uint4 ldg_stream(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}
__device__ __forceinline__ uint4 ldg_keep(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.v4.u32 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

// ------------------------------------------------------------- mbarrier and bulk copies
__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;\n" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void fence_mbar_init() { asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory"); }
__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n" ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];\n" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
// Wait for the phase with the given parity to complete, for at most `budget` SM cycles.
// Returns false on timeout (the caller records an error and stops waiting).
__device__ __forceinline__ bool mbar_wait_bounded(uint32_t bar, uint32_t parity, long long budget) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity))
    if (clock64() - t0 > budget) return false;
  return true;
}
// Start fetching a tensor map (a kernel parameter) so the first copy does not wait for it.
__device__ __forceinline__ void prefetch_tmap(const void* tmap) {
  asm volatile("prefetch.tensormap [%0];\n" ::"l"(reinterpret_cast<uint64_t>(tmap)) : "memory");
}
// 2-D tiled TMA load of one box (coordinates: c0 = innermost element index, c1 = row) into shared
// memory; completion is counted on `bar` in bytes (out-of-bounds elements are zero-filled and counted).
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const void* tmap, int c0, int c1, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];\n" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(c0), "r"(c1), "r"(bar)
      : "memory");
}
// An L2 policy that marks the lines it brings in as the first to evict: decode weights are read
// once per step (far more bytes than L2 holds), and so should not push the KV cache, the
// activations and the small per-step tables out of L2.
__device__ __forceinline__ uint64_t l2_evict_first_policy() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;\n" : "=l"(p));
  return p;
}
// tma_load_2d with an L2 cache policy.
__device__ __forceinline__ void tma_load_2d_policy(uint32_t dst, const void* tmap, int c0, int c1, uint32_t bar,
                                                   uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1, {%2, "
      "%3}], [%4], %5;\n" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(c0), "r"(c1), "r"(bar), "l"(policy)
      : "memory");
}
// 1-D bulk copy global -> shared (async proxy); completion is counted on `bar` in bytes.
// dst and src 16-byte aligned, bytes a multiple of 16.
__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];\n" ::"r"(dst),
               "l"(src), "r"(bytes), "r"(bar)
               : "memory");
}
__device__ __forceinline__ void named_bar_sync(int id, int nthreads) {
  asm volatile("bar.sync %0, %1;\n" ::"r"(id), "r"(nthreads) : "memory");
}
// Named barrier `id` of nthreads threads that also returns whether every one of them passed ok.
__device__ __forceinline__ bool named_bar_all(int id, int nthreads, bool ok) {
  uint32_t r;
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.u32 p, %1, 0;\n bar.red.and.pred p, %2, %3, p;\n selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(r)
      : "r"((uint32_t)ok), "r"(id), "r"(nthreads)
      : "memory");
  return r != 0;
}
__device__ __forceinline__ uint4 lds128(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "r"(addr)
               : "memory");
  return v;
}

// Device-side error bits (reserved workspace word at kErrWordOffset): set by a bounded wait
// that gave up; read and cleared by w8a8_workspace_check.
enum DevErr : unsigned int { DEVERR_CONSUMER_WAIT = 1u, DEVERR_PRODUCER_WAIT = 2u, DEVERR_DRAIN_WAIT = 4u };
constexpr size_t kErrWordOffset = 36864;
constexpr long long kWaitBudgetCycles = 4000000000LL;  // ~2 s at 2 GHz

// --------------------------------------------------------------------- GeGLU fp32 recipe
// gelu_tanh(g) = g / (1 + 2^w), w = -2 log2(e) * sqrt(2/pi) * (g + 0.044715 g^3), each step one
// IEEE fp32 operation rounded to nearest-even, in the order below (no contraction into FMA).
// 2^w = 2^n * p(f), n = rint(w), f = w - n in [-1/2, 1/2], p = degree-7 Taylor polynomial of
// e^{f ln 2} (coefficients (ln 2)^k / k! rounded to fp32), Horner's rule.
__device__ __forceinline__ float exp2_recipe(float w) {
  const float n = rintf(w);
  const float f = __fsub_rn(w, n);
  float p = __uint_as_float(0x377fe5feu);  // (ln2)^7/7!
  p = __fadd_rn(__fmul_rn(p, f), __uint_as_float(0x39218489u));  // (ln2)^6/6!
  p = __fadd_rn(__fmul_rn(p, f), __uint_as_float(0x3aaec3ffu));  // (ln2)^5/5!
  p = __fadd_rn(__fmul_rn(p, f), __uint_as_float(0x3c1d955bu));  // (ln2)^4/4!
  p = __fadd_rn(__fmul_rn(p, f), __uint_as_float(0x3d635847u));  // (ln2)^3/3!
  p = __fadd_rn(__fmul_rn(p, f), __uint_as_float(0x3e75fdf0u));  // (ln2)^2/2!
  p = __fadd_rn(__fmul_rn(p, f), __uint_as_float(0x3f317218u));  // ln2
  p = __fadd_rn(__fmul_rn(p, f), 1.0f);
  const int ni = __float2int_rn(n);                      // |n| <= 126
  const float scale = __int_as_float((ni + 127) << 23);  // 2^n, a normal number
  return __fmul_rn(p, scale);
}

__device__ __forceinline__ float gelu_tanh_recipe(float g) {
  const float g2 = __fmul_rn(g, g);
  const float g3 = __fmul_rn(g2, g);
  const float t = __fadd_rn(g, __fmul_rn(__uint_as_float(0x3d372713u), g3));  // 0.044715
  const float z = __fmul_rn(__uint_as_float(0x3f4c422au), t);                  // sqrt(2/pi)
  float w = __fmul_rn(__uint_as_float(0xc038aa3bu), z);                        // -2 log2(e)
  w = fminf(fmaxf(w, -126.0f), 126.0f);
  const float e = exp2_recipe(w);
  return __fdiv_rn(g, __fadd_rn(1.0f, e));
}

__device__ __forceinline__ float geglu_recipe(float g, float u) { return __fmul_rn(gelu_tanh_recipe(g), u); }

// ------------------------------------------------------------------------- reductions
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// Orderable key for a float (NaN-free): larger float -> larger key.
__device__ __forceinline__ uint32_t float_order_key(float v) {
  const uint32_t b = __float_as_uint(v + 0.0f);  // -0 -> +0
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

}  // namespace w8a8
