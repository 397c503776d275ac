// Per-token activation quantisation (K1), calibration statistics and weight preparation.
//
//   K1   quantize_rows_kernel   Eq. xhat-lmhead, stx, xint8 (LM Head section)
//   K9   act_absmax_kernel      max_t |X_tj| (Eq. delta-attn numerator, LM Head section)
//   K8   colmax / smooth / quant_weight_rows / interleave kernels: Eq. delta-attn, what-lmhead,
//        si, what-ffn
//
// Every step that decides an INT8 code is one IEEE fp32 operation with round-to-nearest-even
// (__fmul_rn, __fdiv_rn, __fsqrt_rn, __float2int_rn), in the order the header documents.  The FP8
// variant (Future Work: e4m3 in place of INT8) runs the same kernels with 448 in place of 127 and
// the hardware's e4m3 conversion (nearest even, saturating) in place of rint and the clamp.
#include <cmath>

#include "common.cuh"

namespace w8a8 {

// ------------------------------------------------------------------------------ K1
// One CTA per row.  Each thread holds up to kVec 16-byte vectors (8 bf16 each) of the row in
// registers between the max pass and the quantise pass; longer rows are re-read.
template <int kVec, bool kFp8>
__global__ void __launch_bounds__(256) quantize_rows_kernel(const uint16_t* __restrict__ X, int K,
                                                           const float* __restrict__ inv_delta,
                                                           int8_t* __restrict__ xq,
                                                           uint16_t* __restrict__ xq_f16,
                                                           float* __restrict__ s_x, int* __restrict__ qsum) {
  pdl_trigger();
  pdl_wait();
  const int row = blockIdx.x;
  const int nvec = K >> 3;
  const uint4* src = reinterpret_cast<const uint4*>(X + (size_t)row * K);
  const float4* idl = reinterpret_cast<const float4*>(inv_delta);
  float xh[kVec][8];
  float amax = 0.0f;
  const bool in_regs = nvec <= kVec * (int)blockDim.x;
  if (in_regs) {
#pragma unroll
    for (int v = 0; v < kVec; ++v) {
      const int vi = threadIdx.x + v * blockDim.x;
      if (vi < nvec) {
        const uint4 w = src[vi];
        const float4 d0 = idl[2 * vi], d1 = idl[2 * vi + 1];
        xh[v][0] = __fmul_rn(bf16_lo(w.x), d0.x);
        xh[v][1] = __fmul_rn(bf16_hi(w.x), d0.y);
        xh[v][2] = __fmul_rn(bf16_lo(w.y), d0.z);
        xh[v][3] = __fmul_rn(bf16_hi(w.y), d0.w);
        xh[v][4] = __fmul_rn(bf16_lo(w.z), d1.x);
        xh[v][5] = __fmul_rn(bf16_hi(w.z), d1.y);
        xh[v][6] = __fmul_rn(bf16_lo(w.w), d1.z);
        xh[v][7] = __fmul_rn(bf16_hi(w.w), d1.w);
#pragma unroll
        for (int e = 0; e < 8; ++e) amax = fmaxf(amax, fabsf(xh[v][e]));
      }
    }
  } else {
    for (int vi = threadIdx.x; vi < nvec; vi += blockDim.x) {
      const uint4 w = src[vi];
      const float4 d0 = idl[2 * vi], d1 = idl[2 * vi + 1];
      amax = fmaxf(amax, fabsf(__fmul_rn(bf16_lo(w.x), d0.x)));
      amax = fmaxf(amax, fabsf(__fmul_rn(bf16_hi(w.x), d0.y)));
      amax = fmaxf(amax, fabsf(__fmul_rn(bf16_lo(w.y), d0.z)));
      amax = fmaxf(amax, fabsf(__fmul_rn(bf16_hi(w.y), d0.w)));
      amax = fmaxf(amax, fabsf(__fmul_rn(bf16_lo(w.z), d1.x)));
      amax = fmaxf(amax, fabsf(__fmul_rn(bf16_hi(w.z), d1.y)));
      amax = fmaxf(amax, fabsf(__fmul_rn(bf16_lo(w.w), d1.z)));
      amax = fmaxf(amax, fabsf(__fmul_rn(bf16_hi(w.w), d1.w)));
    }
  }
  __shared__ float red[32];
  amax = warp_max(amax);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = amax;
  __syncthreads();
  if (threadIdx.x < 32) {
    float v = threadIdx.x < (blockDim.x >> 5) ? red[threadIdx.x] : 0.0f;
    v = warp_max(v);
    if (threadIdx.x == 0) red[0] = v;
  }
  __syncthreads();
  const float m = red[0];
  constexpr float kQmax = kFp8 ? 448.0f : 127.0f;
  const float r = m > 0.0f ? __fdiv_rn(kQmax, m) : 0.0f;  // fl32(127 / m_t)
  if (threadIdx.x == 0) s_x[row] = __fdiv_rn(m, kQmax);  // s_t^x = fl32(m_t / 127)

  int qs = 0;  // sum_k |q_tk| of this thread's codes (the GEMM's exactness certificate)
  auto emit = [&](int vi, const float (&v8)[8]) {
    if constexpr (kFp8) {  // e4m3 codes (xq receives the bytes)
      uint32_t c[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) c[e] = e4m3x2_of(__fmul_rn(v8[2 * e], r), __fmul_rn(v8[2 * e + 1], r));
      reinterpret_cast<uint2*>(xq + (size_t)row * K)[vi] = make_uint2(c[0] | (c[1] << 16), c[2] | (c[3] << 16));
    } else {
      int q[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) q[e] = max(-127, min(127, __float2int_rn(__fmul_rn(v8[e], r))));
#pragma unroll
      for (int e = 0; e < 8; ++e) qs += abs(q[e]);
      if (xq) {
        uint2 packed;
        packed.x = (uint32_t)(q[0] & 0xff) | ((uint32_t)(q[1] & 0xff) << 8) | ((uint32_t)(q[2] & 0xff) << 16) |
                   ((uint32_t)(q[3] & 0xff) << 24);
        packed.y = (uint32_t)(q[4] & 0xff) | ((uint32_t)(q[5] & 0xff) << 8) | ((uint32_t)(q[6] & 0xff) << 16) |
                   ((uint32_t)(q[7] & 0xff) << 24);
        reinterpret_cast<uint2*>(xq + (size_t)row * K)[vi] = packed;
      }
      if (xq_f16) {
        uint4 h;
        h.x = (uint32_t)int_to_f16_bits(q[0]) | ((uint32_t)int_to_f16_bits(q[1]) << 16);
        h.y = (uint32_t)int_to_f16_bits(q[2]) | ((uint32_t)int_to_f16_bits(q[3]) << 16);
        h.z = (uint32_t)int_to_f16_bits(q[4]) | ((uint32_t)int_to_f16_bits(q[5]) << 16);
        h.w = (uint32_t)int_to_f16_bits(q[6]) | ((uint32_t)int_to_f16_bits(q[7]) << 16);
        reinterpret_cast<uint4*>(xq_f16 + (size_t)row * K)[vi] = h;
      }
    }
  };
  if (in_regs) {
#pragma unroll
    for (int v = 0; v < kVec; ++v) {
      const int vi = threadIdx.x + v * blockDim.x;
      if (vi < nvec) emit(vi, xh[v]);
    }
  } else {
    for (int vi = threadIdx.x; vi < nvec; vi += blockDim.x) {
      const uint4 w = src[vi];
      const float4 d0 = idl[2 * vi], d1 = idl[2 * vi + 1];
      float v8[8] = {__fmul_rn(bf16_lo(w.x), d0.x), __fmul_rn(bf16_hi(w.x), d0.y),
                     __fmul_rn(bf16_lo(w.y), d0.z), __fmul_rn(bf16_hi(w.y), d0.w),
                     __fmul_rn(bf16_lo(w.z), d1.x), __fmul_rn(bf16_hi(w.z), d1.y),
                     __fmul_rn(bf16_lo(w.w), d1.z), __fmul_rn(bf16_hi(w.w), d1.w)};
      emit(vi, v8);
    }
  }
  if (qsum) {  // one integer sum per row (exact in any order)
    __shared__ int qred[32];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) qs += __shfl_xor_sync(0xffffffffu, qs, o);
    if ((threadIdx.x & 31) == 0) qred[threadIdx.x >> 5] = qs;
    __syncthreads();
    if (threadIdx.x == 0) {
      int t = 0;
      for (int w = 0; w < (int)(blockDim.x >> 5); ++w) t += qred[w];
      qsum[row] = t;
    }
  }
}

w8a8_status launch_quantize_rows(const uint16_t* X, int M, int K, const float* inv_delta, int8_t* xq,
                                 uint16_t* xq_f16, float* s_x, cudaStream_t st, int* qsum) {
  if (M == 0) return W8A8_OK;
  const int nvec = K / 8;
  const int threads = nvec <= 4 * 128 ? 128 : 256;
  W8A8_CUDA(launch_pdl(quantize_rows_kernel<4, false>, dim3(M), dim3(threads), 0, st, X, K, inv_delta, xq, xq_f16,
                       s_x, qsum));
  return W8A8_OK;
}

w8a8_status launch_quantize_rows_fp8(const uint16_t* X, int M, int K, const float* inv_delta, uint8_t* xq,
                                     float* s_x, cudaStream_t st) {
  if (M == 0) return W8A8_OK;
  const int nvec = K / 8;
  const int threads = nvec <= 4 * 128 ? 128 : 256;
  W8A8_CUDA(launch_pdl(quantize_rows_kernel<4, true>, dim3(M), dim3(threads), 0, st, X, K, inv_delta,
                       reinterpret_cast<int8_t*>(xq), static_cast<uint16_t*>(nullptr), s_x, static_cast<int*>(nullptr)));
  return W8A8_OK;
}

// ------------------------------------------------------------------------------ K9
// Running column max of |X| over rows.  Non-negative floats order like their bit patterns, so
// an unsigned atomicMax on the bits is an exact float max.
__global__ void act_absmax_kernel(const uint16_t* __restrict__ X, int T, int K, int rows_per_block,
                                  float* __restrict__ absmax) {
  const int nvec = K >> 3;
  const int vi = blockIdx.x * blockDim.x + threadIdx.x;
  if (vi >= nvec) return;
  const int r0 = blockIdx.y * rows_per_block;
  const int r1 = min(T, r0 + rows_per_block);
  float m[8] = {0, 0, 0, 0, 0, 0, 0, 0};
  for (int r = r0; r < r1; ++r) {
    const uint4 w = reinterpret_cast<const uint4*>(X + (size_t)r * K)[vi];
    m[0] = fmaxf(m[0], fabsf(bf16_lo(w.x)));
    m[1] = fmaxf(m[1], fabsf(bf16_hi(w.x)));
    m[2] = fmaxf(m[2], fabsf(bf16_lo(w.y)));
    m[3] = fmaxf(m[3], fabsf(bf16_hi(w.y)));
    m[4] = fmaxf(m[4], fabsf(bf16_lo(w.z)));
    m[5] = fmaxf(m[5], fabsf(bf16_hi(w.z)));
    m[6] = fmaxf(m[6], fabsf(bf16_lo(w.w)));
    m[7] = fmaxf(m[7], fabsf(bf16_hi(w.w)));
  }
  unsigned int* out = reinterpret_cast<unsigned int*>(absmax) + vi * 8;
#pragma unroll
  for (int e = 0; e < 8; ++e) atomicMax(out + e, __float_as_uint(m[e]));
}

w8a8_status launch_act_absmax(const uint16_t* X, int T, int K, float* absmax, cudaStream_t st) {
  if (T == 0) return W8A8_OK;
  const int nvec = K / 8;
  const int rows_per_block = 64;
  dim3 grid((nvec + 127) / 128, (T + rows_per_block - 1) / rows_per_block);
  act_absmax_kernel<<<grid, 128, 0, st>>>(X, T, K, rows_per_block, absmax);
  W8A8_LAUNCH_CHECK();
  return W8A8_OK;
}

// ------------------------------------------------------------------------------ K8
// Column max of |W| over rows into `out` (pre-zeroed or holding a running max).
__global__ void colmax_kernel(const uint16_t* __restrict__ W, int N, int K, int rows_per_block,
                              float* __restrict__ out) {
  const int nvec = K >> 3;
  const int vi = blockIdx.x * blockDim.x + threadIdx.x;
  if (vi >= nvec) return;
  const int r0 = blockIdx.y * rows_per_block;
  const int r1 = min(N, r0 + rows_per_block);
  float m[8] = {0, 0, 0, 0, 0, 0, 0, 0};
  for (int r = r0; r < r1; ++r) {
    const uint4 w = reinterpret_cast<const uint4*>(W + (size_t)r * K)[vi];
    m[0] = fmaxf(m[0], fabsf(bf16_lo(w.x)));
    m[1] = fmaxf(m[1], fabsf(bf16_hi(w.x)));
    m[2] = fmaxf(m[2], fabsf(bf16_lo(w.y)));
    m[3] = fmaxf(m[3], fabsf(bf16_hi(w.y)));
    m[4] = fmaxf(m[4], fabsf(bf16_lo(w.z)));
    m[5] = fmaxf(m[5], fabsf(bf16_hi(w.z)));
    m[6] = fmaxf(m[6], fabsf(bf16_lo(w.w)));
    m[7] = fmaxf(m[7], fabsf(bf16_hi(w.w)));
  }
  unsigned int* o = reinterpret_cast<unsigned int*>(out) + vi * 8;
#pragma unroll
  for (int e = 0; e < 8; ++e) atomicMax(o + e, __float_as_uint(m[e]));
}

// delta_j from the activation statistic ax_j and the weight statistic aw_j (held in `delta` on
// entry), Eq. delta-attn.  alpha == 0.5: fl32(sqrt(ax)) / fl32(sqrt(aw)); otherwise fp64 pow,
// rounded once.  delta = 1 where a statistic is zero or the quotient is not finite / zero.
__global__ void smooth_factor_kernel(const float* __restrict__ ax, float* __restrict__ delta,
                                     float* __restrict__ inv_delta, int K, float alpha, int smooth) {
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  if (j >= K) return;
  float d = 1.0f;
  if (smooth) {
    const float a = ax[j], w = delta[j];
    if (alpha == 0.5f) {
      d = __fdiv_rn(__fsqrt_rn(a), __fsqrt_rn(w));
    } else {
      d = (float)(pow((double)a, (double)alpha) / pow((double)w, 1.0 - (double)alpha));
    }
    if (a == 0.0f || w == 0.0f || !isfinite(d) || d == 0.0f) d = 1.0f;
  }
  delta[j] = d;
  inv_delta[j] = __fdiv_rn(1.0f, d);
}

// One CTA per output row p: W_hat = fl32(W * delta), m = max |W_hat|, s = fl32(m / 127),
// q = clamp(rint(fl32(W_hat * fl32(127 / m))), -127, 127) (Eq. si, what-ffn on Eq. what-lmhead).
// The source row is W0 + p*K, or for the gate/up interleave (W1 != nullptr): block q = p / 16,
// r = p % 16, r < 8 -> W0 row 8q + r, else W1 row 8q + r - 8.
template <bool kFp8>
__global__ void __launch_bounds__(256) quant_weight_rows_kernel(const uint16_t* __restrict__ W0,
                                                               const uint16_t* __restrict__ W1, int K,
                                                               const float* __restrict__ delta,
                                                               int8_t* __restrict__ wq, float* __restrict__ s_w,
                                                               uint16_t* __restrict__ wq_f16) {
  const int p = blockIdx.x;
  const uint16_t* src;
  if (W1 == nullptr) {
    src = W0 + (size_t)p * K;
  } else {
    const int q = p >> 4, r = p & 15;
    src = r < 8 ? W0 + (size_t)(8 * q + r) * K : W1 + (size_t)(8 * q + r - 8) * K;
  }
  const int nvec = K >> 3;
  float amax = 0.0f;
  for (int vi = threadIdx.x; vi < nvec; vi += blockDim.x) {
    const uint4 w = reinterpret_cast<const uint4*>(src)[vi];
    const float4 d0 = reinterpret_cast<const float4*>(delta)[2 * vi];
    const float4 d1 = reinterpret_cast<const float4*>(delta)[2 * vi + 1];
    amax = fmaxf(amax, fabsf(__fmul_rn(bf16_lo(w.x), d0.x)));
    amax = fmaxf(amax, fabsf(__fmul_rn(bf16_hi(w.x), d0.y)));
    amax = fmaxf(amax, fabsf(__fmul_rn(bf16_lo(w.y), d0.z)));
    amax = fmaxf(amax, fabsf(__fmul_rn(bf16_hi(w.y), d0.w)));
    amax = fmaxf(amax, fabsf(__fmul_rn(bf16_lo(w.z), d1.x)));
    amax = fmaxf(amax, fabsf(__fmul_rn(bf16_hi(w.z), d1.y)));
    amax = fmaxf(amax, fabsf(__fmul_rn(bf16_lo(w.w), d1.z)));
    amax = fmaxf(amax, fabsf(__fmul_rn(bf16_hi(w.w), d1.w)));
  }
  __shared__ float red[32];
  amax = warp_max(amax);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = amax;
  __syncthreads();
  if (threadIdx.x < 32) {
    float v = threadIdx.x < (blockDim.x >> 5) ? red[threadIdx.x] : 0.0f;
    v = warp_max(v);
    if (threadIdx.x == 0) red[0] = v;
  }
  __syncthreads();
  const float m = red[0];
  constexpr float kQmax = kFp8 ? 448.0f : 127.0f;
  const float r = m > 0.0f ? __fdiv_rn(kQmax, m) : 0.0f;
  if (threadIdx.x == 0) s_w[p] = __fdiv_rn(m, kQmax);
  for (int vi = threadIdx.x; vi < nvec; vi += blockDim.x) {
    const uint4 w = reinterpret_cast<const uint4*>(src)[vi];
    const float4 d0 = reinterpret_cast<const float4*>(delta)[2 * vi];
    const float4 d1 = reinterpret_cast<const float4*>(delta)[2 * vi + 1];
    const float v8[8] = {__fmul_rn(bf16_lo(w.x), d0.x), __fmul_rn(bf16_hi(w.x), d0.y),
                         __fmul_rn(bf16_lo(w.y), d0.z), __fmul_rn(bf16_hi(w.y), d0.w),
                         __fmul_rn(bf16_lo(w.z), d1.x), __fmul_rn(bf16_hi(w.z), d1.y),
                         __fmul_rn(bf16_lo(w.w), d1.z), __fmul_rn(bf16_hi(w.w), d1.w)};
    if constexpr (kFp8) {  // e4m3 codes; an all-zero row has r = 0 and codes 0
      uint32_t c[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) c[e] = e4m3x2_of(__fmul_rn(v8[2 * e], r), __fmul_rn(v8[2 * e + 1], r));
      reinterpret_cast<uint2*>(wq + (size_t)p * K)[vi] = make_uint2(c[0] | (c[1] << 16), c[2] | (c[3] << 16));
    } else {
      int q[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) q[e] = m > 0.0f ? max(-127, min(127, __float2int_rn(__fmul_rn(v8[e], r)))) : 0;
      uint2 packed;
      packed.x = (uint32_t)(q[0] & 0xff) | ((uint32_t)(q[1] & 0xff) << 8) | ((uint32_t)(q[2] & 0xff) << 16) |
                 ((uint32_t)(q[3] & 0xff) << 24);
      packed.y = (uint32_t)(q[4] & 0xff) | ((uint32_t)(q[5] & 0xff) << 8) | ((uint32_t)(q[6] & 0xff) << 16) |
                 ((uint32_t)(q[7] & 0xff) << 24);
      reinterpret_cast<uint2*>(wq + (size_t)p * K)[vi] = packed;
      if (wq_f16) {
        uint4 h;
        h.x = (uint32_t)int_to_f16_bits(q[0]) | ((uint32_t)int_to_f16_bits(q[1]) << 16);
        h.y = (uint32_t)int_to_f16_bits(q[2]) | ((uint32_t)int_to_f16_bits(q[3]) << 16);
        h.z = (uint32_t)int_to_f16_bits(q[4]) | ((uint32_t)int_to_f16_bits(q[5]) << 16);
        h.w = (uint32_t)int_to_f16_bits(q[6]) | ((uint32_t)int_to_f16_bits(q[7]) << 16);
        reinterpret_cast<uint4*>(wq_f16 + (size_t)p * K)[vi] = h;
      }
    }
  }
}

__global__ void interleave_rows_kernel(const uint16_t* __restrict__ W0, const uint16_t* __restrict__ W1,
                                       int K, uint16_t* __restrict__ out) {
  const int p = blockIdx.x;
  const int q = p >> 4, r = p & 15;
  const uint16_t* src = r < 8 ? W0 + (size_t)(8 * q + r) * K : W1 + (size_t)(8 * q + r - 8) * K;
  const int nvec = K >> 3;
  for (int vi = threadIdx.x; vi < nvec; vi += blockDim.x)
    reinterpret_cast<uint4*>(out + (size_t)p * K)[vi] = reinterpret_cast<const uint4*>(src)[vi];
}

static w8a8_status launch_colmax(const uint16_t* W, int N, int K, float* out, cudaStream_t st) {
  const int nvec = K / 8;
  const int rows_per_block = 256;
  dim3 grid((nvec + 127) / 128, (N + rows_per_block - 1) / rows_per_block);
  colmax_kernel<<<grid, 128, 0, st>>>(W, N, K, rows_per_block, out);
  W8A8_LAUNCH_CHECK();
  return W8A8_OK;
}

static w8a8_status prepare_common(const uint16_t* W0, const uint16_t* W1, int rows_each, int K,
                                  const float* act_absmax, float alpha, int smooth, int8_t* wq, float* s_w,
                                  float* delta, float* inv_delta, uint16_t* wq_f16, cudaStream_t st,
                                  bool fp8 = false) {
  const int N = W1 ? 2 * rows_each : rows_each;
  W8A8_CUDA(cudaMemsetAsync(delta, 0, sizeof(float) * K, st));
  if (smooth) {
    w8a8_status s = launch_colmax(W0, rows_each, K, delta, st);
    if (s != W8A8_OK) return s;
    if (W1) {
      s = launch_colmax(W1, rows_each, K, delta, st);
      if (s != W8A8_OK) return s;
    }
  }
  smooth_factor_kernel<<<(K + 255) / 256, 256, 0, st>>>(act_absmax, delta, inv_delta, K, alpha, smooth);
  W8A8_LAUNCH_CHECK();
  if (N > 0) {
    if (fp8)
      quant_weight_rows_kernel<true><<<N, 256, 0, st>>>(W0, W1, K, delta, wq, s_w, nullptr);
    else
      quant_weight_rows_kernel<false><<<N, 256, 0, st>>>(W0, W1, K, delta, wq, s_w, wq_f16);
    W8A8_LAUNCH_CHECK();
  }
  return W8A8_OK;
}

}  // namespace w8a8

using namespace w8a8;

extern "C" w8a8_status w8a8_act_absmax(const uint16_t* X, int T, int K, float* absmax, void* stream) {
  W8A8_CHECK_ARG(T >= 0 && K >= 0, W8A8_ERR_INVALID_ARG, "w8a8_act_absmax: negative size");
  W8A8_CHECK_ARG(K % 16 == 0 && K <= W8A8_MAX_K, W8A8_ERR_SHAPE, "w8a8_act_absmax: K=%d must be a multiple of 16 and <= %d", K, W8A8_MAX_K);
  if (T == 0 || K == 0) return W8A8_OK;
  W8A8_CHECK_ARG(X && absmax, W8A8_ERR_INVALID_ARG, "w8a8_act_absmax: null pointer");
  W8A8_CHECK_ARG(aligned16(X) && aligned16(absmax), W8A8_ERR_ALIGN, "w8a8_act_absmax: pointers must be 16-byte aligned");
  w8a8_status s = check_device();
  if (s != W8A8_OK) return s;
  return launch_act_absmax(X, T, K, absmax, as_stream(stream));
}

static w8a8_status check_prep_args(const char* who, const void* W, int N, int K, const float* act_absmax,
                                   int smooth, const int8_t* wq, const float* s_w, const float* delta,
                                   const float* inv_delta, const uint16_t* wq_f16) {
  W8A8_CHECK_ARG(N >= 0 && K >= 0, W8A8_ERR_INVALID_ARG, "%s: negative size", who);
  W8A8_CHECK_ARG(K % 16 == 0 && K <= W8A8_MAX_K, W8A8_ERR_SHAPE, "%s: K=%d must be a multiple of 16 and <= %d", who, K, W8A8_MAX_K);
  W8A8_CHECK_ARG(W && wq && s_w && delta && inv_delta && (act_absmax || !smooth), W8A8_ERR_INVALID_ARG,
                 "%s: null pointer", who);
  W8A8_CHECK_ARG(aligned16(W) && aligned16(wq) && aligned16(s_w) && aligned16(delta) && aligned16(inv_delta) &&
                     (!act_absmax || aligned16(act_absmax)) && (!wq_f16 || aligned16(wq_f16)),
                 W8A8_ERR_ALIGN, "%s: pointers must be 16-byte aligned", who);
  return W8A8_OK;
}

extern "C" w8a8_status w8a8_prepare_weights(const uint16_t* W, int N, int K, const float* act_absmax, float alpha,
                                            int smooth, int8_t* wq, float* s_w, float* delta, float* inv_delta,
                                            uint16_t* wq_f16, void* stream) {
  w8a8_status s = check_prep_args("w8a8_prepare_weights", W, N, K, act_absmax, smooth, wq, s_w, delta, inv_delta, wq_f16);
  if (s != W8A8_OK) return s;
  W8A8_CHECK_ARG(std::isfinite(alpha) && alpha >= 0.0f && alpha <= 1.0f, W8A8_ERR_INVALID_ARG,
                 "w8a8_prepare_weights: alpha must be in [0, 1]");
  if (K == 0) return W8A8_OK;
  s = check_device();
  if (s != W8A8_OK) return s;
  return prepare_common(W, nullptr, N, K, act_absmax, alpha, smooth, wq, s_w, delta, inv_delta, wq_f16,
                        as_stream(stream));
}

extern "C" w8a8_status w8a8_prepare_gate_up(const uint16_t* W_gate, const uint16_t* W_up, int F, int H,
                                            const float* act_absmax, float alpha, int smooth, int8_t* wq,
                                            float* s_w, float* delta, float* inv_delta, uint16_t* wq_f16,
                                            void* stream) {
  w8a8_status s = check_prep_args("w8a8_prepare_gate_up", W_gate, F, H, act_absmax, smooth, wq, s_w, delta,
                                  inv_delta, wq_f16);
  if (s != W8A8_OK) return s;
  W8A8_CHECK_ARG(W_up && aligned16(W_up), W8A8_ERR_INVALID_ARG, "w8a8_prepare_gate_up: W_up null or unaligned");
  W8A8_CHECK_ARG(F % 8 == 0, W8A8_ERR_SHAPE, "w8a8_prepare_gate_up: F=%d must be a multiple of 8", F);
  W8A8_CHECK_ARG(std::isfinite(alpha) && alpha >= 0.0f && alpha <= 1.0f, W8A8_ERR_INVALID_ARG,
                 "w8a8_prepare_gate_up: alpha must be in [0, 1]");
  if (H == 0) return W8A8_OK;
  s = check_device();
  if (s != W8A8_OK) return s;
  return prepare_common(W_gate, W_up, F, H, act_absmax, alpha, smooth, wq, s_w, delta, inv_delta, wq_f16,
                        as_stream(stream));
}

extern "C" w8a8_status w8a8_interleave_gate_up(const uint16_t* W_gate, const uint16_t* W_up, int F, int H,
                                               uint16_t* out, void* stream) {
  W8A8_CHECK_ARG(F >= 0 && H >= 0, W8A8_ERR_INVALID_ARG, "w8a8_interleave_gate_up: negative size");
  W8A8_CHECK_ARG(F % 8 == 0 && H % 16 == 0 && H <= W8A8_MAX_K, W8A8_ERR_SHAPE,
                 "w8a8_interleave_gate_up: F %% 8 and H %% 16 must be 0");
  if (F == 0 || H == 0) return W8A8_OK;
  W8A8_CHECK_ARG(W_gate && W_up && out, W8A8_ERR_INVALID_ARG, "w8a8_interleave_gate_up: null pointer");
  W8A8_CHECK_ARG(aligned16(W_gate) && aligned16(W_up) && aligned16(out), W8A8_ERR_ALIGN,
                 "w8a8_interleave_gate_up: pointers must be 16-byte aligned");
  w8a8_status s = check_device();
  if (s != W8A8_OK) return s;
  interleave_rows_kernel<<<2 * F, 128, 0, as_stream(stream)>>>(W_gate, W_up, H, out);
  W8A8_LAUNCH_CHECK();
  return W8A8_OK;
}

extern "C" w8a8_status w8a8_quantize_activations(const uint16_t* X, int M, int K, const float* inv_delta,
                                                 int8_t* xq, uint16_t* xq_f16, float* s_x, void* stream) {
  W8A8_CHECK_ARG(M >= 0 && K >= 0, W8A8_ERR_INVALID_ARG, "w8a8_quantize_activations: negative size");
  W8A8_CHECK_ARG(K % 16 == 0 && K <= W8A8_MAX_K, W8A8_ERR_SHAPE, "w8a8_quantize_activations: K=%d must be a multiple of 16 and <= %d", K, W8A8_MAX_K);
  if (M == 0) return W8A8_OK;
  W8A8_CHECK_ARG(X && inv_delta && s_x, W8A8_ERR_INVALID_ARG, "w8a8_quantize_activations: null pointer");
  W8A8_CHECK_ARG(aligned16(X) && aligned16(inv_delta) && aligned16(s_x) && (!xq || aligned16(xq)) &&
                     (!xq_f16 || aligned16(xq_f16)),
                 W8A8_ERR_ALIGN, "w8a8_quantize_activations: pointers must be 16-byte aligned");
  w8a8_status s = check_device();
  if (s != W8A8_OK) return s;
  return launch_quantize_rows(X, M, K, inv_delta, xq, xq_f16, s_x, as_stream(stream), nullptr);
}

// ------------------------------------------------------------------------ FP8 (e4m3) variant
extern "C" w8a8_status w8a8_fp8_prepare_weights(const uint16_t* W, int N, int K, const float* act_absmax, float alpha,
                                                int smooth, uint8_t* wq, float* s_w, float* delta, float* inv_delta,
                                                void* stream) {
  int8_t* codes = reinterpret_cast<int8_t*>(wq);
  w8a8_status s =
      check_prep_args("w8a8_fp8_prepare_weights", W, N, K, act_absmax, smooth, codes, s_w, delta, inv_delta, nullptr);
  if (s != W8A8_OK) return s;
  W8A8_CHECK_ARG(std::isfinite(alpha) && alpha >= 0.0f && alpha <= 1.0f, W8A8_ERR_INVALID_ARG,
                 "w8a8_fp8_prepare_weights: alpha must be in [0, 1]");
  if (K == 0) return W8A8_OK;
  s = check_device();
  if (s != W8A8_OK) return s;
  return prepare_common(W, nullptr, N, K, act_absmax, alpha, smooth, codes, s_w, delta, inv_delta, nullptr,
                        as_stream(stream), true);
}

extern "C" w8a8_status w8a8_fp8_prepare_gate_up(const uint16_t* W_gate, const uint16_t* W_up, int F, int H,
                                                const float* act_absmax, float alpha, int smooth, uint8_t* wq,
                                                float* s_w, float* delta, float* inv_delta, void* stream) {
  int8_t* codes = reinterpret_cast<int8_t*>(wq);
  w8a8_status s = check_prep_args("w8a8_fp8_prepare_gate_up", W_gate, F, H, act_absmax, smooth, codes, s_w, delta,
                                  inv_delta, nullptr);
  if (s != W8A8_OK) return s;
  W8A8_CHECK_ARG(W_up && aligned16(W_up), W8A8_ERR_INVALID_ARG, "w8a8_fp8_prepare_gate_up: W_up null or unaligned");
  W8A8_CHECK_ARG(F % 8 == 0, W8A8_ERR_SHAPE, "w8a8_fp8_prepare_gate_up: F=%d must be a multiple of 8", F);
  W8A8_CHECK_ARG(std::isfinite(alpha) && alpha >= 0.0f && alpha <= 1.0f, W8A8_ERR_INVALID_ARG,
                 "w8a8_fp8_prepare_gate_up: alpha must be in [0, 1]");
  if (H == 0) return W8A8_OK;
  s = check_device();
  if (s != W8A8_OK) return s;
  return prepare_common(W_gate, W_up, F, H, act_absmax, alpha, smooth, codes, s_w, delta, inv_delta, nullptr,
                        as_stream(stream), true);
}

extern "C" w8a8_status w8a8_fp8_quantize_activations(const uint16_t* X, int M, int K, const float* inv_delta,
                                                     uint8_t* xq, float* s_x, void* stream) {
  W8A8_CHECK_ARG(M >= 0 && K >= 0, W8A8_ERR_INVALID_ARG, "w8a8_fp8_quantize_activations: negative size");
  W8A8_CHECK_ARG(K % 16 == 0 && K <= W8A8_MAX_K, W8A8_ERR_SHAPE,
                 "w8a8_fp8_quantize_activations: K=%d must be a multiple of 16 and <= %d", K, W8A8_MAX_K);
  if (M == 0) return W8A8_OK;
  W8A8_CHECK_ARG(X && inv_delta && s_x && xq, W8A8_ERR_INVALID_ARG, "w8a8_fp8_quantize_activations: null pointer");
  W8A8_CHECK_ARG(aligned16(X) && aligned16(inv_delta) && aligned16(s_x) && aligned16(xq), W8A8_ERR_ALIGN,
                 "w8a8_fp8_quantize_activations: pointers must be 16-byte aligned");
  w8a8_status s = check_device();
  if (s != W8A8_OK) return s;
  return launch_quantize_rows_fp8(X, M, K, inv_delta, xq, s_x, as_stream(stream));
}
