// Decode GEMV whose CTAs own whole weight rows (K3 for small layers, and the bf16 pass-through).
//
// At one to eight tokens a decoder layer's linears are small (2.4 to 32 MB) and each one sits on
// the critical path of the next, so their cost is latency more than bandwidth.  The
// weight-streaming kernel splits such a layer's k sum over many CTAs and finishes it with a
// partial-tile protocol through global memory; here every CTA owns R = 8 RW consecutive weight
// rows over the full k range, so each sum ends inside its CTA:
//  * one producer thread streams the CTA's rows through a shared-memory ring with 2-D TMA, starting
//    before the preceding kernel has finished (weights do not depend on it).  A stage holds KS
//    sub-slices of 512 bytes per row (each one or
//    two unswizzled boxes of R rows x 256 elements), so that small-R calls still move enough bytes
//    per pipeline round trip;
//  * the consumer warps (8; 16 on the tensor-core paths of a grid with one CTA per SM) wait for
//    the preceding kernel and stage the activations in shared
//    memory, optionally computing them first from the decoder's residual step (residual add and
//    the two RMSNorms, fused here instead of a separate launch).  The W8A8 path quantises them
//    there, with the arithmetic of the stand-alone per-token quantiser (Eq. stx / xint8,
//    smoothing of Eq. xhat-lmhead), so one launch does K1 and K3;
//  * warp w takes rows w, w + 8, ...; in every sub-slice lane l reads bytes 16 l .. 16 l + 15 of
//    a row's 512 bytes (consecutive lanes read consecutive bytes: no bank conflicts);
//  * INT8: four dp4a per 16 bytes and token, exact INT32 sums (Eq. gemm-final); bf16: fp32 FMAs,
//    sub-slice u of a stage feeding accumulator u mod NA, summed in a fixed order at the end;
//  * the lanes' sums meet in a butterfly (every lane ends with the same value) and lane e runs the
//    epilogue of the warp's output e: dequantisation fl(fl(s_x s_w) acc) (Eq. gemm-final), bias,
//    GeGLU of the FFN section on interleaved gate/up rows (blocks of 8: rows 16q .. 16q+7 are gate
//    rows 8q .. 8q+7, the next 8 the matching up rows; warp w holds both rows of a pair).
// Waits are bounded as in the weight-streaming kernel (error word, no hang).
#include <algorithm>
#include <type_traits>

#include "gemv_small.cuh"
#include "stream_gemm.cuh"
#include "tmap.cuh"

namespace w8a8 {

namespace {

constexpr int kCW = 8;  // consumer warps (16 on the tensor-core paths when the grid has one CTA per SM)
constexpr int kSmemLimit = 227 * 1024;
constexpr int kStatic = 2048;       // static shared memory of the kernel (reduction slots, scales) + slack
constexpr int kSliceBytes = 512;    // bytes of one weight row per sub-slice
constexpr int kMaxInt8K = 8 * 256 * 4;  // K1 keeps a token's smoothed row in registers: 4 vectors of 8 per thread

__device__ __forceinline__ float warp_sum32(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Sum over the first 256 consumer threads in the residual-norm kernel's order (lane tree, then
// warps 0..7 in turn); each of them gets the result (barrier 2: those 256 threads only).
__device__ __forceinline__ float consumer_sum(float v, float* red, int warp, int lane) {
  v = warp_sum32(v);
  named_bar_sync(2, 256);
  if (lane == 0) red[warp] = v;
  named_bar_sync(2, 256);
  float t = 0.0f;
#pragma unroll
  for (int i = 0; i < 8; ++i) t += red[i];
  return t;
}

__device__ __forceinline__ uint32_t f16x2_of(float lo, float hi) {
  uint32_t r;
  asm("cvt.rn.f16x2.f32 %0, %1, %2;\n" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}
__device__ __forceinline__ void ldm_x2(uint32_t addr, uint32_t& r0, uint32_t& r1) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.shared.b16 {%0, %1}, [%2];\n" : "=r"(r0), "=r"(r1) : "r"(addr));
}
__device__ __forceinline__ void ldm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

// Sixteen e4m3 codes (byte j of the vector = code j) as fp32 values (exact).
__device__ __forceinline__ void e4m3x16_to_f32(const uint4& v, float (&x)[16]) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const uint32_t lo = e4m3x2_to_f16x2(w[i]), hi = e4m3x2_to_f16x2(w[i] >> 16);
    const float2 a = __half22float2(*reinterpret_cast<const __half2*>(&lo));
    const float2 b = __half22float2(*reinterpret_cast<const __half2*>(&hi));
    x[4 * i] = a.x;
    x[4 * i + 1] = a.y;
    x[4 * i + 2] = b.x;
    x[4 * i + 3] = b.y;
  }
}

__device__ __forceinline__ void unpack_bf16x8(const uint4& v, float (&x)[8]) {
  x[0] = bf16_lo(v.x); x[1] = bf16_hi(v.x); x[2] = bf16_lo(v.y); x[3] = bf16_hi(v.y);
  x[4] = bf16_lo(v.z); x[5] = bf16_hi(v.z); x[6] = bf16_lo(v.w); x[7] = bf16_hi(v.w);
}

template <int kW, int MT, int RW, int CW>
__global__ void __launch_bounds__((CW + 1) * 32, CW == 8 ? 2 : 1)
    gemv_small_kernel(const __grid_constant__ CUtensorMap tmW, const SmallArgs a) {
  // kW: weights bf16 (SMALL_BF16), INT8 codes (SMALL_INT8) or e4m3 codes (SMALL_FP8: fp32 FMAs on the
  // widened codes at 1-4 token slots, the tensor cores at 8 / 16)
  constexpr bool kInt8 = kW == SMALL_INT8, kFp8 = kW == SMALL_FP8;
  constexpr bool kQ = kInt8 || kFp8;  // one-byte codes, per-token K1, dequantising epilogue
  constexpr float kQmax = kFp8 ? 448.0f : 127.0f;  // largest code magnitude
  constexpr int R = 8 * RW;
  // bf16 at 5-8 tokens: the products run on the tensor cores (mma.sync m16n8k16, the activations
  // as the A operand with token rows 8-15 zero, each 8 weight rows an n-tile), the 8 consumer warps
  // taking alternate k steps of every stage; the weights arrive as 128-byte-swizzled boxes of 64
  // columns and the activation rows are padded by 16 bytes, so the fragment loads hit distinct banks
  constexpr bool kMma = MT >= 8;  // 8 or 16 token slots: the tensor-core paths (16: both halves of the A tile)
  // W8A8 at 5-8 tokens: the same on INT8 codes carried as fp16 (exact): K1 writes the activation
  // codes to shared memory as fp16, each thread widens four consecutive weight bytes (one 32-bit
  // load from 128-byte-swizzled boxes of 128 columns) into two fp16 pairs, and the k order inside
  // an MMA is permuted alike on both operands (thread t's pairs (2t, 2t+1) and (2t+8, 2t+9) hold
  // k 4t .. 4t+3), which leaves the sum unchanged; the fp32 accumulators (at most 128 products per
  // stage, exact) are folded into INT32 after every stage.  The e4m3 path (FP8 variant) does the
  // same with e4m3 codes widened to fp16 by the hardware conversion (exact) and plain fp32
  // accumulation (no fold).
  using Acc = typename std::conditional<kInt8, int, float>::type;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ float s_red[CW];
  __shared__ float s_red8[MT > 4 ? MT : 1][CW];  // 8 / 16-slot K1: per-token maxima of the warps
  __shared__ float s_sx[MT];
  __shared__ unsigned int s_hmax[MT];  // GeGLU epilogue: per-token max |h * 1/delta| of this CTA (float bits)

  const SmallPlan& p = a.p;
  const int S = p.stages, SB = p.stage_bytes, nst = p.nst, kpad = p.kpad, KS = p.ks, nsub = p.nsub;
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t ring = (raw + 1023u) & ~1023u;
  const uint32_t xs = ring + (uint32_t)(S * SB);
  uint64_t* full =
      reinterpret_cast<uint64_t*>(smem_raw + (ring - raw) + (size_t)S * SB + p.xbytes + p.abytes + p.rbytes);
  uint64_t* empty = full + S;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int row0 = blockIdx.x * R;
  if constexpr (CW != kCW) {  // the fused residual norm runs on 8 consumer warps only (not planned)
    if (a.has_rn) {
      if (threadIdx.x == 0) atomicOr(a.err, DEVERR_CONSUMER_WAIT);
      return;
    }
  }

  pdl_trigger();
  if (threadIdx.x == CW * 32) {  // the producer thread: fetch the tensor map before the first copy needs it
    prefetch_tmap(&tmW);
  }
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(smem_u32(full + s), 1);
      mbar_init(smem_u32(empty + s), CW);
    }
    fence_mbar_init();
  }
  __syncthreads();

  // ------------------------------------------------------------------------ producer thread
  if (warp == CW) {
    if (lane != 0) return;
    bool ok = true;
    int it = 0, s = 0;
    uint32_t ph = 0;
    const uint64_t wpol = l2_evict_first_policy();  // each weight row is read once per call
    for (; it < nst; ++it) {
      if (!mbar_wait_bounded(smem_u32(empty + s), ph ^ 1u, kWaitBudgetCycles)) {
        ok = false;
        break;
      }
      const int u0 = it * KS, cnt = min(KS, nsub - u0);
      const uint32_t bar = smem_u32(full + s), dst = ring + (uint32_t)(s * SB);
      mbar_arrive_expect_tx(bar, (uint32_t)(cnt * R * kSliceBytes));
      for (int u = 0; u < cnt; ++u) {
        const uint32_t d = dst + (uint32_t)(u * R * kSliceBytes);
        if constexpr (kQ && kMma) {
#pragma unroll
          for (int j = 0; j < 4; ++j) tma_load_2d_policy(d + j * R * 128, &tmW, (u0 + u) * 512 + 128 * j, row0, bar, wpol);
        } else if constexpr (kQ) {
          tma_load_2d_policy(d, &tmW, (u0 + u) * 512, row0, bar, wpol);
          tma_load_2d_policy(d + R * 256, &tmW, (u0 + u) * 512 + 256, row0, bar, wpol);
        } else if constexpr (kMma) {
#pragma unroll
          for (int j = 0; j < 4; ++j) tma_load_2d_policy(d + j * R * 128, &tmW, (u0 + u) * 256 + 64 * j, row0, bar, wpol);
        } else {
          tma_load_2d_policy(d, &tmW, (u0 + u) * 256, row0, bar, wpol);
        }
      }
      if (++s == S) {
        s = 0;
        ph ^= 1u;
      }
    }
    if (!ok) atomicOr(a.err, DEVERR_PRODUCER_WAIT);
    for (int j = it > S ? it - S : 0; j < it; ++j) {
      if (!mbar_wait_bounded(smem_u32(full + j % S), (uint32_t)((j / S) & 1), kWaitBudgetCycles)) {
        atomicOr(a.err, DEVERR_DRAIN_WAIT);
        break;
      }
    }
    return;
  }

  // ------------------------------------------------------------------------ consumer warps
  const int tid = threadIdx.x;  // 0 .. 255
  // Constants of this warp's rows (per-channel scales, bias) and of K1 (1 / delta): read before
  // waiting for the preceding kernel, so that their latency is off the critical path.
  float swr[RW], bir[RW];
#pragma unroll
  for (int i = 0; i < RW; ++i) {
    const int row = row0 + warp + 8 * i;
    swr[i] = kQ && row < a.N ? a.s_w[row] : 0.0f;
    bir[i] = a.bias && row < a.N ? a.bias[row] : 0.0f;
  }
  float4 idr[4][2];
  if constexpr (kQ) {
    const float4* idl = reinterpret_cast<const float4*>(a.inv_delta);
#pragma unroll
    for (int v = 0; v < 4; ++v) {
      const int vi = tid + v * CW * 32;
      if (vi < (a.K >> 3)) {
        idr[v][0] = idl[2 * vi];
        idr[v][1] = idl[2 * vi + 1];
      }
    }
  }
  // weights of the fused residual norm (constants): this thread's 8 channels
  const int nvk = a.K >> 3;
  float wp[8], wn[8];
  if (a.has_rn && tid < nvk) {
    const float4* p0 = reinterpret_cast<const float4*>(a.rn.w_post + 8 * tid);
    const float4* p1 = reinterpret_cast<const float4*>(a.rn.w_next + 8 * tid);
    const float4 a0 = p0[0], a1 = p0[1], b0 = p1[0], b1 = p1[1];
    wp[0] = a0.x; wp[1] = a0.y; wp[2] = a0.z; wp[3] = a0.w; wp[4] = a1.x; wp[5] = a1.y; wp[6] = a1.z; wp[7] = a1.w;
    wn[0] = b0.x; wn[1] = b0.y; wn[2] = b0.z; wn[3] = b0.w; wn[4] = b1.x; wn[5] = b1.y; wn[6] = b1.z; wn[7] = b1.w;
  }
  pdl_wait();
  uint8_t* xsp = smem_raw + (xs - raw);
  // The bf16 rows behind the activations: the caller's X, or the fused residual norm's output
  // (thread t < K / 8 owns channels 8t .. 8t+7 of every token, as in the residual-norm kernel).
  const uint16_t* xrows = a.X;
  int xstride = a.K;
  // elements between the activation rows in shared memory (bf16, or the fp16 codes of the W8A8
  // tensor-core path; INT8 codes otherwise): padded on the tensor-core paths against bank conflicts
  const int xsb = kMma ? kpad + (kQ ? 16 : 8) : kpad;
  if (a.has_rn) {
    uint16_t* as = kQ ? reinterpret_cast<uint16_t*>(xsp + p.xbytes) : reinterpret_cast<uint16_t*>(xsp);
    for (int m = 0; m < MT; ++m) {
      const bool mine = m < a.M && tid < nvk;
      float yv[8], rv[8];
      float ss = 0.0f;
      if (mine) {
        const uint4 yw = reinterpret_cast<const uint4*>(a.rn.y + (size_t)m * a.K)[tid];
        unpack_bf16x8(yw, yv);
        const float4* rp = reinterpret_cast<const float4*>(a.rn.r_in + (size_t)m * a.K + 8 * tid);
        const float4 r0 = rp[0], r1 = rp[1];
        rv[0] = r0.x; rv[1] = r0.y; rv[2] = r0.z; rv[3] = r0.w; rv[4] = r1.x; rv[5] = r1.y; rv[6] = r1.z; rv[7] = r1.w;
#pragma unroll
        for (int e = 0; e < 8; ++e) ss += yv[e] * yv[e];
      }
      const float inv_y = 1.0f / sqrtf(consumer_sum(ss, s_red, warp, lane) / (float)a.K + a.rn.eps);
      float ss2 = 0.0f;
      if (mine) {
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          rv[e] += yv[e] * inv_y * wp[e];
          ss2 += rv[e] * rv[e];
        }
        if (blockIdx.x == 0) {
          float4* ro = reinterpret_cast<float4*>(a.rn.r_out + (size_t)m * a.K + 8 * tid);
          ro[0] = make_float4(rv[0], rv[1], rv[2], rv[3]);
          ro[1] = make_float4(rv[4], rv[5], rv[6], rv[7]);
        }
      }
      const float inv_r = 1.0f / sqrtf(consumer_sum(ss2, s_red, warp, lane) / (float)a.K + a.rn.eps);
      if (tid < (kpad >> 3)) {  // the padded row: zeros past K and in slots >= M
        uint4 w = make_uint4(0u, 0u, 0u, 0u);
        if (mine) {
          float o[8];
#pragma unroll
          for (int e = 0; e < 8; ++e) o[e] = rv[e] * inv_r * wn[e];
          w.x = (uint32_t)f32_to_bf16_bits(o[0]) | ((uint32_t)f32_to_bf16_bits(o[1]) << 16);
          w.y = (uint32_t)f32_to_bf16_bits(o[2]) | ((uint32_t)f32_to_bf16_bits(o[3]) << 16);
          w.z = (uint32_t)f32_to_bf16_bits(o[4]) | ((uint32_t)f32_to_bf16_bits(o[5]) << 16);
          w.w = (uint32_t)f32_to_bf16_bits(o[6]) | ((uint32_t)f32_to_bf16_bits(o[7]) << 16);
        }
        *reinterpret_cast<uint4*>(as + (size_t)m * (kQ ? kpad : xsb) + 8 * tid) = w;
      }
    }
    named_bar_sync(1, CW * 32);
    xrows = as;
    xstride = kpad;
  }
  if constexpr (kQ) {
    // K1 for every token slot: x_hat = x * (1 / delta), m = max |x_hat|, s = m / 127,
    // q = clamp(rint(x_hat * (127 / m)), -127, 127); slots >= M and the tail past K hold zeros.
    // (e4m3: s = m / 448, q = e4m3(x_hat * (448 / m)), nearest even, saturating.)
    const int nvec = a.K >> 3;
    if constexpr (MT <= 4) {  // one token at a time, all consumer warps on its row
      for (int m = 0; m < MT; ++m) {
        float xh[4][8];
        float amax = 0.0f;
        const bool live = m < a.M;
        if (live) {
          const uint4* src = reinterpret_cast<const uint4*>(xrows + (size_t)m * xstride);
#pragma unroll
          for (int v = 0; v < 4; ++v) {
            const int vi = tid + v * CW * 32;
            if (vi < nvec) {
              const uint4 w = src[vi];
              const float4 d0 = idr[v][0], d1 = idr[v][1];
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
        }
        amax = warp_max(amax);
        if (lane == 0) s_red[warp] = amax;
        named_bar_sync(1, CW * 32);
        float mx = 0.0f;
#pragma unroll
        for (int i = 0; i < CW; ++i) mx = fmaxf(mx, s_red[i]);
        named_bar_sync(1, CW * 32);  // s_red is reused by the next slot
        const float r = mx > 0.0f ? __fdiv_rn(kQmax, mx) : 0.0f;  // fl32(127 / m_t)
        if (tid == 0) {
          const float sx = __fdiv_rn(mx, kQmax);  // s_t^x = fl32(m_t / 127)
          s_sx[m] = sx;
          if (live && a.s_x_dbg && blockIdx.x == 0) a.s_x_dbg[m] = sx;
        }
#pragma unroll
        for (int v = 0; v < 4; ++v) {
          const int vi = tid + v * CW * 32;
          if (vi < nvec) {
            uint2 packed = make_uint2(0u, 0u);
            if (live && kFp8) {  // e4m3 codes (nearest even, saturating), one byte each
              uint32_t c[4];
#pragma unroll
              for (int e = 0; e < 4; ++e)
                c[e] = e4m3x2_of(__fmul_rn(xh[v][2 * e], r), __fmul_rn(xh[v][2 * e + 1], r));
              packed = make_uint2(c[0] | (c[1] << 16), c[2] | (c[3] << 16));
              if (a.xq_dbg && blockIdx.x == 0) *reinterpret_cast<uint2*>(a.xq_dbg + (size_t)m * a.K + 8 * vi) = packed;
            } else if (live) {
              int q[8];
#pragma unroll
              for (int e = 0; e < 8; ++e) q[e] = max(-127, min(127, __float2int_rn(__fmul_rn(xh[v][e], r))));
              packed.x = (uint32_t)(q[0] & 0xff) | ((uint32_t)(q[1] & 0xff) << 8) | ((uint32_t)(q[2] & 0xff) << 16) |
                         ((uint32_t)(q[3] & 0xff) << 24);
              packed.y = (uint32_t)(q[4] & 0xff) | ((uint32_t)(q[5] & 0xff) << 8) | ((uint32_t)(q[6] & 0xff) << 16) |
                         ((uint32_t)(q[7] & 0xff) << 24);
              if (a.xq_dbg && blockIdx.x == 0) *reinterpret_cast<uint2*>(a.xq_dbg + (size_t)m * a.K + 8 * vi) = packed;
            }
            *reinterpret_cast<uint2*>(xsp + (size_t)m * kpad + 8 * vi) = packed;
          }
        }
      }
    } else {  // eight token slots: the whole block on all tokens at once, two passes over the rows
      // pass 1: thread t smooths vectors t, t + 256, ... of every token (eight loads in flight) and
      // keeps each token's running max |x_hat|; one block reduction gives m_t for all tokens
      const float4* idl = reinterpret_cast<const float4*>(a.inv_delta);
      auto smooth8 = [&](const uint4& w, const float4& d0, const float4& d1, float (&xh)[8]) {
        xh[0] = __fmul_rn(bf16_lo(w.x), d0.x);
        xh[1] = __fmul_rn(bf16_hi(w.x), d0.y);
        xh[2] = __fmul_rn(bf16_lo(w.y), d0.z);
        xh[3] = __fmul_rn(bf16_hi(w.y), d0.w);
        xh[4] = __fmul_rn(bf16_lo(w.z), d1.x);
        xh[5] = __fmul_rn(bf16_hi(w.z), d1.y);
        xh[6] = __fmul_rn(bf16_lo(w.w), d1.z);
        xh[7] = __fmul_rn(bf16_hi(w.w), d1.w);
      };
      // tokens m0 .. m0 + 7 of vector vi (eight loads in flight; 16 slots take two groups)
      auto load_tokens = [&](int vi, int m0, uint4 (&w)[8]) {
#pragma unroll
        for (int m = 0; m < 8; ++m)
          w[m] = m0 + m < a.M ? reinterpret_cast<const uint4*>(xrows + (size_t)(m0 + m) * xstride)[vi]
                              : make_uint4(0u, 0u, 0u, 0u);
      };
      float am[MT];
#pragma unroll
      for (int m = 0; m < MT; ++m) am[m] = 0.0f;
      if (a.rowmax_in) {  // the producer's partial maxima stand for pass 1 (the same fp32 products)
        for (int i = tid; i < a.rowmax_n; i += CW * 32)
#pragma unroll
          for (int m = 0; m < MT; ++m) am[m] = fmaxf(am[m], a.rowmax_in[(size_t)i * MT + m]);
      }
      for (int vi = a.rowmax_in ? nvec : tid; vi < nvec; vi += CW * 32) {
        const float4 d0 = idl[2 * vi], d1 = idl[2 * vi + 1];
#pragma unroll
        for (int m0 = 0; m0 < MT; m0 += 8) {
          uint4 w[8];
          load_tokens(vi, m0, w);
#pragma unroll
          for (int m = 0; m < 8; ++m) {
            float xh[8];
            smooth8(w[m], d0, d1, xh);
#pragma unroll
            for (int e = 0; e < 8; ++e) am[m0 + m] = fmaxf(am[m0 + m], fabsf(xh[e]));
          }
        }
      }
#pragma unroll
      for (int m = 0; m < MT; ++m) {
        const float v = warp_max(am[m]);
        if (lane == 0) s_red8[m][warp] = v;
      }
      named_bar_sync(1, CW * 32);
      float rr[MT];
#pragma unroll
      for (int m = 0; m < MT; ++m) {
        float mx = 0.0f;
#pragma unroll
        for (int i = 0; i < CW; ++i) mx = fmaxf(mx, s_red8[m][i]);
        rr[m] = mx > 0.0f ? __fdiv_rn(kQmax, mx) : 0.0f;  // fl32(127 / m_t)
        if (tid == m) {
          const float sx = __fdiv_rn(mx, kQmax);  // s_t^x = fl32(m_t / 127); 0 for slots >= M
          s_sx[m] = sx;
          if (m < a.M && a.s_x_dbg && blockIdx.x == 0) a.s_x_dbg[m] = sx;
        }
      }
      // pass 2: the rows again (L1), quantised; codes of slots >= M are zeros
      for (int vi = tid; vi < nvec; vi += CW * 32) {
        const float4 d0 = idl[2 * vi], d1 = idl[2 * vi + 1];
#pragma unroll
        for (int m0 = 0; m0 < MT; m0 += 8) {
          uint4 w8[8];
          load_tokens(vi, m0, w8);
#pragma unroll
          for (int mi = 0; mi < 8; ++mi) {
          const int m = m0 + mi;
          float xh[8];
          smooth8(w8[mi], d0, d1, xh);
          if constexpr (kFp8) {  // e4m3 codes: their fp16 values for the MMA, the bytes for debugging
            uint32_t c[4];
#pragma unroll
            for (int e = 0; e < 4; ++e)
              c[e] = e4m3x2_of(__fmul_rn(xh[2 * e], rr[m]), __fmul_rn(xh[2 * e + 1], rr[m]));
            reinterpret_cast<uint4*>(xsp + (size_t)m * xsb * 2)[vi] =
                make_uint4(e4m3x2_to_f16x2(c[0]), e4m3x2_to_f16x2(c[1]), e4m3x2_to_f16x2(c[2]), e4m3x2_to_f16x2(c[3]));
            if (a.xq_dbg && blockIdx.x == 0 && m < a.M)
              reinterpret_cast<uint2*>(a.xq_dbg + (size_t)m * a.K)[vi] =
                  make_uint2(c[0] | (c[1] << 16), c[2] | (c[3] << 16));
          } else {
            int q[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) q[e] = max(-127, min(127, __float2int_rn(__fmul_rn(xh[e], rr[m]))));
            if constexpr (kMma) {
              reinterpret_cast<uint4*>(xsp + (size_t)m * xsb * 2)[vi] =
                  make_uint4(f16x2_of((float)q[0], (float)q[1]), f16x2_of((float)q[2], (float)q[3]),
                             f16x2_of((float)q[4], (float)q[5]), f16x2_of((float)q[6], (float)q[7]));
            }
            if (!kMma || (a.xq_dbg && blockIdx.x == 0 && m < a.M)) {
              uint2 packed;
              packed.x = (uint32_t)(q[0] & 0xff) | ((uint32_t)(q[1] & 0xff) << 8) | ((uint32_t)(q[2] & 0xff) << 16) |
                         ((uint32_t)(q[3] & 0xff) << 24);
              packed.y = (uint32_t)(q[4] & 0xff) | ((uint32_t)(q[5] & 0xff) << 8) | ((uint32_t)(q[6] & 0xff) << 16) |
                         ((uint32_t)(q[7] & 0xff) << 24);
              if (!kMma) reinterpret_cast<uint2*>(xsp + (size_t)m * kpad)[vi] = packed;
              if (a.xq_dbg && blockIdx.x == 0 && m < a.M)
                reinterpret_cast<uint2*>(a.xq_dbg + (size_t)m * a.K)[vi] = packed;
            }
          }
          }
        }
      }
    }
    if constexpr (kMma) {  // fp16 codes: zeros from K to the padded length
      const int t8 = (kpad - a.K) >> 3;
      for (int i = tid; i < MT * t8; i += CW * 32) {
        const int m = i / t8, c = i - m * t8;
        *reinterpret_cast<uint4*>(xsp + ((size_t)m * xsb + a.K + 8 * c) * 2) = make_uint4(0u, 0u, 0u, 0u);
      }
    } else {  // INT8 codes: zeros from K to the padded length
      const int tail16 = (kpad - a.K) >> 4;
      for (int i = tid; i < MT * tail16; i += CW * 32) {
        const int m = i / tail16, c = i - m * tail16;
        *reinterpret_cast<uint4*>(xsp + (size_t)m * kpad + a.K + 16 * c) = make_uint4(0u, 0u, 0u, 0u);
      }
    }
  } else if (!a.has_rn) {
    const int vpr = kpad >> 3;  // 16-byte vectors per slot
    const int total = MT * vpr;
    for (int i0 = tid; i0 < total; i0 += 4 * CW * 32) {  // four loads in flight per thread
      uint4 val[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int i = i0 + u * CW * 32;
        const int m = i / vpr, v = i - m * vpr;
        val[u] = make_uint4(0u, 0u, 0u, 0u);
        if (i < total && m < a.M && 8 * v < a.K) val[u] = reinterpret_cast<const uint4*>(a.X + (size_t)m * a.K)[v];
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int i = i0 + u * CW * 32;
        const int m = i / vpr, v = i - m * vpr;
        if (i < total) *reinterpret_cast<uint4*>(xsp + ((size_t)m * xsb + 8 * v) * 2) = val[u];
      }
    }
  }
  named_bar_sync(1, CW * 32);

  // NA independent accumulators per (row, token) keep the FMA / dp4a chains short when a warp has
  // few rows and tokens; sub-slice u of every stage feeds accumulator u mod NA.
  constexpr int NA = RW * MT <= 2 ? 4 : (RW * MT <= 8 ? 2 : 1);
  Acc acc[NA][RW][MT];
#pragma unroll
  for (int c = 0; c < NA; ++c)
#pragma unroll
    for (int i = 0; i < RW; ++i)
#pragma unroll
      for (int m = 0; m < MT; ++m) acc[c][i][m] = 0;
  float mc[2][RW][4];  // MMA path: two accumulator sets (alternate k steps), per n-tile of 8 rows
  int mi32[RW][4];     // W8A8 MMA path: the folded INT32 sums (tokens g, g + 8; rows 8 i + 2 t and + 1)
#pragma unroll
  for (int i = 0; i < RW; ++i) mi32[i][0] = mi32[i][1] = mi32[i][2] = mi32[i][3] = 0;
#pragma unroll
  for (int c = 0; c < 2; ++c)
#pragma unroll
    for (int i = 0; i < RW; ++i) mc[c][i][0] = mc[c][i][1] = mc[c][i][2] = mc[c][i][3] = 0.0f;
  bool ok = true;
  // INT8 sub-slice: two boxes [R][256 B]; lane l reads box l / 16 at byte 16 (l % 16) of the row
  const uint32_t wlane = kQ ? (uint32_t)((lane >> 4) * R * 256 + 16 * (lane & 15)) : (uint32_t)(16 * lane);
  int s = 0;
  uint32_t ph = 0;
  for (int it = 0; it < nst; ++it) {
    if (ok) {
      bool got = true;
      if (lane == 0) got = mbar_wait_bounded(smem_u32(full + s), ph, kWaitBudgetCycles);
      got = __shfl_sync(0xffffffffu, got, 0);
      if (!got) {
        ok = false;
        if (lane == 0) atomicOr(a.err, DEVERR_CONSUMER_WAIT);
      }
    }
    if (ok && kMma) {
      // k steps of 16 of this stage: step q is sub-slice q / 16, 64-column box (q % 16) / 4,
      // chunks 2 (q % 4) and 2 (q % 4) + 1 of its rows; warp w takes steps w, w + 8, ...
      const uint32_t sb = ring + (uint32_t)(s * SB);
      const int u0 = it * KS, cnt = min(KS, nsub - u0);
      const int xr = lane & 7, xh = (lane >> 3) & 1;  // ldmatrix row addresses: token / half
      if constexpr (kQ) {
        // k steps of 16 of this stage: step q is sub-slice q / 32, 128-column box (q % 32) / 8,
        // 16-byte chunk q % 8 of its rows; thread (g, t) reads bytes 4 t .. 4 t + 3 of row g's chunk
        // and of token g's codes
        const int g = lane >> 2, t = lane & 3;
        auto step8 = [&](int q, float (&c)[RW][4]) {
          const int u = q >> 5, kk = q & 31, ch = kk & 7;
          const uint32_t box = sb + (uint32_t)(u * R * kSliceBytes + (kk >> 3) * R * 128);
          const int kg = (u0 + u) * 512 + 16 * kk;
          uint32_t a0, a2, a1 = 0u, a3 = 0u;  // tokens g and, with 16 slots, g + 8
          asm volatile("ld.shared.v2.u32 {%0, %1}, [%2];\n" : "=r"(a0), "=r"(a2) : "r"(xs + (uint32_t)((g * xsb + kg + 4 * t) * 2)));
          if constexpr (MT == 16)
            asm volatile("ld.shared.v2.u32 {%0, %1}, [%2];\n"
                         : "=r"(a1), "=r"(a3)
                         : "r"(xs + (uint32_t)(((g + 8) * xsb + kg + 4 * t) * 2)));
#pragma unroll
          for (int i = 0; i < RW; ++i) {
            uint32_t wb;
            asm volatile("ld.shared.u32 %0, [%1];\n" : "=r"(wb) : "r"(box + (uint32_t)((8 * i + g) * 128 + ((ch ^ g) << 4) + 4 * t)));
            uint32_t b0, b1;
            if constexpr (kFp8) {
              b0 = e4m3x2_to_f16x2(wb);
              b1 = e4m3x2_to_f16x2(wb >> 16);
            } else {
              i8x4_to_f16x2x2(wb, b0, b1);
            }
            mma_f16_16816(c[i], a0, a1, a2, a3, b0, b1);
          }
        };
        // k steps up to K only: the padding past K (to whole 512-byte sub-slices) holds zeros on
        // both operands, so its steps are skipped (1152 k: 72 of 96 steps)
        const int nq = min(32 * cnt, (a.K - u0 * 512) / 16);
        for (int q = warp; q < nq; q += 2 * CW) {
          step8(q, mc[0]);
          if (q + CW < nq) step8(q + CW, mc[1]);
        }
        if constexpr (kInt8) {
#pragma unroll
          for (int i = 0; i < RW; ++i) {  // fold: each set took at most 128 products per output this stage
#pragma unroll
            for (int e = 0; e < (MT == 16 ? 4 : 2); ++e) mi32[i][e] += __float2int_rn(mc[0][i][e]) + __float2int_rn(mc[1][i][e]);
#pragma unroll
            for (int e = 0; e < 4; ++e) mc[0][i][e] = mc[1][i][e] = 0.0f;
          }
        }
      } else {
      auto step = [&](int q, float (&c)[RW][4]) {
        const int u = q >> 4, kk = q & 15, c0 = 2 * (kk & 3);
        const uint32_t box = sb + (uint32_t)(u * R * kSliceBytes + (kk >> 2) * R * 128);
        const int kg = (u0 + u) * 256 + 16 * kk;
        uint32_t a0, a2, a1 = 0u, a3 = 0u;  // 16 slots: matrices (tokens 0-7 | 8-15) x (k lo | k hi)
        if constexpr (MT == 16)
          ldm_x4(xs + (uint32_t)(((xr + 8 * xh) * xsb + kg + 8 * (lane >> 4)) * 2), a0, a1, a2, a3);
        else
          ldm_x2(xs + (uint32_t)((xr * xsb + kg + 8 * xh) * 2), a0, a2);
#pragma unroll
        for (int i = 0; i < RW; i += 2) {
          if (i + 1 < RW) {  // n-tiles i and i + 1: matrices (i, k lo), (i, k hi), (i + 1, lo), (i + 1, hi)
            const int mi = lane >> 3, r = 8 * (i + (mi >> 1)) + xr, ch = c0 + (mi & 1);
            uint32_t b0, b1, b2, b3;
            ldm_x4(box + (uint32_t)(r * 128 + ((ch ^ xr) << 4)), b0, b1, b2, b3);
            mma_bf16_16816(c[i], a0, a1, a2, a3, b0, b1);
            mma_bf16_16816(c[i + 1], a0, a1, a2, a3, b2, b3);
          } else {
            const int r = 8 * i + xr, ch = c0 + xh;
            uint32_t b0, b1;
            ldm_x2(box + (uint32_t)(r * 128 + ((ch ^ xr) << 4)), b0, b1);
            mma_bf16_16816(c[i], a0, a1, a2, a3, b0, b1);
          }
        }
      };
      const int nq = min(16 * cnt, (a.K - u0 * 256) / 16);  // k steps up to K (the padding is zeros)
      for (int q = warp; q < nq; q += 2 * CW) {  // alternate steps feed the two accumulator sets
        step(q, mc[0]);
        if (q + CW < nq) step(q + CW, mc[1]);
      }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(empty + s));
    } else if (ok) {
      const uint32_t sb = ring + (uint32_t)(s * SB);
      const int u0 = it * KS, cnt = min(KS, nsub - u0);
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        if (u >= cnt) break;
        const uint32_t sub = sb + (uint32_t)(u * R * kSliceBytes);
        if constexpr (kInt8) {
          uint4 wv[RW];
#pragma unroll
          for (int i = 0; i < RW; ++i) wv[i] = lds128(sub + wlane + (uint32_t)((warp + 8 * i) * 256));
#pragma unroll
          for (int m = 0; m < MT; ++m) {
            const uint4 xv = lds128(xs + (uint32_t)(m * kpad + (u0 + u) * 512 + 16 * lane));
#pragma unroll
            for (int i = 0; i < RW; ++i) {
              int t = acc[u % NA][i][m];
              t = __dp4a((int)wv[i].x, (int)xv.x, t);
              t = __dp4a((int)wv[i].y, (int)xv.y, t);
              t = __dp4a((int)wv[i].z, (int)xv.z, t);
              t = __dp4a((int)wv[i].w, (int)xv.w, t);
              acc[u % NA][i][m] = t;
            }
          }
        } else if constexpr (kFp8) {  // e4m3 codes widened to fp32 (exact products), fp32 FMAs
          uint4 wv[RW];
#pragma unroll
          for (int i = 0; i < RW; ++i) wv[i] = lds128(sub + wlane + (uint32_t)((warp + 8 * i) * 256));
#pragma unroll
          for (int m = 0; m < MT; ++m) {
            float xf[16];
            e4m3x16_to_f32(lds128(xs + (uint32_t)(m * kpad + (u0 + u) * 512 + 16 * lane)), xf);
#pragma unroll
            for (int i = 0; i < RW; ++i) {
              float wf[16];
              e4m3x16_to_f32(wv[i], wf);
              float t = acc[u % NA][i][m];
#pragma unroll
              for (int e = 0; e < 16; ++e) t = fmaf(wf[e], xf[e], t);
              acc[u % NA][i][m] = t;
            }
          }
        } else {
          uint4 wv[RW];
#pragma unroll
          for (int i = 0; i < RW; ++i) wv[i] = lds128(sub + wlane + (uint32_t)((warp + 8 * i) * kSliceBytes));
#pragma unroll
          for (int m = 0; m < MT; ++m) {
            float x[8];
            unpack_bf16x8(lds128(xs + (uint32_t)((m * kpad + (u0 + u) * 256 + 8 * lane) * 2)), x);
#pragma unroll
            for (int i = 0; i < RW; ++i) {
              float w[8];
              unpack_bf16x8(wv[i], w);
              float t = acc[u % NA][i][m];
#pragma unroll
              for (int e = 0; e < 8; ++e) t = fmaf(w[e], x[e], t);
              acc[u % NA][i][m] = t;
            }
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(empty + s));
    }
    if (++s == S) {
      s = 0;
      ph ^= 1u;
    }
  }
  if constexpr (kMma) {
    // Each warp's sums (accumulators c0 / c1 of n-tile i: token g, rows 8 i + 2 t and + 1; c2 / c3:
    // token g + 8) go to shared memory [warp][row][token]; then every output sums the 8 warps in
    // warp order (W8A8: INT32, exact, then dequantised as fl(fl(s_x s_w) acc)).
    Acc* part = reinterpret_cast<Acc*>(xsp + p.xbytes + p.abytes);
    const int g = lane >> 2, t = lane & 3;
    if (ok) {
#pragma unroll
      for (int i = 0; i < RW; ++i) {
#pragma unroll
        for (int h = 0; h < MT / 8; ++h) {  // token half: g, then g + 8
          const int m = g + 8 * h;
          if constexpr (kInt8) {
            part[(warp * R + 8 * i + 2 * t) * MT + m] = mi32[i][2 * h];
            part[(warp * R + 8 * i + 2 * t + 1) * MT + m] = mi32[i][2 * h + 1];
          } else {
            part[(warp * R + 8 * i + 2 * t) * MT + m] = mc[0][i][2 * h] + mc[1][i][2 * h];
            part[(warp * R + 8 * i + 2 * t + 1) * MT + m] = mc[0][i][2 * h + 1] + mc[1][i][2 * h + 1];
          }
        }
      }
    }
    if (!named_bar_all(1, CW * 32, ok)) return;
    auto total = [&](int r, int m) {
      Acc v = 0;
#pragma unroll
      for (int w = 0; w < CW; ++w) v += part[(w * R + r) * MT + m];
      float y;
      if constexpr (kInt8) {
        y = __fmul_rn(__fmul_rn(s_sx[m], a.s_w[row0 + r]), __int2float_rn(v));
        if (a.acc_dbg) a.acc_dbg[(size_t)m * a.N + row0 + r] = v;
      } else if constexpr (kFp8) {
        y = __fmul_rn(__fmul_rn(s_sx[m], a.s_w[row0 + r]), v);
      } else {
        y = v;
      }
      return a.bias ? __fadd_rn(y, a.bias[row0 + r]) : y;
    };
    if (a.kind == EPI_GEGLU) {  // pair b of block j: gate row 16 j + b, up row 16 j + 8 + b
      if (a.rowmax_out && tid < MT) s_hmax[tid] = 0u;
      if (a.rowmax_out) named_bar_sync(1, CW * 32);
      for (int e = tid; e < (R / 2) * MT; e += CW * 32) {
        const int pr = e / MT, m = e % MT, j = pr >> 3, b = pr & 7;
        const int gr = 16 * j + b;
        if (m >= a.M || row0 + gr + 8 >= a.N) continue;
        const int hc = ((row0 + 16 * j) >> 1) + b;  // h channel
        const uint16_t hb = f32_to_bf16_bits(geglu_recipe(total(gr, m), total(gr + 8, m)));
        a.y[(size_t)m * (a.N >> 1) + hc] = hb;
        if (a.rowmax_out) {  // |x_hat| of the down projection's quantiser, as its K1 computes it
          const float v = fabsf(__fmul_rn(bf16_bits_to_f32(hb), a.next_inv_delta[hc]));
          if (!(v != v)) atomicMax(&s_hmax[m], __float_as_uint(v));  // K1's fmaxf passes over NaN too
        }
      }
      if (a.rowmax_out) {
        named_bar_sync(1, CW * 32);
        if (tid < MT) a.rowmax_out[(size_t)blockIdx.x * MT + tid] = __uint_as_float(s_hmax[tid]);
      }
    } else {
      for (int e = tid; e < R * MT; e += CW * 32) {
        const int r = e / MT, m = e % MT;
        if (m >= a.M || row0 + r >= a.N) continue;
        a.y[(size_t)m * a.N + row0 + r] = f32_to_bf16_bits(total(r, m));
      }
    }
    return;
  }
  if (!ok) return;
#pragma unroll
  for (int c = 1; c < NA; ++c)  // fixed order: ((a0 + a1) + a2) + a3
#pragma unroll
    for (int i = 0; i < RW; ++i)
#pragma unroll
      for (int m = 0; m < MT; ++m) acc[0][i][m] += acc[c][i][m];

  // butterfly: every lane ends with the full sum (a + b == b + a, so partners agree bit for bit)
#pragma unroll
  for (int i = 0; i < RW; ++i)
#pragma unroll
    for (int m = 0; m < MT; ++m) {
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) acc[0][i][m] += __shfl_xor_sync(0xffffffffu, acc[0][i][m], o);
    }
  // The epilogue: lane e of the warp writes the warp's output e (every lane holds every sum), so
  // the outputs' arithmetic (dequantisation, GeGLU) runs side by side on the lanes instead of in
  // turn on one lane.  Lane e picks its sums, scales and bias by selects, not by indexing.
  auto value = [&](Acc v, float sw, float bi, int row, int m) -> float {
    float y;
    if constexpr (kInt8) {
      y = __fmul_rn(__fmul_rn(s_sx[m], sw), __int2float_rn(v));
      if (a.acc_dbg) a.acc_dbg[(size_t)m * a.N + row] = v;
    } else if constexpr (kFp8) {
      y = __fmul_rn(__fmul_rn(s_sx[m], sw), v);
    } else {
      y = v;
    }
    return a.bias ? __fadd_rn(y, bi) : y;
  };
  if (a.kind == EPI_GEGLU) {  // output e = (pair j, token m): gate row slot 2 j, up row slot 2 j + 1
    if (lane >= (RW / 2) * MT) return;
    const int j = lane / MT, m = lane - j * MT;
    Acc ga = 0, ua = 0;
    float sg = 0.0f, su = 0.0f, bg = 0.0f, bu = 0.0f;
#pragma unroll
    for (int jj = 0; jj < RW / 2; ++jj) {
      if (jj == j) {
        sg = swr[2 * jj];
        su = swr[2 * jj + 1];
        bg = bir[2 * jj];
        bu = bir[2 * jj + 1];
      }
#pragma unroll
      for (int mm = 0; mm < MT; ++mm)
        if (jj == j && mm == m) {
          ga = acc[0][2 * jj][mm];
          ua = acc[0][2 * jj + 1][mm];
        }
    }
    const int gi = row0 + 16 * j + warp, ui = gi + 8;
    if (ui >= a.N || m >= a.M) return;
    const int hid = ((row0 + 16 * j) >> 1) + warp;
    const float g = value(ga, sg, bg, gi, m), u = value(ua, su, bu, ui, m);
    a.y[(size_t)m * (a.N >> 1) + hid] = f32_to_bf16_bits(geglu_recipe(g, u));
  } else {  // output e = (row slot i, token m)
    if (lane >= RW * MT) return;
    const int i = lane / MT, m = lane - i * MT;
    Acc av = 0;
    float sw = 0.0f, bi = 0.0f;
#pragma unroll
    for (int ii = 0; ii < RW; ++ii) {
      if (ii == i) {
        sw = swr[ii];
        bi = bir[ii];
      }
#pragma unroll
      for (int mm = 0; mm < MT; ++mm)
        if (ii == i && mm == m) av = acc[0][ii][mm];
    }
    const int row = row0 + warp + 8 * i;
    if (row >= a.N || m >= a.M) return;
    a.y[(size_t)m * a.N + row] = f32_to_bf16_bits(value(av, sw, bi, row, m));
  }
}

template <int kW, int MT, int RW, int CW>
w8a8_status launch_t(const SmallArgs& a, cudaStream_t st) {
  static bool attr_set[64] = {};
  int dev = 0;
  W8A8_CUDA(cudaGetDevice(&dev));
  if (dev >= 0 && dev < 64 && !attr_set[dev]) {
    W8A8_CUDA(cudaFuncSetAttribute(gemv_small_kernel<kW, MT, RW, CW>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                   kSmemLimit - kStatic));
    attr_set[dev] = true;
  }
  constexpr int EB = kW == SMALL_BF16 ? 2 : 1;
  CUtensorMap tw;
  if (MT >= 8)  // the tensor-core paths: 128-byte boxes (64 bf16 or 128 INT8 columns), 128-byte swizzle
    W8A8_TRY(make_tmap_2d(&tw, a.W, EB, (uint64_t)a.K, (uint64_t)a.N, (uint64_t)a.K * EB, 128 / EB, 8 * RW, 128));
  else
    W8A8_TRY(make_tmap_2d(&tw, a.W, EB, (uint64_t)a.K, (uint64_t)a.N, (uint64_t)a.K * EB, 256, 8 * RW, 0));
  W8A8_CUDA(launch_pdl(gemv_small_kernel<kW, MT, RW, CW>, dim3(a.p.P), dim3((CW + 1) * 32), (size_t)a.p.smem_bytes, st,
                       tw, a));
  return W8A8_OK;
}

// accumulator registers a warp may hold (tokens x rows): larger products spill (e4m3 fewer: its
// widened operands take 32 more); the tensor-core paths (8 / 16 token slots) hold 8 (+ 2 or 4
// INT32) per n-tile of 8 rows whatever the token count
constexpr bool slots_fit(int kw, int MT, int RW) {
  return MT >= 8 || MT * RW <= (kw == SMALL_INT8 ? 48 : kw == SMALL_FP8 ? 12 : 32);
}

template <int kW, int MT, int RW>
w8a8_status launch_checked(const SmallArgs& a, cudaStream_t st) {
  if constexpr (slots_fit(kW, MT, RW)) {
    if constexpr (MT >= 8 && RW == 1) {
      if (a.p.cw == 16) return launch_t<kW, MT, RW, 16>(a, st);
    }
    return launch_t<kW, MT, RW, kCW>(a, st);
  } else {
    W8A8_CHECK_ARG(false, W8A8_ERR_SHAPE, "small GEMV: %d tokens x %d rows per warp not built", MT, RW);
  }
}

template <int kW, int MT>
w8a8_status launch_mt(const SmallArgs& a, cudaStream_t st) {
  switch (a.p.RW) {
    case 1: return launch_checked<kW, MT, 1>(a, st);
    case 2: return launch_checked<kW, MT, 2>(a, st);
    case 4: return launch_checked<kW, MT, 4>(a, st);
    default: return launch_checked<kW, MT, 6>(a, st);
  }
}

template <int kW>
w8a8_status launch_typed(const SmallArgs& a, cudaStream_t st) {
  switch (a.p.MT) {
    case 1: return launch_mt<kW, 1>(a, st);
    case 2: return launch_mt<kW, 2>(a, st);
    case 4: return launch_mt<kW, 4>(a, st);
    case 8: return launch_mt<kW, 8>(a, st);
    default: return launch_mt<kW, 16>(a, st);
  }
}

}  // namespace

SmallPlan make_small_plan(int wkind, int M, int N, int K, int kind, int sm_count, bool fused_norm) {
  SmallPlan p{};
  const bool int8_weights = wkind != SMALL_BF16;  // one-byte codes (INT8 or e4m3)
  if (fused_norm && K > 2048) return p;  // one 8-channel vector per consumer thread
  if (M < 1 || M > 16 || N < 1 || K < 16 || K % 16 != 0) return p;
  if (M > 8 && fused_norm) return p;  // the decoder fuses its residual step at 1-8 tokens only
  if (kind != EPI_BF16 && kind != EPI_GEGLU) return p;
  if (kind == EPI_GEGLU && N % 16 != 0) return p;
  // e4m3: fp32 FMAs on the widened codes at 1-2 tokens (one token: 22 us per FFN block against 35 on
  // the tensor cores); from 3 tokens the 8-slot tensor-core path (4 tokens x 6 rows of FMAs spill)
  p.MT = M > 8 ? 16 : (wkind == SMALL_FP8 && M > 2) ? 8 : M <= 1 ? 1 : M <= 2 ? 2 : M <= 4 ? 4 : 8;
  if (int8_weights && p.MT <= 4 && K > kMaxInt8K) return p;
  // fewest rows per CTA (more CTAs) that still fit in two CTAs per SM
  static const int kRw[] = {1, 2, 4, 6};
  for (int rw : kRw) {
    if (kind == EPI_GEGLU && (rw & 1)) continue;
    if ((long long)(N + 8 * rw - 1) / (8 * rw) <= 2LL * sm_count) {
      p.RW = rw;
      break;
    }
  }
  if (p.RW == 0) return p;
  if (!slots_fit(wkind, p.MT, p.RW)) return p;  // registers
  const int R = 8 * p.RW;
  p.P = (N + R - 1) / R;
  const int cps = p.P > sm_count ? 2 : 1;
  p.sub = int8_weights ? 512 : 256;
  p.nsub = (K + p.sub - 1) / p.sub;
  p.kpad = p.nsub * p.sub;
  const bool mma = p.MT >= 8;  // the kernel's tensor-core paths (same rule): padded bf16 / fp16 rows
  p.xbytes = mma ? p.MT * (p.kpad + (int8_weights ? 16 : 8)) * 2 : p.MT * p.kpad * (int8_weights ? 1 : 2);
  p.abytes = fused_norm && int8_weights ? p.MT * p.kpad * 2 : 0;
  // 16 consumer warps where a tensor-core grid has one CTA per SM (one row block per warp group
  // of 8 rows: the down and o projections at 5-16 tokens): twice the warps to hide the MMA and
  // widening latencies of a CTA that has the SM to itself
  p.cw = mma && p.RW == 1 && p.P <= sm_count && !fused_norm ? 16 : kCW;
  p.rbytes = mma ? p.cw * R * p.MT * 4 : 0;  // the warps' partial sums
  const int budget = kSmemLimit / cps - kStatic - 1024 - p.xbytes - p.abytes - p.rbytes - 16 * 16;
  // sub-slices per stage: 4 for warps with one or two rows, fewer for wider CTAs; each stage must
  // fit twice in the ring unless one stage covers everything
  for (int ks = p.RW <= 2 ? 4 : p.RW == 4 ? 2 : 1; ks >= 1; ks >>= 1) {
    const int nst = (p.nsub + ks - 1) / ks, sb = ks * R * kSliceBytes;
    const int stages = std::min(std::min(16, nst), budget / sb);
    if (stages >= std::min(nst, 2)) {
      p.ks = ks;
      p.nst = nst;
      p.stage_bytes = sb;
      p.stages = stages;
      break;
    }
  }
  if (p.ks == 0) return p;
  p.smem_bytes = 1024 + p.stages * p.stage_bytes + p.xbytes + p.abytes + p.rbytes + 16 * p.stages;
  p.ok = 1;
  return p;
}

w8a8_status launch_small_gemv(int wkind, const SmallArgs& a, cudaStream_t st) {
  if (a.M == 0 || a.N == 0) return W8A8_OK;
  W8A8_CHECK_ARG(a.p.ok, W8A8_ERR_SHAPE, "small GEMV: no plan for M=%d N=%d K=%d", a.M, a.N, a.K);
  void *v0, *v1;
  take_kernel_events(&v0, &v1);
  cudaEvent_t e0 = reinterpret_cast<cudaEvent_t>(v0), e1 = reinterpret_cast<cudaEvent_t>(v1);
  if (e0) W8A8_CUDA(cudaEventRecord(e0, st));
  const w8a8_status s = wkind == SMALL_FP8    ? launch_typed<SMALL_FP8>(a, st)
                        : wkind == SMALL_INT8 ? launch_typed<SMALL_INT8>(a, st)
                                              : launch_typed<SMALL_BF16>(a, st);
  if (e1) W8A8_CUDA(cudaEventRecord(e1, st));
  return s;
}

}  // namespace w8a8
